"""The save path on the GPU: KV pages gathered from the paged cache into a staging
pool (device or pinned host memory), states snapshotted to host slots, and the
completion dependency the paper checked with a delayed save (Section 3.1,
Section 5.3 and Table 5: D2H page comparisons, delayed-save wait pairs).
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2609_15030_gb300 as hs
from hs_inputs import HYBRID12, gen_block_table
from tests.gpu_helpers import device

pytestmark = pytest.mark.gpu
POISON = 0xEE


def _cache(dev, L, nb, P, seed):
    c = torch.empty((L, nb * P), dtype=torch.uint8, device=dev)
    c.view(torch.int32).random_(generator=torch.Generator(device=dev).manual_seed(seed))
    return c


@pytest.mark.parametrize("where", ["device", "pinned_host"])
def test_save_pages_match_the_oracle(where):
    dev = device()
    L, nb, P, n_pages = 3, 96, HYBRID12.page_bytes, 41
    cache = _cache(dev, L, nb, P, 5)
    bt = gen_block_table(21, 0, n_pages, nb)
    extra = 2                                            # staging pages past n_pages stay poisoned
    if where == "device":
        st = torch.full((L, (n_pages + extra) * P), POISON, dtype=torch.uint8, device=dev)
    else:
        st = torch.full((L, (n_pages + extra) * P), POISON, dtype=torch.uint8).pin_memory()
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_save_kv_pages(hs.ptr_array([cache[l] for l in range(L)], dev),
                        hs.ptr_array([st[l] for l in range(L)], dev), L,
                        torch.from_numpy(bt).to(dev), n_pages, P, nb, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    h_cache = [cache[l].cpu().numpy() for l in range(L)]
    ref = [np.full((n_pages + extra) * P, POISON, np.uint8) for _ in range(L)]
    oracle.gather_pages(h_cache, ref, bt, n_pages, P)
    got = st.cpu().numpy()
    for l in range(L):
        assert np.array_equal(got[l], ref[l]), l
        assert got[l][:n_pages * P].any()                 # the compared bytes are not all zero


def test_save_then_restore_round_trip():
    """Pages saved from one cache and restored into a poisoned one at the same blocks
    come back bit for bit; other blocks stay poisoned (Table 5's two directions)."""
    dev = device()
    L, nb, P, n_pages = 3, 80, HYBRID12.page_bytes, 37
    a = _cache(dev, L, nb, P, 9)
    bt = torch.from_numpy(gen_block_table(22, 0, n_pages, nb)).to(dev)
    st = torch.empty((L, n_pages * P), dtype=torch.uint8).pin_memory()
    b = torch.full((L, nb * P), POISON, dtype=torch.uint8, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    ap = hs.ptr_array([a[l] for l in range(L)], dev)
    sp = hs.ptr_array([st[l] for l in range(L)], dev)
    bp = hs.ptr_array([b[l] for l in range(L)], dev)
    hs.hs_save_kv_pages(ap, sp, L, bt, n_pages, P, nb, err)
    hs.hs_restore_kv_pages(sp, bp, L, bt, n_pages, P, nb, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    av, bv = a.view(L, nb, P), b.view(L, nb, P)
    idx = bt.long()
    assert torch.equal(bv[:, idx], av[:, idx])
    mask = torch.ones(nb, dtype=torch.bool, device=dev)
    mask[idx] = False
    assert bool((bv[:, mask] == POISON).all())


def test_save_out_of_range_block_reports_and_skips():
    dev = device()
    P, nb = 4096, 6
    cache = _cache(dev, 1, nb, P, 3)
    st = torch.full((3 * P,), POISON, dtype=torch.uint8, device=dev)
    bt = torch.tensor([4, 6, 1], dtype=torch.int32, device=dev)          # 6 is out of range
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_save_kv_pages(hs.ptr_array([cache], dev), hs.ptr_array([st], dev), 1, bt, 3, P, nb, err)
    torch.cuda.synchronize()
    assert err.item() == hs.HS_DEVERR_BLOCK_OOB
    c = cache.cpu().numpy().reshape(nb, P)
    s = st.cpu().numpy().reshape(3, P)
    assert np.array_equal(s[0], c[4]) and np.array_equal(s[2], c[1])
    assert (s[1] == POISON).all()


def test_checkpoint_states_to_pinned_host_slots():
    """States snapshotted straight into pinned host slots (the checkpoint half of the
    save), bit for bit."""
    dev = device()
    n, fe = 4, HYBRID12.n_heads * HYBRID12.d * HYBRID12.d
    src = [torch.randn(fe, device=dev) for _ in range(n)]
    dst = [torch.full((fe,), -3.0).pin_memory() for _ in range(n)]
    hs.hs_checkpoint_states(hs.ptr_array(src, dev), hs.ptr_array(dst, dev), n, fe)
    torch.cuda.synchronize()
    for s, d in zip(src, dst):
        assert torch.equal(s.cpu().view(torch.int32), d.view(torch.int32))


def _driver():
    for name in ("libcuda.so.1", "libcuda.so"):
        try:
            return ctypes.CDLL(name)
        except OSError:
            continue
    pytest.skip("CUDA driver library not found")


def test_delayed_saves_complete_before_dependent_reuse():
    """Each save is followed, on its stream, by a host step that sleeps 500 ms before
    the save counts as complete (the paper's injected delay); the reuse stream waits on
    the completion event of every save before it overwrites those cache blocks.  The
    host staging must hold the pre-overwrite pages, the cache the new ones, and every
    overwrite must start after its delayed save ended (Section 3.1, Table 5)."""
    dev = device()
    drv = _driver()
    # the injected delay: the driver calls libc usleep(500000) on its own thread (the
    # host-function argument is the microsecond count), so no Python runs there
    usleep = ctypes.cast(ctypes.CDLL("libc.so.6").usleep, ctypes.c_void_p)
    drv.cuLaunchHostFunc.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
    drv.cuLaunchHostFunc.restype = ctypes.c_int

    L, nb, P, n_saves, m = 3, 64, HYBRID12.page_bytes, 3, 8
    cache = _cache(dev, L, nb, P, 31)
    before = cache.clone()
    new_pages = _cache(dev, L, m, P, 32)                 # what each reuse writes into its blocks
    s_save, s_reuse = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    cp = hs.ptr_array([cache[l] for l in range(L)], dev)
    npp = hs.ptr_array([new_pages[l] for l in range(L)], dev)
    # disjoint block sets, one per save; every buffer and pointer array stays referenced
    # until the streams drain
    perm = gen_block_table(40, 0, n_saves * m, nb)
    bts = [torch.from_numpy(perm[i * m:(i + 1) * m].copy()).to(dev) for i in range(n_saves)]
    stagings = [torch.full((L, m * P), POISON, dtype=torch.uint8).pin_memory() for _ in range(n_saves)]
    sps = [hs.ptr_array([st[l] for l in range(L)], dev) for st in stagings]
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(n_saves)]
    torch.cuda.synchronize()
    for i in range(n_saves):
        e_save0, e_saved, e_reuse = events[i]
        e_save0.record(s_save)
        hs.hs_save_kv_pages(cp, sps[i], L, bts[i], m, P, nb, err, stream=s_save)
        assert drv.cuLaunchHostFunc(ctypes.c_void_p(s_save.cuda_stream), usleep,
                                    ctypes.c_void_p(500000)) == 0
        e_saved.record(s_save)
        s_reuse.wait_event(e_saved)                      # the actual completion, not submission
        e_reuse.record(s_reuse)
        hs.hs_restore_kv_pages(npp, cp, L, bts[i], m, P, nb, err, stream=s_reuse)
    torch.cuda.synchronize()
    assert err.item() == 0
    cv, bv, nv = cache.view(L, nb, P), before.view(L, nb, P), new_pages.view(L, m, P)
    for i in range(n_saves):
        idx = bts[i].long()
        # saved bytes are the pages as they were before the dependent overwrite
        assert torch.equal(stagings[i].view(L, m, P), bv[:, idx].cpu())
        # the overwrite happened, and only after the delayed save had completed
        assert torch.equal(cv[:, idx], nv)
        assert events[i][0].elapsed_time(events[i][2]) >= 500.0


@pytest.mark.parametrize("where", ["device", "pinned_host"])
def test_fp8_rank_slices_restore_and_save(where):
    """FP8 KV pages (16 tokens x 8 KV heads x 128, one byte per element) moved as four
    tensor-parallel ranks' head slices (Table 1: TP=4, FP8 KV; Section 5.2: per-rank
    transfers): the four restores reassemble the oracle's full-page scatter bit for bit
    with untouched blocks poisoned, and each rank's save is its oracle gather."""
    dev = device()
    tokens, kvh, hd, TP = 16, 8, 128, 4
    rows, row_bytes = 2 * tokens, kvh * hd
    P = rows * row_bytes
    cb = row_bytes // TP
    L, nb, n_pages = 3, 72, 29
    rng = np.random.default_rng(17)
    full = [rng.integers(0, 256, size=n_pages * P, dtype=np.uint8) for _ in range(L)]
    bt = gen_block_table(23, 0, n_pages, nb)
    d_bt = torch.from_numpy(bt).to(dev)
    cache = torch.full((L, nb * P), POISON, dtype=torch.uint8, device=dev)
    cp = hs.ptr_array([cache[l] for l in range(L)], dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    keep = []
    for r in range(TP):
        st = np.stack([f.reshape(n_pages, rows, row_bytes)[:, :, r * cb:(r + 1) * cb].reshape(-1)
                       for f in full])
        t = torch.from_numpy(st)
        t = t.to(dev) if where == "device" else t.pin_memory()
        keep.append(t)
        hs.hs_restore_kv_page_slices(hs.ptr_array([t[l] for l in range(L)], dev), cp, L, d_bt,
                                     n_pages, P, rows, r * cb, cb, nb, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    want = [np.full(nb * P, POISON, np.uint8) for _ in range(L)]
    oracle.scatter_pages(full, want, bt, n_pages, P)
    got = cache.cpu().numpy()
    for l in range(L):
        assert np.array_equal(got[l], want[l]), l
    # each rank saves its slice back
    for r in range(TP):
        out = torch.full((L, n_pages * rows * cb), POISON, dtype=torch.uint8)
        out = out.to(dev) if where == "device" else out.pin_memory()
        hs.hs_save_kv_page_slices(cp, hs.ptr_array([out[l] for l in range(L)], dev), L, d_bt,
                                  n_pages, P, rows, r * cb, cb, nb, err)
        torch.cuda.synchronize()
        assert err.item() == 0
        ref = [np.zeros(n_pages * rows * cb, np.uint8) for _ in range(L)]
        oracle.gather_slices([got[l] for l in range(L)], ref, bt, n_pages, P, rows, r * cb, cb)
        o = out.cpu().numpy()
        for l in range(L):
            assert np.array_equal(o[l], ref[l]), (r, l)


def test_rank_slices_with_a_row_split_that_does_not_divide_the_block():
    """Slices of 3 x 16 bytes (a 3-head rank of 12 one-byte-per-dim heads... any split):
    the general per-vector path; restore then save round-trips bit for bit."""
    dev = device()
    L, nb, n_pages, rows, row_bytes, off, cb = 2, 20, 9, 24, 192, 64, 48
    P = rows * row_bytes
    rng = np.random.default_rng(19)
    st = torch.from_numpy(rng.integers(0, 256, size=(L, n_pages * rows * cb), dtype=np.uint8)).to(dev)
    cache = torch.full((L, nb * P), POISON, dtype=torch.uint8, device=dev)
    bt = torch.from_numpy(gen_block_table(24, 0, n_pages, nb)).to(dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    cp = hs.ptr_array([cache[l] for l in range(L)], dev)
    hs.hs_restore_kv_page_slices(hs.ptr_array([st[l] for l in range(L)], dev), cp, L, bt, n_pages,
                                 P, rows, off, cb, nb, err)
    back = torch.zeros_like(st)
    hs.hs_save_kv_page_slices(cp, hs.ptr_array([back[l] for l in range(L)], dev), L, bt, n_pages,
                              P, rows, off, cb, nb, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert torch.equal(back, st)
    want = [np.full(nb * P, POISON, np.uint8) for _ in range(L)]
    oracle.scatter_slices([st[l].cpu().numpy() for l in range(L)], want, bt.cpu().numpy(), n_pages,
                          P, rows, off, cb)
    got = cache.cpu().numpy()
    for l in range(L):
        assert np.array_equal(got[l], want[l])


@pytest.mark.parametrize("rows,row_bytes,off,cb", [
    (32, 2048, 1024, 1024),   # bf16 pages, two ranks: 2,048 vectors per slice (wide instantiation)
    (33, 1024, 256, 256),     # 528 vectors: just past the narrow instantiation's limit
    (32, 1024, 512, 256),     # 512 vectors: the narrow one's largest slice
    (1, 8192, 0, 8192),       # one contiguous 8 KiB row per page
])
def test_rank_slices_of_every_width_round_trip(rows, row_bytes, off, cb):
    """Slices on either side of the launch's choice between its narrow (at most 512 vectors per
    slice, eight CTAs per SM) and wide instantiations: the restore matches the oracle's slice
    scatter into a poisoned cache and the save gives the staging back bit for bit."""
    dev = device()
    L, nb, n_pages = 3, 40, 17
    P = rows * row_bytes
    rng = np.random.default_rng(rows * 7 + cb)
    st = torch.from_numpy(rng.integers(0, 256, size=(L, n_pages * rows * cb), dtype=np.uint8)).to(dev)
    cache = torch.full((L, nb * P), POISON, dtype=torch.uint8, device=dev)
    bt = torch.from_numpy(gen_block_table(25, rows, n_pages, nb)).to(dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    cp = hs.ptr_array([cache[l] for l in range(L)], dev)
    hs.hs_restore_kv_page_slices(hs.ptr_array([st[l] for l in range(L)], dev), cp, L, bt, n_pages,
                                 P, rows, off, cb, nb, err)
    back = torch.zeros_like(st)
    hs.hs_save_kv_page_slices(cp, hs.ptr_array([back[l] for l in range(L)], dev), L, bt, n_pages,
                              P, rows, off, cb, nb, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert torch.equal(back, st)
    want = [np.full(nb * P, POISON, np.uint8) for _ in range(L)]
    oracle.scatter_slices([st[l].cpu().numpy() for l in range(L)], want, bt.cpu().numpy(), n_pages,
                          P, rows, off, cb)
    got = cache.cpu().numpy()
    for l in range(L):
        assert np.array_equal(got[l], want[l]), l
