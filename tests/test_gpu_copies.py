"""KV page scatter and state copies on the GPU, bit-exact against the oracle.

The byte checks follow the paper's instrumented run (Section 5.3, Table 5):
destinations are poisoned before the restore, restored pages must equal the
staging bytes, untouched pages must stay poisoned, and the compared bytes
must be nonzero so that equality is not vacuous (the early all-zero tail
check of Section 3.1).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_15030_gb300 as hs
from hs_inputs import HYBRID12, KVSTRESS, TINY, gen_block_table, gen_kv_pages
from tests.gpu_helpers import device

pytestmark = pytest.mark.gpu
POISON = 0xFF


def _scatter_case(dev, n_layers, n_pages, page_bytes, num_blocks, seed):
    staging = [gen_kv_pages(seed, l, n_pages, page_bytes) for l in range(n_layers)]
    bt = gen_block_table(seed, 0, n_pages, num_blocks)
    d_st = [torch.from_numpy(s.reshape(-1)).to(dev) for s in staging]
    d_cache = [torch.full((num_blocks * page_bytes,), POISON, dtype=torch.uint8, device=dev)
               for _ in range(n_layers)]
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_kv_pages(hs.ptr_array(d_st, dev), hs.ptr_array(d_cache, dev), n_layers,
                           torch.from_numpy(bt).to(dev), n_pages, page_bytes, num_blocks, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    # oracle on host
    h_cache = [np.full(num_blocks * page_bytes, POISON, np.uint8) for _ in range(n_layers)]
    oracle.scatter_pages([s.reshape(-1) for s in staging], h_cache, bt, n_pages, page_bytes)
    for l in range(n_layers):
        got = d_cache[l].cpu().numpy()
        assert np.array_equal(got, h_cache[l]), l
        restored = got.reshape(num_blocks, page_bytes)[bt]
        assert restored.any()                                  # nonzero effective bytes
    untouched = np.setdiff1d(np.arange(num_blocks), bt)
    assert (d_cache[0].cpu().numpy().reshape(num_blocks, page_bytes)[untouched] == POISON).all()


def test_scatter_tiny_config():
    dev = device()
    _scatter_case(dev, TINY.n_full, 12, TINY.page_bytes, 40, seed=0)      # c = 192 -> 12 pages


@pytest.mark.parametrize("n_pages", [1, 7, 96, 287])
def test_scatter_hybrid_shapes(n_pages):
    dev = device()
    _scatter_case(dev, HYBRID12.n_full, n_pages, HYBRID12.page_bytes, 600, seed=n_pages)


def test_scatter_odd_page_size():
    dev = device()
    _scatter_case(dev, 2, 33, 16 * 37, 100, seed=3)          # page size not a power of two


def test_scatter_out_of_range_block_reports_and_skips():
    dev = device()
    P, nb = 4096, 8
    st = torch.arange(3 * P, dtype=torch.int32, device=dev).view(torch.uint8)[:3 * P].contiguous()
    cache = torch.full((nb * P,), POISON, dtype=torch.uint8, device=dev)
    bt = torch.tensor([2, 9, 5], dtype=torch.int32, device=dev)     # 9 is out of range
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_kv_pages(hs.ptr_array([st], dev), hs.ptr_array([cache], dev), 1, bt, 3, P, nb,
                           err)
    torch.cuda.synchronize()
    assert err.item() == hs.HS_DEVERR_BLOCK_OOB
    c = cache.cpu().numpy().reshape(nb, P)
    s = st.cpu().numpy().reshape(3, P)
    assert np.array_equal(c[2], s[0]) and np.array_equal(c[5], s[2])
    assert (np.delete(c, [2, 5], axis=0) == POISON).all()


def test_scatter_misaligned_layer_pointer_reports():
    dev = device()
    P = 256
    st = torch.ones(2 * P + 16, dtype=torch.uint8, device=dev)
    cache = torch.full((4 * P,), POISON, dtype=torch.uint8, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_kv_pages(hs.ptr_array([st.data_ptr() + 8], dev), hs.ptr_array([cache], dev), 1,
                           torch.tensor([0, 1], dtype=torch.int32, device=dev), 2, P, 4, err)
    torch.cuda.synchronize()
    assert err.item() == hs.HS_DEVERR_MISALIGNED
    assert (cache.cpu().numpy() == POISON).all()


def test_scatter_full_size_kv_stress_sampled():
    """48 layers x 256 pages x 64 KiB (one 4096-token request of the KV stress
    workload) into a 2 GiB-per-layer-set cache; every page is compared."""
    dev = device()
    L, n_pages, P = KVSTRESS.n_full, 4096 // KVSTRESS.page, KVSTRESS.page_bytes
    nb = 640
    st = torch.empty((L, n_pages * P), dtype=torch.uint8, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    st.view(torch.int32).random_(generator=g)
    cache = torch.full((L, nb * P), POISON, dtype=torch.uint8, device=dev)
    bt = torch.from_numpy(gen_block_table(4, 0, n_pages, nb)).to(dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_kv_pages(hs.ptr_array([st[l] for l in range(L)], dev),
                           hs.ptr_array([cache[l] for l in range(L)], dev), L, bt, n_pages, P, nb,
                           err)
    torch.cuda.synchronize()
    assert err.item() == 0
    c = cache.view(L, nb, P)
    s = st.view(L, n_pages, P)
    assert torch.equal(c[:, bt.long()], s)
    mask = torch.ones(nb, dtype=torch.bool, device=dev)
    mask[bt.long()] = False
    assert bool((c[:, mask] == POISON).all())


@pytest.mark.parametrize("fn", ["hs_restore_state", "hs_checkpoint_states"])
def test_state_copy_bit_exact(fn):
    dev = device()
    n, fe = 9, HYBRID12.n_heads * HYBRID12.d * HYBRID12.d      # nine 1 MiB layer states
    rng = np.random.default_rng(3)
    src_h = [rng.standard_normal(fe).astype(np.float32) for _ in range(n)]
    src_h[0][:7] = [np.nan, -0.0, np.inf, -np.inf, 1e-45, 3.4e38, -1e-38]   # every bit pattern kind
    src = [torch.from_numpy(x).to(dev) for x in src_h]
    dst = [torch.full((fe,), -7.0, device=dev) for _ in range(n)]
    getattr(hs, fn)(hs.ptr_array(src, dev), hs.ptr_array(dst, dev), n, fe)
    torch.cuda.synchronize()
    ref = [np.full(fe, -7.0, np.float32) for _ in range(n)]
    oracle.copy_slots(src_h, ref, fe)
    for d, r in zip(dst, ref):
        assert np.array_equal(d.cpu().numpy().view(np.uint32), r.view(np.uint32))


def test_state_copy_unaligned_and_ragged():
    dev = device()
    fe = 16384 * 3 + 5                                  # several pieces and a ragged tail
    base = torch.arange(fe + 3, dtype=torch.float32, device=dev)
    dst = torch.zeros(fe + 3, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_state(hs.ptr_array([base.data_ptr() + 4], dev),
                        hs.ptr_array([dst.data_ptr() + 8], dev), 1, fe, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert torch.equal(dst[2:2 + fe], base[1:1 + fe])
    assert dst[0].item() == 0 and dst[1].item() == 0 and dst[-1].item() == 0


def test_state_copy_null_slot_reports():
    dev = device()
    a = torch.ones(64, device=dev)
    b = torch.zeros(64, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_state(hs.ptr_array([a, 0], dev), hs.ptr_array([b, b], dev), 2, 64, err)
    torch.cuda.synchronize()
    assert err.item() == hs.HS_DEVERR_NULL
    assert torch.equal(b, a)


def test_scatter_from_pinned_host_staging():
    """Staging pages in pinned host memory (device-accessible): the scatter reads them
    directly over the host link, as the paper's CPU cache tier is read (Section 5.5)."""
    dev = device()
    L, n_pages, P, nb = 3, 40, HYBRID12.page_bytes, 128
    st = torch.empty((L, n_pages * P), dtype=torch.uint8).pin_memory()
    st.view(torch.int32).random_(generator=torch.Generator().manual_seed(11))
    cache = torch.full((L, nb * P), POISON, dtype=torch.uint8, device=dev)
    bt = torch.from_numpy(gen_block_table(12, 0, n_pages, nb)).to(dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_kv_pages(hs.ptr_array([st[l] for l in range(L)], dev),
                           hs.ptr_array([cache[l] for l in range(L)], dev), L, bt, n_pages, P, nb,
                           err)
    torch.cuda.synchronize()
    assert err.item() == 0
    c = cache.view(L, nb, P).cpu()
    assert torch.equal(c[:, bt.long().cpu()], st.view(L, n_pages, P))
    mask = torch.ones(nb, dtype=torch.bool)
    mask[bt.long().cpu()] = False
    assert bool((c[:, mask] == POISON).all())


def _request_case(dev, n_layers, n_pages, page_bytes, num_blocks, n_slots, floats_each, seed):
    staging = [gen_kv_pages(seed, l, n_pages, page_bytes) for l in range(n_layers)]
    bt = gen_block_table(seed, 0, n_pages, num_blocks)
    rng = np.random.default_rng(seed)
    src_h = [rng.standard_normal(floats_each).astype(np.float32) for _ in range(n_slots)]
    d_st = [torch.from_numpy(s.reshape(-1)).to(dev) for s in staging]
    d_cache = [torch.full((num_blocks * page_bytes,), POISON, dtype=torch.uint8, device=dev)
               for _ in range(n_layers)]
    src = [torch.from_numpy(x).to(dev) for x in src_h]
    dst = [torch.full((floats_each,), -7.0, device=dev) for _ in range(n_slots)]
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_request(hs.ptr_array(d_st, dev), hs.ptr_array(d_cache, dev), n_layers,
                          torch.from_numpy(bt).to(dev), n_pages, page_bytes, num_blocks,
                          hs.ptr_array(src, dev), hs.ptr_array(dst, dev), n_slots, floats_each, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    h_cache = [np.full(num_blocks * page_bytes, POISON, np.uint8) for _ in range(n_layers)]
    if n_pages:
        oracle.scatter_pages([s.reshape(-1) for s in staging], h_cache, bt, n_pages, page_bytes)
    for l in range(n_layers):
        assert np.array_equal(d_cache[l].cpu().numpy(), h_cache[l]), l
    ref = [np.full(floats_each, -7.0, np.float32) for _ in range(n_slots)]
    if floats_each:
        oracle.copy_slots(src_h, ref, floats_each)
    for d, r in zip(dst, ref):
        assert np.array_equal(d.cpu().numpy().view(np.uint32), r.view(np.uint32))


@pytest.mark.parametrize("n_pages", [1, 96, 287])
def test_restore_request_hybrid_shapes(n_pages):
    """The one-launch restore of a hybrid request (Section 2.1, Section 5.2): the
    3 attention layers' pages and the 9 linear layers' 1 MiB states, bit-exact
    against the oracle's scatter and slot copy."""
    dev = device()
    _request_case(dev, HYBRID12.n_full, n_pages, HYBRID12.page_bytes, 600, 9,
                  HYBRID12.n_heads * HYBRID12.d * HYBRID12.d, seed=n_pages)


@pytest.mark.parametrize("case", [dict(n_pages=0), dict(n_layers=0), dict(n_slots=0),
                                  dict(floats_each=0), dict(floats_each=16 * 4100),
                                  dict(page_bytes=16 * 37, n_pages=33)])
def test_restore_request_empty_and_ragged_parts(case):
    dev = device()
    a = dict(n_layers=2, n_pages=5, page_bytes=4096, num_blocks=64, n_slots=3,
             floats_each=4096 * 4)
    a.update(case)
    _request_case(dev, a["n_layers"], a["n_pages"], a["page_bytes"], a["num_blocks"],
                  a["n_slots"], a["floats_each"], seed=11)


def test_restore_request_reports_and_skips_bad_units():
    """An out-of-range block, a NULL state slot and a misaligned state slot are
    reported and skipped; every other unit is still copied."""
    dev = device()
    P, nb, fe = 4096, 8, 16384 * 2 + 4
    st = torch.arange(3 * P // 4, dtype=torch.int32, device=dev).view(torch.uint8).contiguous()
    cache = torch.full((nb * P,), POISON, dtype=torch.uint8, device=dev)
    bt = torch.tensor([2, 9, 5], dtype=torch.int32, device=dev)
    a = torch.randn(fe, device=dev)
    b = torch.randn(fe + 4, device=dev)
    good = torch.zeros(fe, device=dev)
    nul = torch.zeros(fe, device=dev)
    mis = torch.zeros(fe + 4, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_request(hs.ptr_array([st], dev), hs.ptr_array([cache], dev), 1, bt, 3, P, nb,
                          hs.ptr_array([a, 0, b.data_ptr() + 4], dev),
                          hs.ptr_array([good, nul, mis], dev), 3, fe, err)
    torch.cuda.synchronize()
    assert err.item() in (hs.HS_DEVERR_BLOCK_OOB, hs.HS_DEVERR_NULL, hs.HS_DEVERR_MISALIGNED)
    c = cache.cpu().numpy().reshape(nb, P)
    s = st.cpu().numpy().reshape(3, P)
    assert np.array_equal(c[2], s[0]) and np.array_equal(c[5], s[2])
    assert (np.delete(c, [2, 5], axis=0) == POISON).all()
    assert torch.equal(good, a)
    assert not nul.any() and not mis.any()
    # each kind alone gives its own code
    for srcs, dsts, table, code in [([a], [good], [2, 9, 5], hs.HS_DEVERR_BLOCK_OOB),
                                    ([0], [good], [2, 1, 5], hs.HS_DEVERR_NULL),
                                    ([b.data_ptr() + 4], [mis], [2, 1, 5],
                                     hs.HS_DEVERR_MISALIGNED)]:
        err.zero_()
        hs.hs_restore_request(hs.ptr_array([st], dev), hs.ptr_array([cache], dev), 1,
                              torch.tensor(table, dtype=torch.int32, device=dev), 3, P, nb,
                              hs.ptr_array(srcs, dev), hs.ptr_array(dsts, dev), 1, fe, err)
        torch.cuda.synchronize()
        assert err.item() == code


def test_restore_request_from_pinned_host():
    """Staging pages and checkpoint slots in pinned host memory, read by the kernel
    over the C2C link (a restore straight from the host tier)."""
    dev = device()
    L, n_pages, P, nb, n_slots, fe = 3, 40, HYBRID12.page_bytes, 200, 9, 16384 * 4
    staging = [gen_kv_pages(5, l, n_pages, P).reshape(-1) for l in range(L)]
    h_st = [torch.from_numpy(s).pin_memory() for s in staging]
    rng = np.random.default_rng(5)
    src_h = [rng.standard_normal(fe).astype(np.float32) for _ in range(n_slots)]
    h_src = [torch.from_numpy(x).pin_memory() for x in src_h]
    bt = gen_block_table(5, 0, n_pages, nb)
    cache = [torch.full((nb * P,), POISON, dtype=torch.uint8, device=dev) for _ in range(L)]
    dst = [torch.zeros(fe, device=dev) for _ in range(n_slots)]
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_restore_request(hs.ptr_array(h_st, dev), hs.ptr_array(cache, dev), L,
                          torch.from_numpy(bt).to(dev), n_pages, P, nb, hs.ptr_array(h_src, dev),
                          hs.ptr_array(dst, dev), n_slots, fe, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    h_cache = [np.full(nb * P, POISON, np.uint8) for _ in range(L)]
    oracle.scatter_pages(staging, h_cache, bt, n_pages, P)
    for l in range(L):
        assert np.array_equal(cache[l].cpu().numpy(), h_cache[l])
    for d, r in zip(dst, src_h):
        assert np.array_equal(d.cpu().numpy().view(np.uint32), r.view(np.uint32))
