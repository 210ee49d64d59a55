"""Host-only checks of the C-ABI library (no GPU needed).

* libhs.so loads and exports every function include/*.h declares;
* hs_align_prefix (host integer code) matches the oracle bit-exactly;
* every argument error is reported before any CUDA call.
"""
import ctypes
import glob
import os
import re

import numpy as np
import pytest

import oracle
import paper_2609_15030_gb300 as hs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_15030_gb300 import build
    build.build()


def _declared():
    names = set()
    for h in sorted(glob.glob(os.path.join(ROOT, "include", "*.h"))):
        txt = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"\b(hs_[a-z0-9_]+)\s*\(", txt))
    return sorted(names)


def test_exports_every_declared_symbol():
    import ctypes
    lib = ctypes.CDLL(hs.LIB_PATH)
    names = _declared()
    assert "hs_linattn_prefill_from_state" in names and len(names) >= 8
    for n in names:
        assert hasattr(lib, n), n
    assert set(hs.EXPORTED) <= set(names)


def test_status_strings_and_version():
    for s in range(7):
        assert hs.hs_status_string(s).startswith("HS_")
    assert "unknown" in hs.hs_status_string(99)
    assert hs.hs_version() >= 100


def _rows():
    out = []
    for line in open(os.path.join(ROOT, "tests", "golden", "table4_alignment.txt")):
        line = line.strip()
        if line and not line.startswith("#"):
            out.append([int(x) for x in line.split()])
    return out


def test_align_table4():
    C = 1792
    for N, _, _, B_after, suffix in _rows():
        c, npg, tail = hs.hs_align_prefix(N, N, list(range(C, N + 1, C)), 16)
        assert (c, tail) == (B_after, suffix)
        assert npg == c // 16


def test_align_matches_oracle_bit_exact():
    rng = np.random.default_rng(77)
    for _ in range(4000):
        N = int(rng.integers(1, 400))
        hit = int(rng.integers(0, N + 1))
        P = int(rng.choice([1, 2, 16, 32]))
        avail = sorted(set(int(x) for x in rng.integers(0, N + 50, size=int(rng.integers(0, 20)))))
        assert hs.hs_align_prefix(N, hit, avail, P) == oracle.align_prefix(N, hit, avail, P)


def test_align_config_lengths():
    # sweep / hybrid / long-context lengths, complete and partial (L-37) hits
    for C, P, Ls in ((512, 16, range(512, 4609, 512)), (256, 16, range(512, 4609, 512)),
                     (512, 32, (16384, 32768, 65536))):
        for L in Ls:
            for hit in (L, L - 37):
                av = list(range(C, L + 1, C))
                assert hs.hs_align_prefix(L, hit, av, P) == oracle.align_prefix(L, hit, av, P)


@pytest.mark.parametrize("args", [
    (0, 0, [], 16), (10, 11, [], 16), (10, -1, [], 16), (10, 5, [], 0),
    (10, 10, [4, 4], 2), (10, 10, [8, 4], 2), (10, 10, [-4], 2)])
def test_align_invalid(args):
    with pytest.raises(hs.HsError) as e:
        hs.hs_align_prefix(*args)
    assert e.value.status == hs.HS_ERR_INVALID_ARG


def test_num_checkpoints_matches_oracle():
    rng = np.random.default_rng(5)
    for _ in range(500):
        B = int(rng.integers(1, 6))
        pos0 = rng.integers(0, 5000, size=B)
        nt = rng.integers(0, 3000, size=B)
        C = int(rng.choice([0, 64, 256, 512]))
        want = sum(oracle.n_checkpoints(int(p), int(n), C) for p, n in zip(pos0, nt))
        assert hs.hs_linattn_num_checkpoints(pos0, nt, C) == want


FAKE = 1 << 20        # a 16-byte aligned non-null address that is never dereferenced


@pytest.mark.parametrize("fn", ["hs_restore_kv_pages", "hs_save_kv_pages"])
def test_kv_pages_host_validation(fn):
    def call(**kw):
        a = dict(staging_layers=FAKE, cache_layers=FAKE, n_layers=1, block_table=FAKE, n_pages=1,
                 page_bytes=64, num_blocks=4, d_err=None, stream=0)
        a.update(kw)
        getattr(hs, fn)(**a)
    for kw, code in [(dict(n_layers=-1), hs.HS_ERR_INVALID_ARG),
                     (dict(page_bytes=0), hs.HS_ERR_INVALID_ARG),
                     (dict(page_bytes=24), hs.HS_ERR_MISALIGNED),
                     (dict(staging_layers=None), hs.HS_ERR_INVALID_ARG),
                     (dict(block_table=None), hs.HS_ERR_INVALID_ARG),
                     (dict(n_pages=5, num_blocks=4), hs.HS_ERR_INVALID_ARG)]:
        with pytest.raises(hs.HsError) as e:
            call(**kw)
        assert e.value.status == code, kw
    call(n_layers=0)          # no-ops return OK without touching the GPU
    call(n_pages=0)


@pytest.mark.parametrize("fn", ["hs_restore_kv_page_slices", "hs_save_kv_page_slices"])
def test_kv_page_slices_host_validation(fn):
    def call(**kw):
        a = dict(staging_layers=FAKE, cache_layers=FAKE, n_layers=1, block_table=FAKE, n_pages=1,
                 page_bytes=1024, rows=4, col_off=64, col_bytes=64, num_blocks=4, d_err=None,
                 stream=0)
        a.update(kw)
        if fn == "hs_save_kv_page_slices":
            a["cache_layers"], a["staging_layers"] = a.pop("cache_layers"), a.pop("staging_layers")
        getattr(hs, fn)(**a)
    for kw, code in [(dict(rows=0), hs.HS_ERR_INVALID_ARG),
                     (dict(rows=3), hs.HS_ERR_INVALID_ARG),            # 3 does not divide 1024
                     (dict(col_off=224, col_bytes=64), hs.HS_ERR_INVALID_ARG),   # past the row
                     (dict(col_bytes=0), hs.HS_ERR_INVALID_ARG),
                     (dict(col_off=8), hs.HS_ERR_MISALIGNED),
                     (dict(col_bytes=40), hs.HS_ERR_MISALIGNED),
                     (dict(page_bytes=1032, rows=2), hs.HS_ERR_MISALIGNED),
                     (dict(block_table=None), hs.HS_ERR_INVALID_ARG),
                     (dict(n_pages=5, num_blocks=4), hs.HS_ERR_INVALID_ARG)]:
        with pytest.raises(hs.HsError) as e:
            call(**kw)
        assert e.value.status == code, kw
    call(n_layers=0)
    call(n_pages=0)


def test_restore_request_host_validation():
    def call(**kw):
        a = dict(staging_layers=FAKE, cache_layers=FAKE, n_layers=1, block_table=FAKE, n_pages=1,
                 page_bytes=64, num_blocks=4, src_slots=FAKE, dst_slots=FAKE, n_slots=2,
                 floats_each=16, d_err=None, stream=0)
        a.update(kw)
        hs.hs_restore_request(**a)
    for kw, code in [(dict(n_layers=-1), hs.HS_ERR_INVALID_ARG),
                     (dict(n_slots=-1), hs.HS_ERR_INVALID_ARG),
                     (dict(floats_each=-4), hs.HS_ERR_INVALID_ARG),
                     (dict(page_bytes=0), hs.HS_ERR_INVALID_ARG),
                     (dict(page_bytes=24), hs.HS_ERR_MISALIGNED),
                     (dict(floats_each=18), hs.HS_ERR_MISALIGNED),
                     (dict(staging_layers=None), hs.HS_ERR_INVALID_ARG),
                     (dict(block_table=None), hs.HS_ERR_INVALID_ARG),
                     (dict(src_slots=None), hs.HS_ERR_INVALID_ARG),
                     (dict(n_pages=5, num_blocks=4), hs.HS_ERR_INVALID_ARG)]:
        with pytest.raises(hs.HsError) as e:
            call(**kw)
        assert e.value.status == code, kw
    # both parts empty: OK without touching the GPU (a missing part's pointers are not read)
    call(n_layers=0, n_slots=0)
    call(n_pages=0, staging_layers=None, floats_each=0, src_slots=None)


def test_state_copy_host_validation():
    for fn in (hs.hs_restore_state, hs.hs_checkpoint_states):
        with pytest.raises(hs.HsError):
            fn(FAKE, FAKE, -1, 16, stream=0)
        with pytest.raises(hs.HsError):
            fn(None, FAKE, 2, 16, stream=0)
        fn(FAKE, FAKE, 0, 16, stream=0)
        fn(None, None, 3, 0, stream=0)


def test_prefill_host_validation():
    def call(shape_kw=None, **kw):
        sk = dict(batch=1, n_heads=2, d_k=64, d_v=64, max_tokens=8)
        sk.update(shape_kw or {})
        a = dict(q=FAKE, k=FAKE, v=FAKE, log_g=FAKE, o=FAKE, state=FAKE, pos0=[0], n_tokens=[8],
                 ckpt_interval=64, ckpt_slots=None, d_err=None, stream=0)
        a.update(kw)
        hs.hs_linattn_prefill_from_state(hs.make_shape(**sk), **a)
    cases = [
        (dict(shape_kw=dict(d_k=96, d_v=96)), hs.HS_ERR_UNSUPPORTED),
        (dict(shape_kw=dict(d_k=64, d_v=128)), hs.HS_ERR_UNSUPPORTED),
        (dict(shape_kw=dict(batch=hs.HS_MAX_BATCH + 1), pos0=[0] * (hs.HS_MAX_BATCH + 1),
          n_tokens=[1] * (hs.HS_MAX_BATCH + 1)),
         hs.HS_ERR_UNSUPPORTED),
        (dict(ckpt_interval=96), hs.HS_ERR_UNSUPPORTED),
        (dict(ckpt_interval=-64), hs.HS_ERR_INVALID_ARG),
        (dict(shape_kw=dict(n_heads=0)), hs.HS_ERR_INVALID_ARG),
        (dict(n_tokens=[9]), hs.HS_ERR_INVALID_ARG),
        (dict(pos0=[-1]), hs.HS_ERR_INVALID_ARG),
        (dict(q=None), hs.HS_ERR_INVALID_ARG),
        (dict(state=None), hs.HS_ERR_INVALID_ARG),
        (dict(o=FAKE + 4), hs.HS_ERR_MISALIGNED),
        (dict(log_g=FAKE + 8), hs.HS_ERR_MISALIGNED),
        (dict(shape_kw=dict(kernel=7)), hs.HS_ERR_INVALID_ARG),
        (dict(shape_kw=dict(kernel=hs.HS_LINATTN_SINGLE_TOKEN), n_tokens=[2]),
         hs.HS_ERR_UNSUPPORTED),                       # the single-token kernel: n_tokens <= 1
    ]
    for kw, code in cases:
        with pytest.raises(hs.HsError) as e:
            call(**kw)
        assert e.value.status == code, kw
    call(shape_kw=dict(batch=0), pos0=[], n_tokens=[])    # empty batch: OK, nothing launched
    call(n_tokens=[0], q=None, k=None, v=None, log_g=None, o=None)   # empty tails: OK


def test_stalled_prefill_hook_host_validation():
    """The failure-detection hook exists in the tensor-core kernel only; other kernel
    choices are refused on the host, and its argument checks are the prefill's."""
    a = dict(q=FAKE, k=FAKE, v=FAKE, log_g=FAKE, o=FAKE, state=FAKE, pos0=[0], n_tokens=[8],
             ckpt_interval=64, ckpt_slots=None, d_err=None, stream=0)
    for kernel in (hs.HS_LINATTN_AUTO, hs.HS_LINATTN_RECURRENT, hs.HS_LINATTN_SINGLE_TOKEN):
        with pytest.raises(hs.HsError) as e:
            hs.hs_test_prefill_stalled(hs.make_shape(1, 2, 128, 128, 8, kernel), **a)
        assert e.value.status == hs.HS_ERR_UNSUPPORTED
    with pytest.raises(hs.HsError) as e:
        hs.hs_test_prefill_stalled(hs.make_shape(1, 2, 128, 128, 8, hs.HS_LINATTN_CHUNKED_TC),
                                   **dict(a, pos0=[-1]))
    assert e.value.status == hs.HS_ERR_INVALID_ARG


def test_packed_prefill_host_validation():
    def call(**kw):
        a = dict(q=FAKE, k=FAKE, v=FAKE, log_g=FAKE, o=FAKE, state=FAKE, pos0=[0, 5],
                 n_tokens=[8, 3], cu_rows=[0, 8, 11], ckpt_interval=64, ckpt_slots=None,
                 d_err=None, stream=0)
        a.update(kw)
        hs.hs_linattn_prefill_packed(hs.make_shape(2, 2, 64, 64, 0), **a)
    for kw, code in [(dict(cu_rows=[0, 8, 10]), hs.HS_ERR_INVALID_ARG),     # problem 1 too long
                     (dict(cu_rows=[0, 12, 11]), hs.HS_ERR_INVALID_ARG),    # not monotone
                     (dict(cu_rows=[-1, 8, 11]), hs.HS_ERR_INVALID_ARG),
                     (dict(cu_rows=[0, 2 ** 31 - 2, 2 ** 31 + 8]), hs.HS_ERR_UNSUPPORTED),
                     (dict(n_tokens=[9, 3]), hs.HS_ERR_INVALID_ARG)]:
        with pytest.raises(hs.HsError) as e:
            call(**kw)
        assert e.value.status == code, kw
    lib = hs.load()
    shape = hs.make_shape(2, 2, 64, 64, 0)
    p0 = (ctypes.c_int64 * 2)(0, 5)
    nt = (ctypes.c_int32 * 2)(8, 3)
    rc = lib.hs_linattn_prefill_packed(ctypes.byref(shape), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE,
                                       ctypes.addressof(p0), ctypes.addressof(nt), None, 64, None,
                                       None, None)
    assert rc == hs.HS_ERR_INVALID_ARG                       # cu_rows is required
    call(n_tokens=[0, 0], q=None, k=None, v=None, log_g=None, o=None)   # empty tails: OK


def test_scan_prefill_host_validation():
    """hs_linattn_prefill_scan: the prefill's argument checks plus its workspace, and the
    workspace size it asks for, all on the host before any CUDA call."""
    sh = hs.make_shape(2, 4, 128, 128, 200)
    # two states per segment: problem 0 spans [100, 300) -> 4 segments, problem 1 [0, 64) -> 1
    assert hs.hs_linattn_scan_workspace_bytes(sh, [100, 0], [200, 64]) == 2 * 5 * 4 * 128 * 128 * 4
    assert hs.hs_linattn_scan_workspace_bytes(sh, [0, 0], [0, 0]) == 0
    need = 2 * 5 * 4 * 128 * 128 * 4

    def call(shape=sh, **kw):
        a = dict(q=FAKE, k=FAKE, v=FAKE, log_g=FAKE, o=FAKE, state=FAKE, pos0=[100, 0],
                 n_tokens=[200, 64], ckpt_interval=64, ckpt_slots=None, workspace=FAKE,
                 workspace_bytes=need, d_err=None, stream=0)
        a.update(kw)
        hs.hs_linattn_prefill_scan(shape, **a)
    cases = [
        (dict(workspace=None), hs.HS_ERR_INVALID_ARG),
        (dict(workspace_bytes=need - 16), hs.HS_ERR_INVALID_ARG),
        (dict(workspace=FAKE + 8), hs.HS_ERR_MISALIGNED),
        (dict(shape=hs.make_shape(2, 4, 128, 128, 200, hs.HS_LINATTN_RECURRENT)),
         hs.HS_ERR_UNSUPPORTED),
        (dict(shape=hs.make_shape(2, 4, 96, 96, 200)), hs.HS_ERR_UNSUPPORTED),
        (dict(n_tokens=[201, 64]), hs.HS_ERR_INVALID_ARG),
        (dict(pos0=[-1, 0]), hs.HS_ERR_INVALID_ARG),
        (dict(ckpt_interval=96), hs.HS_ERR_UNSUPPORTED),
        (dict(state=None), hs.HS_ERR_INVALID_ARG),
        (dict(o=FAKE + 4), hs.HS_ERR_MISALIGNED),
    ]
    for kw, code in cases:
        with pytest.raises(hs.HsError) as e:
            call(**kw)
        assert e.value.status == code, kw
    call(n_tokens=[0, 0], q=None, workspace=None, workspace_bytes=0)   # nothing to compute: OK
    # (segment, head) units are 32-bit: 40,000 segments x 65,536 heads is refused
    big = hs.make_shape(1, 65536, 128, 128, 64 * 40000)
    with pytest.raises(hs.HsError) as e:
        hs.hs_linattn_scan_workspace_bytes(big, [0], [64 * 40000])
    assert e.value.status == hs.HS_ERR_UNSUPPORTED


def test_noalloc_scan_rejects_on_the_host():
    """hs_linattn_prefill_scan_noalloc: calls whose workspace would exceed the fixed 16 MiB
    are refused with HS_ERR_TOO_LARGE, and argument errors are reported, before any CUDA call
    (this host has no GPU, so a call that reached the CUDA runtime would fail otherwise)."""
    assert hs.HS_NOALLOC_SCRATCH_BYTES == 16 << 20
    sh = hs.make_shape(1, 16, 128, 128, 1024)
    # 512 tokens from 4096: 8 segments x 16 heads x 2 states of 64 KiB = exactly the limit
    assert hs.hs_linattn_scan_workspace_bytes(sh, [4096], [512]) == hs.HS_NOALLOC_SCRATCH_BYTES

    def call(shape=sh, **kw):
        a = dict(q=FAKE, k=FAKE, v=FAKE, log_g=FAKE, o=FAKE, state=FAKE, pos0=[4096],
                 n_tokens=[512], ckpt_interval=512, ckpt_slots=None, d_err=None, stream=0)
        a.update(kw)
        hs.hs_linattn_prefill_scan_noalloc(shape, **a)
    cases = [
        (dict(n_tokens=[513]), hs.HS_ERR_TOO_LARGE),            # one more segment
        (dict(pos0=[4095]), hs.HS_ERR_TOO_LARGE),               # off the grid: 9 segments
        (dict(shape=hs.make_shape(2, 16, 128, 128, 1024), pos0=[0, 0], n_tokens=[256, 320]),
         hs.HS_ERR_TOO_LARGE),
        (dict(shape=hs.make_shape(1, 16, 128, 128, 1024, hs.HS_LINATTN_RECURRENT)),
         hs.HS_ERR_UNSUPPORTED),
        (dict(n_tokens=[1025]), hs.HS_ERR_INVALID_ARG),
        (dict(ckpt_interval=-64), hs.HS_ERR_INVALID_ARG),
        (dict(ckpt_interval=96), hs.HS_ERR_UNSUPPORTED),
        (dict(q=None), hs.HS_ERR_INVALID_ARG),
        (dict(state=None, o=FAKE + 4), hs.HS_ERR_INVALID_ARG),
        (dict(o=FAKE + 4), hs.HS_ERR_MISALIGNED),
    ]
    for kw, code in cases:
        with pytest.raises(hs.HsError) as e:
            call(**kw)
        assert e.value.status == code, kw
    assert "fixed workspace" in hs.hs_status_string(hs.HS_ERR_TOO_LARGE)
    call(n_tokens=[0], q=None, state=None)      # nothing to compute: OK, no set-up


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    import importlib
    mod = importlib.import_module("paper_2609_15030_gb300")
    monkeypatch.setattr(mod, "LIB_PATH", str(tmp_path / "absent.so"))
    monkeypatch.setattr(mod, "_lib", None)
    with pytest.raises(RuntimeError):
        mod.hs_version()


def test_c_client_compiles_links_and_runs(tmp_path):
    """The public headers are C: a C11 client (tests/c_client/hs_client.c) compiles with
    -Wall -Werror, links against libhs.so and runs its host-only checks."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    cuda_inc = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")
    exe = tmp_path / "hs_client"
    libdir = os.path.dirname(hs.LIB_PATH)
    subprocess.run([gcc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
                    "-I", cuda_inc, os.path.join(ROOT, "tests", "c_client", "hs_client.c"),
                    "-o", str(exe), "-L", libdir, "-l:libhs.so", f"-Wl,-rpath,{libdir}"], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "FAIL" not in r.stdout and r.stdout.count("ok ") >= 12
