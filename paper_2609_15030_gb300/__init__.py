"""Python binding of libhs (checkpoint-aligned restore-and-resume, sm_103a).

Argument marshalling only: every function forwards to the C entry point of
the same name in ``libhs.so`` (declared in ``include/hs.h``); all GPU work
runs in the library's kernels.  Tensors are accepted wherever the C call
takes a pointer (their ``data_ptr()`` is passed); plain ints are passed as
addresses.  A non-OK status raises ``HsError``.

The library is built in-tree by ``paper_2609_15030_gb300.build.build()``.
If ``libhs.so`` is missing, every call raises: there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libhs.so")

HS_OK = 0
HS_ERR_INVALID_ARG = 1
HS_ERR_MISALIGNED = 2
HS_ERR_UNSUPPORTED = 3
HS_ERR_CUDA = 4
HS_ERR_DEVICE_CHECK = 5
HS_ERR_TOO_LARGE = 6

HS_DEVERR_NONE = 0
HS_DEVERR_BLOCK_OOB = 1
HS_DEVERR_MISALIGNED = 2
HS_DEVERR_NULL = 3
HS_DEVERR_TIMEOUT = 4

HS_MAX_BATCH = 384
HS_CHUNK = 64
HS_SHORT_SEGMENT = 8
HS_NOALLOC_SCRATCH_BYTES = 16 << 20

HS_LINATTN_AUTO = 0
HS_LINATTN_RECURRENT = 1
HS_LINATTN_CHUNKED_TC = 2
HS_LINATTN_SINGLE_TOKEN = 3

EXPORTED = ("hs_status_string", "hs_version", "hs_align_prefix", "hs_restore_kv_pages",
            "hs_save_kv_pages", "hs_restore_kv_page_slices", "hs_save_kv_page_slices",
            "hs_restore_state", "hs_checkpoint_states", "hs_linattn_prefill_from_state",
            "hs_linattn_num_checkpoints", "hs_linattn_prefill_packed", "hs_restore_request",
            "hs_test_prefill_stalled", "hs_linattn_prefill_scan", "hs_linattn_scan_workspace_bytes",
            "hs_linattn_prefill_scan_noalloc")


class HsError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {hs_status_string(status)}")


class hs_linattn_shape(C.Structure):
    _fields_ = [("batch", C.c_int32), ("n_heads", C.c_int32), ("d_k", C.c_int32),
                ("d_v", C.c_int32), ("max_tokens", C.c_int64), ("kernel", C.c_int32),
                ("reserved", C.c_int32)]


_lock = threading.Lock()
_lib = None


def load() -> C.CDLL:
    """Load libhs.so; raises if it has not been built (no fallback path exists)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"{LIB_PATH} not found: build it with "
                                   "paper_2609_15030_gb300.build.build()")
            L = C.CDLL(LIB_PATH)
            vp, i32, i64 = C.c_void_p, C.c_int32, C.c_int64
            L.hs_status_string.argtypes = [C.c_int]
            L.hs_status_string.restype = C.c_char_p
            L.hs_version.argtypes = []
            L.hs_version.restype = i32
            L.hs_align_prefix.argtypes = [i64, i64, vp, i32, i32, vp, vp, vp]
            L.hs_restore_kv_pages.argtypes = [vp, vp, i32, vp, i32, i64, i64, vp, vp]
            L.hs_save_kv_pages.argtypes = [vp, vp, i32, vp, i32, i64, i64, vp, vp]
            L.hs_restore_request.argtypes = [vp, vp, i32, vp, i32, i64, i64, vp, vp, i32, i64, vp, vp]
            for name in ("hs_restore_kv_page_slices", "hs_save_kv_page_slices"):
                getattr(L, name).argtypes = [vp, vp, i32, vp, i32, i64, i32, i64, i64, i64, vp, vp]
            L.hs_restore_state.argtypes = [vp, vp, i32, i64, vp, vp]
            L.hs_checkpoint_states.argtypes = [vp, vp, i32, i64, vp, vp]
            L.hs_linattn_prefill_from_state.argtypes = [C.POINTER(hs_linattn_shape), vp, vp, vp,
                                                        vp, vp, vp, vp, vp, i32, vp, vp, vp]
            L.hs_linattn_num_checkpoints.argtypes = [i32, vp, vp, i32, vp]
            L.hs_linattn_prefill_packed.argtypes = [C.POINTER(hs_linattn_shape), vp, vp, vp, vp,
                                                    vp, vp, vp, vp, vp, i32, vp, vp, vp]
            L.hs_test_prefill_stalled.argtypes = L.hs_linattn_prefill_from_state.argtypes
            L.hs_linattn_prefill_scan.argtypes = [C.POINTER(hs_linattn_shape), vp, vp, vp, vp, vp,
                                                  vp, vp, vp, i32, vp, vp, i64, vp, vp]
            L.hs_linattn_scan_workspace_bytes.argtypes = [C.POINTER(hs_linattn_shape), vp, vp, vp]
            L.hs_linattn_prefill_scan_noalloc.argtypes = [C.POINTER(hs_linattn_shape), vp, vp, vp,
                                                          vp, vp, vp, vp, vp, i32, vp, vp, vp]
            for name in EXPORTED[2:]:
                getattr(L, name).restype = C.c_int
            _lib = L
    return _lib


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):           # numpy (host arrays)
        return x.ctypes.data
    raise TypeError(f"cannot pass {type(x)} as a pointer")


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(rc: int, where: str):
    if rc != HS_OK:
        raise HsError(rc, where)


def hs_status_string(status: int) -> str:
    return load().hs_status_string(int(status)).decode()


def hs_version() -> int:
    return load().hs_version()


def ptr_array(tensors, device):
    """Device int64 tensor holding the data pointers of ``tensors`` (a device pointer array)."""
    import torch
    return torch.tensor([_ptr(t) for t in tensors], dtype=torch.int64, device=device)


def hs_align_prefix(N: int, hit_len: int, avail, page_size: int):
    """Strict-prefix alignment; returns (c, n_pages, tail)."""
    av = (C.c_int64 * len(avail))(*[int(a) for a in avail]) if len(avail) else None
    c, npg, tail = C.c_int64(), C.c_int64(), C.c_int64()
    rc = load().hs_align_prefix(int(N), int(hit_len), C.cast(av, C.c_void_p) if av else None,
                                len(avail), int(page_size), C.addressof(c), C.addressof(npg),
                                C.addressof(tail))
    _check(rc, "hs_align_prefix")
    return c.value, npg.value, tail.value


def hs_restore_kv_pages(staging_layers, cache_layers, n_layers: int, block_table, n_pages: int,
                        page_bytes: int, num_blocks: int, d_err=None, stream=None):
    rc = load().hs_restore_kv_pages(_ptr(staging_layers), _ptr(cache_layers), int(n_layers),
                                    _ptr(block_table), int(n_pages), int(page_bytes),
                                    int(num_blocks), _ptr(d_err), _stream(stream))
    _check(rc, "hs_restore_kv_pages")


def hs_restore_request(staging_layers, cache_layers, n_layers: int, block_table, n_pages: int,
                       page_bytes: int, num_blocks: int, src_slots, dst_slots, n_slots: int,
                       floats_each: int, d_err=None, stream=None):
    rc = load().hs_restore_request(_ptr(staging_layers), _ptr(cache_layers), int(n_layers),
                                   _ptr(block_table), int(n_pages), int(page_bytes),
                                   int(num_blocks), _ptr(src_slots), _ptr(dst_slots), int(n_slots),
                                   int(floats_each), _ptr(d_err), _stream(stream))
    _check(rc, "hs_restore_request")


def hs_save_kv_pages(cache_layers, staging_layers, n_layers: int, block_table, n_pages: int,
                     page_bytes: int, num_blocks: int, d_err=None, stream=None):
    rc = load().hs_save_kv_pages(_ptr(cache_layers), _ptr(staging_layers), int(n_layers),
                                 _ptr(block_table), int(n_pages), int(page_bytes),
                                 int(num_blocks), _ptr(d_err), _stream(stream))
    _check(rc, "hs_save_kv_pages")


def hs_restore_kv_page_slices(staging_layers, cache_layers, n_layers: int, block_table,
                              n_pages: int, page_bytes: int, rows: int, col_off: int,
                              col_bytes: int, num_blocks: int, d_err=None, stream=None):
    rc = load().hs_restore_kv_page_slices(_ptr(staging_layers), _ptr(cache_layers), int(n_layers),
                                          _ptr(block_table), int(n_pages), int(page_bytes),
                                          int(rows), int(col_off), int(col_bytes), int(num_blocks),
                                          _ptr(d_err), _stream(stream))
    _check(rc, "hs_restore_kv_page_slices")


def hs_save_kv_page_slices(cache_layers, staging_layers, n_layers: int, block_table, n_pages: int,
                           page_bytes: int, rows: int, col_off: int, col_bytes: int,
                           num_blocks: int, d_err=None, stream=None):
    rc = load().hs_save_kv_page_slices(_ptr(cache_layers), _ptr(staging_layers), int(n_layers),
                                       _ptr(block_table), int(n_pages), int(page_bytes),
                                       int(rows), int(col_off), int(col_bytes), int(num_blocks),
                                       _ptr(d_err), _stream(stream))
    _check(rc, "hs_save_kv_page_slices")


def hs_restore_state(src_slots, dst_slots, n: int, floats_each: int, d_err=None, stream=None):
    rc = load().hs_restore_state(_ptr(src_slots), _ptr(dst_slots), int(n), int(floats_each),
                                 _ptr(d_err), _stream(stream))
    _check(rc, "hs_restore_state")


def hs_checkpoint_states(live_states, ckpt_slots, n: int, floats_each: int, d_err=None,
                         stream=None):
    rc = load().hs_checkpoint_states(_ptr(live_states), _ptr(ckpt_slots), int(n),
                                     int(floats_each), _ptr(d_err), _stream(stream))
    _check(rc, "hs_checkpoint_states")


def make_shape(batch, n_heads, d_k, d_v, max_tokens, kernel=HS_LINATTN_AUTO):
    return hs_linattn_shape(int(batch), int(n_heads), int(d_k), int(d_v), int(max_tokens),
                            int(kernel), 0)


def _prefill_call(name, shape, q, k, v, log_g, o, state, pos0, n_tokens, ckpt_interval,
                  ckpt_slots, d_err, stream):
    B = int(shape.batch)
    p0 = (C.c_int64 * max(B, 1))(*[int(x) for x in pos0])
    nt = (C.c_int32 * max(B, 1))(*[int(x) for x in n_tokens])
    rc = getattr(load(), name)(C.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(log_g), _ptr(o),
                               _ptr(state), C.addressof(p0), C.addressof(nt), int(ckpt_interval),
                               _ptr(ckpt_slots), _ptr(d_err), _stream(stream))
    _check(rc, name)


def hs_linattn_prefill_from_state(shape: hs_linattn_shape, q, k, v, log_g, o, state, pos0,
                                  n_tokens, ckpt_interval: int, ckpt_slots=None, d_err=None,
                                  stream=None):
    """pos0 / n_tokens: host sequences (ints) of length shape.batch."""
    _prefill_call("hs_linattn_prefill_from_state", shape, q, k, v, log_g, o, state, pos0,
                  n_tokens, ckpt_interval, ckpt_slots, d_err, stream)


def hs_test_prefill_stalled(shape: hs_linattn_shape, q, k, v, log_g, o, state, pos0, n_tokens,
                            ckpt_interval: int, ckpt_slots=None, d_err=None, stream=None):
    """Failure-detection hook (include/hs_test.h): the tensor-core prefill with one wait that
    nothing completes; each CTA's bounded wait runs out and it reports HS_DEVERR_TIMEOUT."""
    _prefill_call("hs_test_prefill_stalled", shape, q, k, v, log_g, o, state, pos0, n_tokens,
                  ckpt_interval, ckpt_slots, d_err, stream)


def hs_linattn_scan_workspace_bytes(shape: hs_linattn_shape, pos0, n_tokens) -> int:
    """Bytes of workspace hs_linattn_prefill_scan needs for these arguments."""
    B = int(shape.batch)
    p0 = (C.c_int64 * max(B, 1))(*[int(x) for x in pos0])
    nt = (C.c_int32 * max(B, 1))(*[int(x) for x in n_tokens])
    out = C.c_int64()
    rc = load().hs_linattn_scan_workspace_bytes(C.byref(shape), C.addressof(p0), C.addressof(nt),
                                                C.addressof(out))
    _check(rc, "hs_linattn_scan_workspace_bytes")
    return out.value


def hs_linattn_prefill_scan(shape: hs_linattn_shape, q, k, v, log_g, o, state, pos0, n_tokens,
                            ckpt_interval: int, ckpt_slots, workspace, workspace_bytes: int,
                            d_err=None, stream=None):
    """Segment-parallel prefill (same arguments as hs_linattn_prefill_from_state plus a device
    workspace of hs_linattn_scan_workspace_bytes bytes)."""
    B = int(shape.batch)
    p0 = (C.c_int64 * max(B, 1))(*[int(x) for x in pos0])
    nt = (C.c_int32 * max(B, 1))(*[int(x) for x in n_tokens])
    rc = load().hs_linattn_prefill_scan(C.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(log_g),
                                        _ptr(o), _ptr(state), C.addressof(p0), C.addressof(nt),
                                        int(ckpt_interval), _ptr(ckpt_slots), _ptr(workspace),
                                        int(workspace_bytes), _ptr(d_err), _stream(stream))
    _check(rc, "hs_linattn_prefill_scan")


def hs_linattn_prefill_scan_noalloc(shape: hs_linattn_shape, q, k, v, log_g, o, state, pos0,
                                    n_tokens, ckpt_interval: int, ckpt_slots=None, d_err=None,
                                    stream=None):
    """hs_linattn_prefill_scan with the library's fixed per-device workspace of
    HS_NOALLOC_SCRATCH_BYTES, for callers that cannot allocate device memory at this point (a
    serving engine whose HBM is already handed to its KV-cache pool).  Allocates nothing: the
    host arrays below are ctypes buffers.  Calls that overlap on the GPU share the workspace
    and race; the first call on a device does a one-time set-up and belongs before any stream
    capture."""
    B = int(shape.batch)
    p0 = (C.c_int64 * max(B, 1))(*[int(x) for x in pos0])
    nt = (C.c_int32 * max(B, 1))(*[int(x) for x in n_tokens])
    rc = load().hs_linattn_prefill_scan_noalloc(C.byref(shape), _ptr(q), _ptr(k), _ptr(v),
                                                _ptr(log_g), _ptr(o), _ptr(state),
                                                C.addressof(p0), C.addressof(nt),
                                                int(ckpt_interval), _ptr(ckpt_slots),
                                                _ptr(d_err), _stream(stream))
    _check(rc, "hs_linattn_prefill_scan_noalloc")


def hs_linattn_prefill_packed(shape: hs_linattn_shape, q, k, v, log_g, o, state, pos0, n_tokens,
                              cu_rows, ckpt_interval: int, ckpt_slots=None, d_err=None,
                              stream=None):
    """Packed token layout: token t of problem b is row cu_rows[b] + t.  pos0 / n_tokens /
    cu_rows: host sequences of length batch, batch, batch + 1."""
    B = int(shape.batch)
    p0 = (C.c_int64 * max(B, 1))(*[int(x) for x in pos0])
    nt = (C.c_int32 * max(B, 1))(*[int(x) for x in n_tokens])
    cu = (C.c_int64 * max(B + 1, 1))(*[int(x) for x in cu_rows])
    rc = load().hs_linattn_prefill_packed(C.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(log_g),
                                          _ptr(o), _ptr(state), C.addressof(p0), C.addressof(nt),
                                          C.addressof(cu), int(ckpt_interval), _ptr(ckpt_slots),
                                          _ptr(d_err), _stream(stream))
    _check(rc, "hs_linattn_prefill_packed")


def hs_linattn_num_checkpoints(pos0, n_tokens, ckpt_interval: int) -> int:
    B = len(pos0)
    p0 = (C.c_int64 * max(B, 1))(*[int(x) for x in pos0])
    nt = (C.c_int32 * max(B, 1))(*[int(x) for x in n_tokens])
    tot = C.c_int64()
    rc = load().hs_linattn_num_checkpoints(B, C.addressof(p0), C.addressof(nt), int(ckpt_interval),
                                           C.addressof(tot))
    _check(rc, "hs_linattn_num_checkpoints")
    return tot.value
