"""Python side of the float64 CPU oracle.

TEST INFRASTRUCTURE ONLY: imported by tests/, by ``__graft_entry__.smoke()``
and by the CPU-baseline leg of ``bench.py``; never by the library.  It shares
no code with the CUDA path; the only module both sides use is ``hs_inputs``
(seeded random inputs).

``hs_oracle.c`` holds the arithmetic (plain definitions, see its header);
this file compiles it with gcc, loads it with ctypes and loops it over
requests and heads.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hs_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
# a prebuilt oracle library to load instead (tests/test_oracle_mutants.py runs the pins
# against deliberately broken copies of hs_oracle.c this way)
_LIB_OVERRIDE = os.environ.get("HS_ORACLE_LIB")
_lock = threading.Lock()
_lib = None


def compile_to(src: str, out: str) -> None:
    """gcc -O2 of one oracle source into a shared library (no fast-math)."""
    subprocess.run(["gcc", "-O2", "-fPIC", "-shared", "-std=c11", "-fno-fast-math",
                    "-o", out, src, "-lm"], check=True)


def build(force: bool = False) -> str:
    """Compile hs_oracle.c into liboracle.so (plain gcc, -O2, no fast-math)."""
    if _LIB_OVERRIDE:
        return _LIB_OVERRIDE
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".{os.getpid()}.tmp"
        compile_to(_SRC, tmp)
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            i64p = C.POINTER(C.c_int64)
            L.oracle_align_prefix.argtypes = [C.c_int64, C.c_int64, i64p, C.c_int32, C.c_int32,
                                              i64p, i64p, i64p]
            L.oracle_align_prefix.restype = C.c_int
            L.oracle_align_prerepair.argtypes = [C.c_int64, C.c_int64, i64p, i64p]
            L.oracle_align_prerepair.restype = None
            L.oracle_scatter_pages.argtypes = [C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p,
                                               C.c_int32, C.c_int64]
            L.oracle_scatter_pages.restype = None
            L.oracle_gather_pages.argtypes = [C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p,
                                              C.c_int32, C.c_int64]
            L.oracle_gather_pages.restype = None
            L.oracle_slices.argtypes = [C.c_int32, C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p,
                                        C.c_int32, C.c_int64, C.c_int32, C.c_int64, C.c_int64]
            L.oracle_slices.restype = None
            L.oracle_copy_slots.argtypes = [C.c_void_p, C.c_void_p, C.c_int32, C.c_int64]
            L.oracle_copy_slots.restype = None
            L.oracle_restore_bytes.argtypes = [C.c_int64] * 7
            L.oracle_restore_bytes.restype = C.c_int64
            L.oracle_gla_head.argtypes = [C.c_int64, C.c_int32, C.c_int32,
                                          C.c_void_p, C.c_void_p, C.c_int64,
                                          C.c_void_p, C.c_int64,
                                          C.c_void_p, C.c_int64,
                                          C.c_void_p, C.c_void_p, C.c_int64,
                                          C.c_int64, C.c_int64, C.c_void_p]
            L.oracle_gla_head.restype = C.c_int64
            _lib = L
    return _lib


# ---------------------------------------------------------------------------
# alignment
# ---------------------------------------------------------------------------

def align_prefix(N: int, hit_len: int, avail, page_size: int):
    """Strict-prefix alignment (Section 2.2, Section 3.2). Returns (c, n_pages, tail)."""
    av = np.ascontiguousarray(np.asarray(list(avail), dtype=np.int64))
    c, npg, tail = C.c_int64(), C.c_int64(), C.c_int64()
    rc = lib().oracle_align_prefix(int(N), int(hit_len),
                                   av.ctypes.data_as(C.POINTER(C.c_int64)), len(av),
                                   int(page_size), C.byref(c), C.byref(npg), C.byref(tail))
    if rc != 0:
        raise ValueError("invalid alignment arguments")
    return c.value, npg.value, tail.value


def align_prerepair(N: int, C_: int):
    """Pre-repair (faulty) behaviour of Section 3.2. Returns (B, p)."""
    B, p = C.c_int64(), C.c_int64()
    lib().oracle_align_prerepair(int(N), int(C_), C.byref(B), C.byref(p))
    return B.value, p.value


def restore_bytes(n_full, n_pages, page_bytes, n_lin, n_heads, d_k, d_v) -> int:
    return lib().oracle_restore_bytes(int(n_full), int(n_pages), int(page_bytes), int(n_lin),
                                      int(n_heads), int(d_k), int(d_v))


# ---------------------------------------------------------------------------
# copies
# ---------------------------------------------------------------------------

def _ptr_array(arrs):
    return (C.c_void_p * len(arrs))(*[a.ctypes.data for a in arrs])


def scatter_pages(staging_layers, cache_layers, block_table, n_pages: int, page_bytes: int):
    """In place on cache_layers (list of uint8 arrays)."""
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    lib().oracle_scatter_pages(_ptr_array(staging_layers), _ptr_array(cache_layers),
                               len(cache_layers), bt.ctypes.data, int(n_pages), int(page_bytes))


def gather_pages(cache_layers, staging_layers, block_table, n_pages: int, page_bytes: int):
    """In place on staging_layers (list of uint8 arrays): the save of Section 3.1."""
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    lib().oracle_gather_pages(_ptr_array(cache_layers), _ptr_array(staging_layers),
                              len(staging_layers), bt.ctypes.data, int(n_pages), int(page_bytes))


def scatter_slices(staging_layers, cache_layers, block_table, n_pages: int, page_bytes: int,
                   rows: int, col_off: int, col_bytes: int):
    """One rank's slice of every page row, staging -> cache, in place on cache_layers."""
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    lib().oracle_slices(0, _ptr_array(staging_layers), _ptr_array(cache_layers), len(cache_layers),
                        bt.ctypes.data, int(n_pages), int(page_bytes), int(rows), int(col_off),
                        int(col_bytes))


def gather_slices(cache_layers, staging_layers, block_table, n_pages: int, page_bytes: int,
                  rows: int, col_off: int, col_bytes: int):
    """One rank's slice of every page row, cache -> staging, in place on staging_layers."""
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    lib().oracle_slices(1, _ptr_array(staging_layers), _ptr_array(cache_layers),
                        len(staging_layers), bt.ctypes.data, int(n_pages), int(page_bytes),
                        int(rows), int(col_off), int(col_bytes))


def copy_slots(src, dst, floats_each: int):
    lib().oracle_copy_slots(_ptr_array(src), _ptr_array(dst), len(src), int(floats_each))


# ---------------------------------------------------------------------------
# gated linear attention, token by token
# ---------------------------------------------------------------------------

def n_checkpoints(pos0: int, n: int, C_: int) -> int:
    if C_ <= 0 or n <= 0:
        return 0
    return (pos0 + n) // C_ - pos0 // C_


def gla(q, k, v, a, pos0, n_tokens, S0=None, C_: int = 0, heads=None, threads: int = 1):
    """Run the token-by-token oracle over a batch.

    q, k: uint16 [B, T, nH, d_k]; v: uint16 [B, T, nH, d_v]; a: float32
    [B, T, nH, d_k]; pos0, n_tokens: per request.  S0: float32/float64
    [B, nH, d_k, d_v] or None (zero state).  heads: optional subset of head
    indices (others are left at zero in the outputs).
    Returns (o [B, T, nH, d_v] float64, S [B, nH, d_k, d_v] float64,
    ckpts: list over requests of float64 [n_ck, nH, d_k, d_v]).
    """
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    a = np.ascontiguousarray(a, dtype=np.float32)
    B, T, nH, dk = q.shape
    dv = v.shape[-1]
    heads = list(range(nH)) if heads is None else list(heads)
    S = np.zeros((B, nH, dk, dv), np.float64) if S0 is None else np.array(S0, dtype=np.float64)
    S = np.ascontiguousarray(S)
    o = np.zeros((B, T, nH, dv), np.float64)
    cks = [np.zeros((n_checkpoints(int(pos0[b]), int(n_tokens[b]), C_), nH, dk, dv), np.float64)
           for b in range(B)]
    L = lib()
    jobs = []
    for b in range(B):
        n = int(n_tokens[b])
        assert 0 <= n <= T
        for h in heads:
            jobs.append((b, h, n))

    def run(job):
        b, h, n = job
        nck = cks[b].shape[0]
        if n == 0:
            return
        tmp = np.zeros((nck, dk, dv), np.float64) if nck else None
        Sh = np.ascontiguousarray(S[b, h])
        got = L.oracle_gla_head(n, dk, dv,
                                q[b, 0, h].ctypes.data, k[b, 0, h].ctypes.data, nH * dk,
                                v[b, 0, h].ctypes.data, nH * dv,
                                a[b, 0, h].ctypes.data, nH * dk,
                                Sh.ctypes.data, o[b, 0, h].ctypes.data, nH * dv,
                                int(pos0[b]), int(C_),
                                tmp.ctypes.data if tmp is not None else None)
        assert got == nck
        S[b, h] = Sh
        if nck:
            cks[b][:, h] = tmp

    if threads <= 1:
        for j in jobs:
            run(j)
    else:
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(run, jobs))
    return o, S, cks
