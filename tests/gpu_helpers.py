"""Shared helpers for the GPU tests: run the library through the C-ABI on
seeded inputs and compare with the oracle."""
import numpy as np
import torch

import paper_2609_15030_gb300 as hs

TOL = 2e-3       # max-normalised relative error bound for outputs and states


def device():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_15030_gb300 import build
    build.build()
    return torch.device("cuda:0")


def to_dev(x: np.ndarray, dev):
    if x.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev)
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def maxnorm_err(x: np.ndarray, r: np.ndarray, axes) -> float:
    """max over the kept axes of max|x-r| / max|r| over ``axes`` (per-tensor normalised)."""
    num = np.max(np.abs(x - r), axis=axes)
    den = np.max(np.abs(r), axis=axes)
    den = np.where(den == 0, 1.0, den)
    return float(np.max(num / den))


def run_prefill(inp, pos0, n_tokens, S0, C, dev, kernel=hs.HS_LINATTN_AUTO, want_ckpts=True,
                stream=None):
    """Run hs_linattn_prefill_from_state on numpy inputs; returns numpy (o, S, ckpt list)."""
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    B, T, nH, d = inp.q.shape
    state = to_dev(np.zeros((B, nH, d, d), np.float32) if S0 is None
                   else np.asarray(S0, np.float32), dev)
    o = torch.zeros((B, T, nH, d), dtype=torch.float32, device=dev)
    nck = hs.hs_linattn_num_checkpoints(pos0, n_tokens, C) if want_ckpts else 0
    slots = torch.full((max(nck, 1), nH, d, d), float("nan"), device=dev)
    ptrs = hs.ptr_array([slots[i] for i in range(nck)], dev) if nck else None
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    shape = hs.make_shape(B, nH, d, d, T, kernel)
    hs.hs_linattn_prefill_from_state(shape, q, k, v, a, o, state, pos0, n_tokens, C,
                                     ptrs, err, stream=stream)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    cks, i = [], 0
    for b in range(B):
        m = 0 if not want_ckpts or C == 0 or n_tokens[b] == 0 else \
            (pos0[b] + n_tokens[b]) // C - pos0[b] // C
        cks.append(slots[i:i + m].cpu().numpy())
        i += m
    return o.cpu().numpy(), state.cpu().numpy(), cks


def run_scan_prefill(inp, pos0, n_tokens, S0, C, dev, kernel=hs.HS_LINATTN_AUTO):
    """hs_linattn_prefill_scan on numpy inputs; returns numpy (o, S, checkpoint list)."""
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    B, T, nH, d = inp.q.shape
    state = to_dev(np.zeros((B, nH, d, d), np.float32) if S0 is None
                   else np.asarray(S0, np.float32), dev)
    o = torch.full((B, T, nH, d), float("nan"), device=dev)
    nck = hs.hs_linattn_num_checkpoints(pos0, n_tokens, C)
    slots = torch.full((max(nck, 1), nH, d, d), float("nan"), device=dev)
    ptrs = hs.ptr_array([slots[i] for i in range(nck)], dev) if nck else None
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    shape = hs.make_shape(B, nH, d, d, T, kernel)
    nb = hs.hs_linattn_scan_workspace_bytes(shape, pos0, n_tokens)
    ws = torch.full((max(nb // 4, 4),), float("nan"), device=dev)   # stale contents must not matter
    hs.hs_linattn_prefill_scan(shape, q, k, v, a, o, state, pos0, n_tokens, C, ptrs, ws, nb, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    cks, i = [], 0
    for b in range(B):
        m = 0 if C == 0 or n_tokens[b] == 0 else (pos0[b] + n_tokens[b]) // C - pos0[b] // C
        cks.append(slots[i:i + m].cpu().numpy())
        i += m
    return o.cpu().numpy(), state.cpu().numpy(), cks
