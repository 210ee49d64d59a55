"""The segment-parallel prefill (hs_linattn_prefill_scan) on the GPU against the float64 oracle.

Same parity bar as the sequential prefill: outputs, final states and checkpoints within a
max-normalised relative error of 2e-3 per (request, head) tensor; and its own resume from a
checkpoint on the absolute chunk grid reproduces its own full recomputation bit for bit (the
paper's matched checkpoint schedule, Section 4.1 and Table 2).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_15030_gb300 as hs
from hs_inputs import gen_linear, gen_state
from tests.gpu_helpers import TOL, device, maxnorm_err, run_scan_prefill as run_scan, to_dev

pytestmark = pytest.mark.gpu


def _check_oracle(inp, pos0, n_tokens, S0, C, got):
    o, S, cks = got
    ro, rS, rcks = oracle.gla(inp.q, inp.k, inp.v, inp.a, pos0, n_tokens, S0=S0, C_=C)
    for b, n in enumerate(n_tokens):
        if n:
            assert maxnorm_err(o[b, :n], ro[b, :n], axes=(0, 2)) <= TOL, b
            assert np.isnan(o[b, n:]).all()                 # rows past the tail untouched
    assert maxnorm_err(S, rS, axes=(2, 3)) <= TOL
    for b in range(len(n_tokens)):
        assert cks[b].shape == rcks[b].shape
        if cks[b].shape[0]:
            assert maxnorm_err(cks[b], rcks[b], axes=(2, 3)) <= TOL, b


CASES = {
    # the single-layer sweep's resumed tail: one problem of 16 heads, 512 tokens from c = 4096
    "sweep_tail": dict(B=1, nH=16, d=128, T=512, pos0=[4096], n=[512], C=512, gates="uniform",
                       s0=True),
    # a recomputation from the zero state emitting a checkpoint every chunk
    "recompute_c64": dict(B=1, nH=4, d=128, T=1024, pos0=[0], n=[1024], C=64, gates="uniform",
                          s0=False),
    # the tiny stack at head width 64 (strong decay: the segments take the exact path)
    "tiny_d64": dict(B=1, nH=2, d=64, T=256, pos0=[0], n=[256], C=64, gates="sigmoid", s0=False),
    # a batch with resume points off the grid, ragged and short tails and an empty one
    "ragged_batch": dict(B=5, nH=3, d=128, T=200, pos0=[100, 0, 640, 64, 7],
                         n=[37, 200, 5, 129, 0], C=128, gates="uniform", s0=True),
}


@pytest.mark.parametrize("name", list(CASES))
def test_scan_matches_the_oracle(name):
    dev = device()
    c = CASES[name]
    inp = gen_linear(len(name), 0, c["B"], c["T"], c["nH"], c["d"], c["d"], c["gates"])
    S0 = gen_state(len(name), 1, c["B"], c["nH"], c["d"], c["d"]) if c["s0"] else None
    got = run_scan(inp, c["pos0"], c["n"], S0, c["C"], dev)
    _check_oracle(inp, c["pos0"], c["n"], S0, c["C"], got)


@pytest.mark.parametrize("d,N,c,C", [(128, 1024, 512, 512), (128, 700, 256, 128),
                                     (64, 512, 192, 64), (128, 4608, 4096, 512)])
def test_scan_resume_equals_its_recompute_bitwise(d, N, c, C):
    """The scan's full recomputation of [0,N) against its own resume from the checkpoint it
    emitted at c: outputs of [c,N), the final state and the later checkpoints, bit for bit.
    At N = 4608 the recomputation's output pass gives each CTA two segments and the resume's
    one, so this also checks that grouping segments changes no output."""
    dev = device()
    inp = gen_linear(N + d, 0, 1, N, 4, d, d, "uniform")
    o_f, S_f, ck_f = run_scan(inp, [0], [N], None, C, dev)
    m = c // C - 1
    sub = type(inp)(*(x[:, c:N].copy() for x in (inp.q, inp.k, inp.v, inp.a)))
    o_r, S_r, ck_r = run_scan(sub, [c], [N - c], ck_f[0][m][None], C, dev)
    assert np.array_equal(o_r[0].view(np.uint32), o_f[0, c:N].view(np.uint32))
    assert np.array_equal(S_r.view(np.uint32), S_f.view(np.uint32))
    assert np.array_equal(ck_r[0].view(np.uint32), ck_f[0][m + 1:].view(np.uint32))
    _check_oracle(inp, [0], [N], None, C, (o_f, S_f, ck_f))


def test_scan_zero_gates_and_strong_decay():
    """Zero gates (a = -1e4) inside segments and a stretch of strong decay: the segments the
    tensor-core kernel sends to its exact path still chain correctly through the scan."""
    dev = device()
    inp = gen_linear(77, 0, 2, 320, 4, 128, 128, "uniform")
    a = inp.a.copy()
    a[0, 70] = -1e4                      # forgets everything before token 70 of problem 0
    a[1, 130:190] = -1.2                 # strong decay across a chunk boundary
    a[1, 250] = -1e4
    inp = type(inp)(inp.q, inp.k, inp.v, a)
    S0 = gen_state(78, 1, 2, 4, 128, 128)
    got = run_scan(inp, [64, 0], [256, 320], S0, 64, dev)
    _check_oracle(inp, [64, 0], [256, 320], S0, 64, got)


def test_scan_more_segments_than_one_launch_holds():
    """512 segments (two problems of 16,384 tokens): each tensor-core pass takes two launches."""
    dev = device()
    inp = gen_linear(91, 0, 2, 16384, 2, 64, 64, "uniform")
    got = run_scan(inp, [0, 0], [16384, 16384], None, 4096, dev)
    _check_oracle(inp, [0, 0], [16384, 16384], None, 4096, got)


def test_scan_and_sequential_prefill_agree():
    """Within the parity bar of each other on the sweep's shape (they are not bit-identical:
    the state enters each segment through the scan's fma instead of the tensor cores)."""
    dev = device()
    inp = gen_linear(5, 0, 1, 512, 16, 128, 128, "uniform")
    S0 = gen_state(6, 1, 1, 16, 128, 128)
    from tests.gpu_helpers import run_prefill
    o1, S1, _ = run_prefill(inp, [1024], [512], S0, 512, dev)
    o2, S2, _ = run_scan(inp, [1024], [512], S0, 512, dev)
    assert maxnorm_err(o2[0], o1[0], axes=(0, 2)) <= TOL
    assert maxnorm_err(S2, S1, axes=(2, 3)) <= TOL


def test_scan_checkpoint_slot_errors_are_reported():
    """A NULL or misaligned checkpoint slot read from the device pointer array: the scan
    reports it in d_err (first error wins) and skips that slot's write."""
    dev = device()
    N, nH, d = 128, 2, 128
    inp = gen_linear(8, 0, 1, N, nH, d, d)
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    state = torch.zeros((1, nH, d, d), device=dev)
    o = torch.zeros((1, N, nH, d), device=dev)
    slot = torch.zeros(nH * d * d + 4, device=dev)
    shape = hs.make_shape(1, nH, d, d, N)
    nb = hs.hs_linattn_scan_workspace_bytes(shape, [0], [N])
    ws = torch.empty(nb // 4, device=dev)
    for ptrs, code in (([slot.data_ptr() + 4, slot.data_ptr()], hs.HS_DEVERR_MISALIGNED),
                       ([0, slot.data_ptr()], hs.HS_DEVERR_NULL)):
        err = torch.zeros(1, dtype=torch.int32, device=dev)
        state.zero_()
        hs.hs_linattn_prefill_scan(shape, q, k, v, a, o, state, [0], [N], 64,
                                   hs.ptr_array(ptrs, dev), ws, nb, err)
        torch.cuda.synchronize()
        assert err.item() == code


def test_scan_graph_replay_equals_eager_call():
    """The three launches of one call captured in a CUDA graph and replayed twice give the
    bytes of the eager call (the workspace's stale contents do not matter either)."""
    dev = device()
    B, nH, d, T, C = 2, 8, 128, 448, 128
    inp = gen_linear(12, 0, B, T, nH, d, d, "uniform")
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    S0 = torch.from_numpy(gen_state(12, 1, B, nH, d, d)).to(dev)
    pos0, n = [256, 37], [448, 300]
    shape = hs.make_shape(B, nH, d, d, T)
    nck = hs.hs_linattn_num_checkpoints(pos0, n, C)
    state = torch.empty_like(S0)
    o = torch.empty((B, T, nH, d), device=dev)
    slots = torch.empty((nck, nH, d, d), device=dev)
    ptrs = hs.ptr_array([slots[i] for i in range(nck)], dev)
    nb = hs.hs_linattn_scan_workspace_bytes(shape, pos0, n)
    ws = torch.empty(nb // 4, device=dev)
    s = torch.cuda.Stream(dev)

    def reset():
        state.copy_(S0)
        o.fill_(float("nan"))
        slots.fill_(float("nan"))
        ws.fill_(float("nan"))
        torch.cuda.synchronize()

    def bits():
        return [t.view(torch.int32).cpu().numpy() for t in (o, state, slots)]

    reset()
    hs.hs_linattn_prefill_scan(shape, q, k, v, a, o, state, pos0, n, C, ptrs, ws, nb, None,
                               s.cuda_stream)
    torch.cuda.synchronize()
    ref = bits()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s, capture_error_mode="relaxed"):
        hs.hs_linattn_prefill_scan(shape, q, k, v, a, o, state, pos0, n, C, ptrs, ws, nb, None,
                                   torch.cuda.current_stream(dev).cuda_stream)
    for _ in range(2):
        reset()
        g.replay()
        torch.cuda.synchronize()
        for x, y in zip(bits(), ref):
            assert np.array_equal(x, y)


def test_scan_exact_segments_inside_spans():
    """Segments that take the exact path (strong decay, a zero gate) in the middle of the
    output pass's multi-segment spans: the oracle bar, and the resume from a checkpoint
    (two segments per CTA) equal to the recomputation (three per CTA) bit for bit."""
    dev = device()
    B, nH, d, N, C, c = 2, 4, 128, 2560, 512, 1024
    inp = gen_linear(41, 0, B, N, nH, d, d, "uniform")
    a = inp.a.copy()
    a[0, 600:700] = -1.2          # strong decay over two chunks (exact path)
    a[0, 1500] = -1e4             # a zero gate after the resume point
    a[1, 1100:1180] = -1.2
    inp = type(inp)(inp.q, inp.k, inp.v, a)
    o_f, S_f, ck_f = run_scan(inp, [0, 0], [N, N], None, C, dev)
    _check_oracle(inp, [0, 0], [N, N], None, C, (o_f, S_f, ck_f))
    m = c // C - 1
    sub = type(inp)(*(x[:, c:N].copy() for x in (inp.q, inp.k, inp.v, inp.a)))
    S_c = np.stack([ck_f[b][m] for b in range(B)])
    o_r, S_r, ck_r = run_scan(sub, [c, c], [N - c, N - c], S_c, C, dev)
    assert np.array_equal(o_r.view(np.uint32), o_f[:, c:N].view(np.uint32))
    assert np.array_equal(S_r.view(np.uint32), S_f.view(np.uint32))
    for b in range(B):
        assert np.array_equal(ck_r[b].view(np.uint32), ck_f[b][m + 1:].view(np.uint32))
