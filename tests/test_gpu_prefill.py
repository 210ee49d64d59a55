"""Gated linear-attention prefill on the GPU against the float64 oracle.

Parity bar: outputs, final states and checkpoints within a max-normalised
relative error of 2e-3 per (request, head) tensor; resuming from a
checkpoint on the absolute chunk grid must reproduce the GPU's own full
recomputation bit for bit (the paper's matched checkpoint schedule, Section
4.1 and Table 2), for outputs, final states and emitted checkpoints.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_15030_gb300 as hs
from hs_inputs import (LONG24, LONG_LENGTHS, SWEEP, SWEEP_LENGTHS, TINY, bf16_bits_to_f32,
                       f32_to_bf16_bits, gen_linear, gen_state)
from tests.gpu_helpers import TOL, device, maxnorm_err, run_prefill, to_dev

pytestmark = pytest.mark.gpu
KERNELS = [pytest.param(hs.HS_LINATTN_RECURRENT, id="recurrent"),
           pytest.param(hs.HS_LINATTN_CHUNKED_TC, id="tc")]


def _needs(kernel, d):
    """Every kernel implements both head widths (d = 64 and 128)."""
    assert d in (64, 128)


def _check(o, S, cks, ro, rS, rcks, pos0, n_tokens, what=""):
    for b, n in enumerate(n_tokens):
        if n:
            e = maxnorm_err(o[b, :n], ro[b, :n], axes=(0, 2))
            assert e <= TOL, f"{what} outputs b={b}: {e:.3g}"
    e = maxnorm_err(S, rS, axes=(2, 3))
    assert e <= TOL, f"{what} state: {e:.3g}"
    for b in range(len(n_tokens)):
        assert cks[b].shape == rcks[b].shape
        if cks[b].shape[0]:
            e = maxnorm_err(cks[b], rcks[b], axes=(2, 3))
            assert e <= TOL, f"{what} checkpoints b={b}: {e:.3g}"


def _resume_equals_recompute(inp, N, c, C, dev, kernel):
    """GPU full recomputation of [0,N) vs GPU resume from its own checkpoint at c."""
    o_f, S_f, ck_f = run_prefill(inp, [0], [N], None, C, dev, kernel)
    m = c // C - 1
    S_c = ck_f[0][m][None] if c > 0 else None
    sub = type(inp)(*(x[:, c:N].copy() for x in (inp.q, inp.k, inp.v, inp.a)))
    o_r, S_r, ck_r = run_prefill(sub, [c], [N - c], S_c, C, dev, kernel)
    assert np.array_equal(o_r[0].view(np.uint32), o_f[0, c:N].view(np.uint32))
    assert np.array_equal(S_r.view(np.uint32), S_f.view(np.uint32))
    assert np.array_equal(ck_r[0].view(np.uint32), ck_f[0][m + 1:].view(np.uint32))
    return o_f, S_f, ck_f


@pytest.mark.parametrize("kernel", KERNELS)
def test_tiny_hybrid_config(kernel):
    """Tiny stack: N=256, C=64, complete hit -> c=192; 64-token tail vs full recompute of 256."""
    _needs(kernel, TINY.d)
    dev = device()
    N, C = 256, TINY.ckpt
    c, _, tail = hs.hs_align_prefix(N, N, list(range(C, N + 1, C)), TINY.page)
    assert (c, tail) == (192, 64)
    inp = gen_linear(0, 0, 1, N, TINY.n_heads, TINY.d, TINY.d, gates=TINY.gates)
    o_f, S_f, ck_f = _resume_equals_recompute(inp, N, c, C, dev, kernel)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], C_=C)
    _check(o_f, S_f, ck_f, ro, rS, rck, [0], [N], "tiny")


def test_head_width_64_fast_path_resumes_bitwise():
    """d = 64 on the tensor cores (M = 128 products with half the TMEM lanes unused): gates
    U(-0.1, 0) keep every segment on the fp16 path; resuming from the checkpoint at 512
    reproduces the recomputation bit for bit and both follow the oracle."""
    dev = device()
    N, C, nH, d = 1000, 128, 8, 64
    inp = gen_linear(17, 0, 1, N, nH, d, d)
    o_f, S_f, ck_f = _resume_equals_recompute(inp, N, 512, C, dev, hs.HS_LINATTN_CHUNKED_TC)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], C_=C, threads=16)
    _check(o_f, S_f, ck_f, ro, rS, rck, [0], [N], "d64 fast")


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("L", SWEEP_LENGTHS)
def test_sweep_config_complete_and_partial_hit(kernel, L):
    """Single-layer sweep: 16 heads, d=128, C=512; complete hit and hit = L-37."""
    dev = device()
    C = SWEEP.ckpt
    inp = gen_linear(1, 0, 1, L, SWEEP.n_heads, SWEEP.d, SWEEP.d, gates=SWEEP.gates)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [L], C_=C, threads=16)
    for hit in (L, L - 37):
        c, _, tail = hs.hs_align_prefix(L, hit, list(range(C, L + 1, C)), SWEEP.page)
        assert tail >= 1 and c % C == 0
        o_f, S_f, ck_f = _resume_equals_recompute(inp, L, c, C, dev, kernel)
        _check(o_f, S_f, ck_f, ro, rS, rck, [0], [L], f"L={L} hit={hit}")


@pytest.mark.parametrize("kernel", KERNELS)
def test_ragged_prompt_lengths(kernel):
    """Complete hits at N = L-37 leave a ragged last chunk; several tail lengths."""
    dev = device()
    C = 128
    for N in (1, 3, 63, 65, 130, 475):
        inp = gen_linear(2, N, 1, N, 4, 128, 128)
        c, _, _ = hs.hs_align_prefix(N, N, list(range(C, N + 1, C)), 16)
        o_f, S_f, ck_f = _resume_equals_recompute(inp, N, c, C, dev, kernel)
        ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], C_=C)
        _check(o_f, S_f, ck_f, ro, rS, rck, [0], [N], f"N={N}")


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("d", [64, 128])
def test_batch_mixed_positions_from_nonzero_state(kernel, d):
    _needs(kernel, d)
    dev = device()
    B, T, nH = 5, 200, 3
    pos0 = [0, 64, 128 + 5, 1000, 7]
    n_tok = [200, 0, 77, 129, 1]
    inp = gen_linear(3, 0, B, T, nH, d, d)
    S0 = gen_state(3, 0, B, nH, d, d)
    o, S, cks = run_prefill(inp, pos0, n_tok, S0, 64, dev, kernel)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, pos0, n_tok, S0=S0, C_=64)
    _check(o, S, cks, ro, rS, rck, pos0, n_tok, "batch")
    np.testing.assert_array_equal(S[1], S0[1])          # empty tail leaves the state untouched


@pytest.mark.parametrize("kernel", KERNELS)
def test_mixed_gate_strengths_take_both_paths(kernel):
    """Chunks whose per-dimension decay is too strong for the factorised fp16
    operands (the tensor-core kernel's exact path) interleaved with ordinary
    chunks; both must match the oracle and keep resume == recompute bitwise."""
    dev = device()
    N, C, nH, d = 448, 64, 4, 128
    inp = gen_linear(12, 0, 1, N, nH, d, d)
    inp.a[:, 70:75, :, :7] = -30.0          # strong decay on a few key dims in chunk 1
    inp.a[:, 200, 1] = -1e4                 # a zero gate for head 1 in chunk 3
    inp.a[:, 300:364, 2] = -1.2             # steady strong decay over a whole chunk
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], C_=C)
    for c in (64, 192, 320):
        o_f, S_f, ck_f = _resume_equals_recompute(inp, N, c, C, dev, kernel)
    _check(o_f, S_f, ck_f, ro, rS, rck, [0], [N], "mixed gates")


def _scaled(bits, f):
    return f32_to_bf16_bits(bf16_bits_to_f32(bits) * np.float32(f))


@pytest.mark.parametrize("case", ["big_v", "big_qk", "positive_gates", "big_state"])
def test_fp16_range_guards_take_the_exact_path(case):
    """Inputs outside the fast path's fp16 range (values, the bound on the intra-chunk
    scores, growing gates, a large restored state) in some chunks: those chunks take
    the exact path, the others stay fast; all match the oracle, resume == recompute."""
    dev = device()
    N, C, nH, d = 448, 64, 4, 128
    inp = gen_linear(15, 0, 1, N, nH, d, d)
    S0 = gen_state(15, 0, 1, nH, d, d)
    if case == "big_v":
        inp.v[:, 130:150] = _scaled(inp.v[:, 130:150], 2.0 ** 17)
    elif case == "big_qk":
        inp.q[:, 200:260] = _scaled(inp.q[:, 200:260], 64.0)
        inp.k[:, 200:260] = _scaled(inp.k[:, 200:260], 64.0)
    elif case == "positive_gates":
        inp.a[:, 64:128] = 0.02
    else:
        S0 = (S0 * 2.0 ** 16).astype(np.float32)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], S0=S0, C_=C)
    o, S, cks = run_prefill(inp, [0], [N], S0, C, dev, hs.HS_LINATTN_CHUNKED_TC)
    _check(o, S, cks, ro, rS, rck, [0], [N], case)
    # resume from the GPU's own checkpoints reproduces the full run bit for bit
    for c in (64, 192):
        m = c // C - 1
        sub = type(inp)(*(x[:, c:N].copy() for x in (inp.q, inp.k, inp.v, inp.a)))
        o_r, S_r, ck_r = run_prefill(sub, [c], [N - c], cks[0][m][None], C, dev,
                                     hs.HS_LINATTN_CHUNKED_TC)
        assert np.array_equal(o_r[0].view(np.uint32), o[0, c:N].view(np.uint32))
        assert np.array_equal(S_r.view(np.uint32), S.view(np.uint32))
        assert np.array_equal(ck_r[0].view(np.uint32), cks[0][m + 1:].view(np.uint32))


@pytest.mark.parametrize("kernel", [pytest.param(hs.HS_LINATTN_CHUNKED_TC, id="tc"),
                                    pytest.param(hs.HS_LINATTN_AUTO, id="auto")])
def test_state_bound_band_resumes_bitwise(kernel):
    """A decision inside a fast run only has a bound on the state it starts from (the state
    before the previous segment plus that segment's largest update).  Here the bound exceeds
    the fp16 limit 2^15 while the state itself, halved by chunk 0's gates, stays far below it:
    a full run from S0 must decide chunk 1 on the measured state, as a run resumed from the
    checkpoint at 64 does, so the two agree bit for bit (and stay within 2e-3 of the oracle)."""
    dev = device()
    N, C, nH, d = 192, 64, 2, 128
    inp = gen_linear(41, 0, 1, N, nH, d, d)
    inp.a[0, :64] = np.float32(np.log(0.5) / 64)           # chunk 0 decays the state by 1/2
    for x in (inp.k, inp.v):                                  # a large update in chunk 0
        x[0, :64] = f32_to_bf16_bits(bf16_bits_to_f32(x[0, :64]) * np.float32(24.0))
    S0 = gen_state(41, 0, 1, nH, d, d)
    S0 = (S0 * np.float32(31000.0 / np.abs(S0).max())).astype(np.float32)
    kb = np.abs(bf16_bits_to_f32(inp.k[0, :64])).max()
    vb = np.abs(bf16_bits_to_f32(inp.v[0, :64])).max()
    assert np.abs(S0).max() + 64 * kb * vb > 2.0 ** 15       # the bound fails ...
    o_f, S_f, ck_f = run_prefill(inp, [0], [N], S0, C, dev, kernel)
    assert np.abs(ck_f[0][0]).max() < 2.0 ** 14               # ... the state does not
    sub = type(inp)(*(x[:, 64:N].copy() for x in (inp.q, inp.k, inp.v, inp.a)))
    o_r, S_r, ck_r = run_prefill(sub, [64], [N - 64], ck_f[0][0][None], C, dev, kernel)
    assert np.array_equal(o_r[0].view(np.uint32), o_f[0, 64:N].view(np.uint32))
    assert np.array_equal(S_r.view(np.uint32), S_f.view(np.uint32))
    assert np.array_equal(ck_r[0].view(np.uint32), ck_f[0][1:].view(np.uint32))
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], S0=S0, C_=C)
    _check(o_f, S_f, ck_f, ro, rS, rck, [0], [N], "state-bound band")


@pytest.mark.parametrize("kernel", [pytest.param(hs.HS_LINATTN_CHUNKED_TC, id="tc"),
                                    pytest.param(hs.HS_LINATTN_AUTO, id="auto")])
@pytest.mark.parametrize("seed", [3, 7, 9])
def test_dominant_token_whose_own_score_cancels(kernel, seed):
    """One token's q . k cancels to about 1 % of sum_d |q_d k_d| while its v, scaled by 2^17,
    makes its output the head's largest by far: its error is the error of its own score
    A_ii = q_i . k_i, which the fast path sums in float32 from the bf16 inputs (fp16 operands
    would round each term to 11 bits and leave errors of up to 6.5e-3 here)."""
    dev = device()
    inp = gen_linear(seed, 0, 1, 64, 1, 128, 128)
    q = bf16_bits_to_f32(inp.q[0, 63, 0]).astype(np.float64)
    k = bf16_bits_to_f32(inp.k[0, 63, 0]).astype(np.float64)
    k = k - (q @ k - 0.005) / (q @ q) * q
    inp.k[0, 63, 0] = f32_to_bf16_bits(k.astype(np.float32))
    inp.v[0, 63, 0] = f32_to_bf16_bits(bf16_bits_to_f32(inp.v[0, 63, 0]) * np.float32(2.0 ** 17))
    o, S, cks = run_prefill(inp, [0], [64], None, 64, dev, kernel)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [64], C_=64)
    assert np.abs(ro[0, 63]).max() > 30 * np.abs(ro[0, :63]).max()
    _check(o, S, cks, ro, rS, rck, [0], [64], "cancelling score")


@pytest.mark.parametrize("pattern", ["first", "middle_pair", "last", "all"])
def test_exact_segments_at_run_boundaries(pattern):
    """Segments sent to the exact path (growing gates) where a run of fast segments
    would start, two in a row between two runs, at the last long segment before a
    trailing short one, and everywhere; the call starts off the grid with a leading
    short segment.  All match the oracle, and resuming on the grid from the call's own
    checkpoint reproduces it bit for bit."""
    dev = device()
    pos0, N, C, nH, d = 60, 329, 64, 4, 128      # segments: 4 | 5 x 64 | 5 tokens
    inp = gen_linear(21, 0, 1, N, nH, d, d)
    S0 = gen_state(21, 0, 1, nH, d, d)
    for k in {"first": [0], "middle_pair": [2, 3], "last": [4], "all": range(5)}[pattern]:
        inp.a[:, 4 + 64 * k:4 + 64 * (k + 1)] = 0.02
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [pos0], [N], S0=S0, C_=C)
    o, S, cks = run_prefill(inp, [pos0], [N], S0, C, dev, hs.HS_LINATTN_CHUNKED_TC)
    _check(o, S, cks, ro, rS, rck, [pos0], [N], pattern)
    c = 192
    t, m = c - pos0, c // C - pos0 // C - 1
    sub = type(inp)(*(x[:, t:N].copy() for x in (inp.q, inp.k, inp.v, inp.a)))
    o_r, S_r, ck_r = run_prefill(sub, [c], [N - t], cks[0][m][None], C, dev,
                                 hs.HS_LINATTN_CHUNKED_TC)
    assert np.array_equal(o_r[0, :N - t].view(np.uint32), o[0, t:N].view(np.uint32))
    assert np.array_equal(S_r.view(np.uint32), S.view(np.uint32))
    assert np.array_equal(ck_r[0].view(np.uint32), cks[0][m + 1:].view(np.uint32))


@pytest.mark.parametrize("where", ["short_call", "full_segment"])
def test_zero_gate_inside_an_exact_segment(where):
    """A zero gate (a = -1e4) followed, in the same segment, by growing gates (the exact
    path): the decay factors of the tokens after the zero gate are differences of
    cumulative log-gates, which must stay accurate (the state is reset by the zero gate
    and then grows).  Outputs and final state against the oracle."""
    dev = device()
    nH, d, C = 2, 128, 512
    if where == "short_call":
        pos0, n = 221, 18                  # one 18-token segment inside a chunk
        z, g0, g1 = 7, 2, 18
    else:
        pos0, n = 192, 64                  # one whole chunk
        z, g0, g1 = 10, 11, 64
    inp = gen_linear(60250, 0, 1, n, nH, d, d)
    inp.a[0, g0:g1] = 0.02
    inp.a[0, z] = -1e4
    S0 = gen_state(60250, 0, 1, nH, d, d) * 100.0
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [pos0], [n], S0=S0, C_=C)
    for kernel in (hs.HS_LINATTN_CHUNKED_TC, hs.HS_LINATTN_AUTO):
        o, S, cks = run_prefill(inp, [pos0], [n], S0, C, dev, kernel)
        _check(o, S, cks, ro, rS, rck, [pos0], [n], f"{where} kernel {kernel}")


@pytest.mark.parametrize("n_strong", [6, 9, 12])
def test_strong_decay_early_in_each_chunk(n_strong):
    """The first n_strong tokens of every chunk carry a log-gate of -1.2, so each chunk's
    total log2-decay is about -(10.4, 15.6, 20.8) - 4: around the fast path's limit of -10
    (beyond it Q~ = q 2^Lam of the chunk's last tokens would sit in fp16's subnormal range)
    and, for the larger two, past the fp16 range of K~.  Three chunks from a resumed
    position with a checkpoint in the middle, both kernels against the oracle."""
    dev = device()
    nH, d, C = 2, 128, 128
    pos0, n = 128, 192
    inp = gen_linear(60300 + n_strong, 0, 1, n, nH, d, d)
    for c0 in range(0, n, 64):
        inp.a[0, c0:c0 + n_strong] = -1.2
    S0 = gen_state(60300 + n_strong, 0, 1, nH, d, d)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [pos0], [n], S0=S0, C_=C)
    for kernel in (hs.HS_LINATTN_CHUNKED_TC, hs.HS_LINATTN_AUTO):
        o, S, cks = run_prefill(inp, [pos0], [n], S0, C, dev, kernel)
        _check(o, S, cks, ro, rS, rck, [pos0], [n], f"n_strong {n_strong} kernel {kernel}")


@pytest.mark.parametrize("kernel", [hs.HS_LINATTN_AUTO, hs.HS_LINATTN_CHUNKED_TC,
                                    hs.HS_LINATTN_RECURRENT, hs.HS_LINATTN_SINGLE_TOKEN])
def test_largest_batch(kernel):
    """HS_MAX_BATCH problems in one call (the largest launch parameter block): one head
    each, random resume points and tails (one token each for the single-token kernel),
    checkpoints every 64, from random states; every problem against the oracle."""
    dev = device()
    rng = np.random.default_rng(384)
    B, nH, d, C = hs.HS_MAX_BATCH, 1, 128, 64
    pos0 = [int(x) for x in rng.integers(0, 300, B)]
    if kernel == hs.HS_LINATTN_SINGLE_TOKEN:
        n_tok = [int(x) for x in rng.integers(0, 2, B)]
    else:
        n_tok = [int(x) for x in rng.integers(0, 100, B)]
    T = max(max(n_tok), 1)
    inp = gen_linear(384, 0, B, T, nH, d, d)
    S0 = gen_state(384, 0, B, nH, d, d)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, pos0, n_tok, S0=S0, C_=C, threads=16)
    o, S, cks = run_prefill(inp, pos0, n_tok, S0, C, dev, kernel)
    _check(o, S, cks, ro, rS, rck, pos0, n_tok, f"batch {B} kernel {kernel}")


@pytest.mark.parametrize("case", range(16))
def test_random_configurations(case):
    """Seeded random calls: batch 1-3, 1-3 heads, resume points anywhere in [0, 320), tails
    of 0-399 tokens, checkpoint interval 0/64/128/192, from a random state, with growing
    gates (the exact path) on up to two random token ranges; the tensor-core kernel and
    AUTO against the oracle.  Odd cases use the head width 64."""
    dev = device()
    rng = np.random.default_rng(1000 + case)
    B, nH, d = int(rng.integers(1, 4)), int(rng.integers(1, 4)), (128 if case % 2 == 0 else 64)
    C = int(rng.choice([0, 64, 128, 192]))
    pos0 = [int(x) for x in rng.integers(0, 320, B)]
    n_tok = [int(x) for x in rng.integers(0, 400, B)]
    T = max(max(n_tok), 1)
    inp = gen_linear(2000 + case, 0, B, T, nH, d, d)
    for _ in range(int(rng.integers(0, 3))):
        b, t0 = int(rng.integers(B)), int(rng.integers(T))
        inp.a[b, t0:t0 + int(rng.integers(1, 80))] = 0.02
    S0 = gen_state(2000 + case, 0, B, nH, d, d)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, pos0, n_tok, S0=S0, C_=C, threads=8)
    for kernel in (hs.HS_LINATTN_CHUNKED_TC, hs.HS_LINATTN_AUTO):
        o, S, cks = run_prefill(inp, pos0, n_tok, S0, C, dev, kernel)
        _check(o, S, cks, ro, rS, rck, pos0, n_tok, f"case {case} kernel {kernel}")


@pytest.mark.parametrize("kernel", KERNELS)
def test_decode_steps_continue_the_prefill(kernel):
    """Hybrid workload shape: tail prefill then single-token decode steps off the grid."""
    dev = device()
    N, c, steps, nH, d = 512, 256, 16, 16, 128
    inp = gen_linear(4, 0, 1, N + steps, nH, d, d)
    ro, rS, _ = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N + steps], threads=16)
    _, S_c, _ = oracle.gla(inp.q[:, :c], inp.k[:, :c], inp.v[:, :c], inp.a[:, :c], [0], [c],
                           threads=16)
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    state = to_dev(S_c.astype(np.float32), dev)
    o = torch.zeros((1, N + steps, nH, d), device=dev)
    T = N + steps
    err = torch.zeros(1, dtype=torch.int32, device=dev)

    def call(p0, n):
        # views starting at token p0; the token extent stays T so strides are unchanged
        off = p0 * nH * d
        hs.hs_linattn_prefill_from_state(hs.make_shape(1, nH, d, d, T - p0, kernel),
                                         q.view(-1)[off:], k.view(-1)[off:], v.view(-1)[off:],
                                         a.view(-1)[off:], o.view(-1)[off:], state, [p0], [n], 0,
                                         None, err)
    call(c, N - c)
    for s in range(steps):
        call(N + s, 1)
    torch.cuda.synchronize()
    assert err.item() == 0
    got = o.cpu().numpy()
    assert maxnorm_err(got[0, c:], ro[0, c:], axes=(0, 2)) <= TOL
    assert maxnorm_err(state.cpu().numpy(), rS, axes=(2, 3)) <= TOL


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("d", [64, 128])
def test_zero_and_identity_gates(kernel, d):
    _needs(kernel, d)
    dev = device()
    N, nH = 150, 2
    for fill in (-1e4, 0.0):
        inp = gen_linear(5, 0, 1, N, nH, d, d)
        inp.a[:] = fill
        S0 = gen_state(5, 0, 1, nH, d, d)
        o, S, cks = run_prefill(inp, [0], [N], S0, 64, dev, kernel)
        ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], S0=S0, C_=64)
        _check(o, S, cks, ro, rS, rck, [0], [N], f"gate={fill}")


@pytest.mark.parametrize("kernel", KERNELS)
def test_fused_checkpoints_equal_standalone_writer(kernel):
    """A prefill ending on a checkpoint boundary: its fused checkpoint equals a
    snapshot of the live state taken by hs_checkpoint_states, bit for bit."""
    dev = device()
    N, C, nH, d = 512, 256, 8, 128
    inp = gen_linear(6, 0, 1, N, nH, d, d)
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    state = torch.zeros((1, nH, d, d), device=dev)
    o = torch.zeros((1, N, nH, d), device=dev)
    slots = torch.zeros((2, nH, d, d), device=dev)
    snap = torch.zeros((nH, d, d), device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_linattn_prefill_from_state(hs.make_shape(1, nH, d, d, N, kernel), q, k, v, a, o, state,
                                     [0], [N], C, hs.ptr_array([slots[0], slots[1]], dev), err)
    hs.hs_checkpoint_states(hs.ptr_array([state], dev), hs.ptr_array([snap], dev), 1,
                            nH * d * d, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert torch.equal(slots[1].view(torch.int32), snap.view(torch.int32))


@pytest.mark.parametrize("kernel", KERNELS)
def test_checkpoint_slot_errors_are_reported(kernel):
    dev = device()
    N, nH, d = 128, 2, 128
    inp = gen_linear(7, 0, 1, N, nH, d, d)
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    state = torch.zeros((1, nH, d, d), device=dev)
    o = torch.zeros((1, N, nH, d), device=dev)
    slot = torch.zeros(nH * d * d + 4, device=dev)
    for ptrs, code in (([slot.data_ptr() + 4, slot.data_ptr()], hs.HS_DEVERR_MISALIGNED),
                       ([0, slot.data_ptr()], hs.HS_DEVERR_NULL)):
        err = torch.zeros(1, dtype=torch.int32, device=dev)
        state.zero_()
        hs.hs_linattn_prefill_from_state(hs.make_shape(1, nH, d, d, N, kernel), q, k, v, a, o,
                                         state, [0], [N], 64, hs.ptr_array(ptrs, dev), err)
        torch.cuda.synchronize()
        assert err.item() == code


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("L", LONG_LENGTHS)
def test_long_context_full_size_sampled_heads(kernel, L):
    """Long-context stack shape at L = 16384, 32768 and 65536: batch 4, 32 heads, d=128,
    C=512, inputs drawn on the device; sampled (request, head) pairs against the oracle,
    and the resumed tail (hit = L-37) bitwise against the full recomputation."""
    dev = device()
    from hs_inputs import torch_gen_linear
    C, B, nH, d = LONG24.ckpt, LONG24.batch, LONG24.n_heads, LONG24.d
    q, k, v, a = torch_gen_linear(11, 0, B, L, nH, d, dev)
    state = torch.zeros((B, nH, d, d), device=dev)
    o = torch.zeros((B, L, nH, d), device=dev)
    nck = hs.hs_linattn_num_checkpoints([0] * B, [L] * B, C)
    slots = torch.zeros((nck, nH, d, d), device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_linattn_prefill_from_state(hs.make_shape(B, nH, d, d, L, kernel), q, k, v, a, o, state,
                                     [0] * B, [L] * B, C,
                                     hs.ptr_array([slots[i] for i in range(nck)], dev), err)
    torch.cuda.synchronize()
    assert err.item() == 0
    c, _, tail = hs.hs_align_prefix(L, L - 37, list(range(C, L + 1, C)), LONG24.page)
    per = L // C
    # resume every request from its checkpoint at c
    st2 = torch.stack([slots[b * per + c // C - 1] for b in range(B)]).contiguous()
    o2 = torch.zeros((B, tail, nH, d), device=dev)
    sl2 = torch.zeros((B, nH, d, d), device=dev)
    hs.hs_linattn_prefill_from_state(hs.make_shape(B, nH, d, d, tail, kernel),
                                     q[:, c:].contiguous(), k[:, c:].contiguous(),
                                     v[:, c:].contiguous(), a[:, c:].contiguous(), o2, st2,
                                     [c] * B, [tail] * B, C,
                                     hs.ptr_array([sl2[b] for b in range(B)], dev), err)
    torch.cuda.synchronize()
    assert torch.equal(o2.view(torch.int32), o[:, c:].view(torch.int32))
    assert torch.equal(st2.view(torch.int32), state.view(torch.int32))
    assert torch.equal(sl2.view(torch.int32), slots[per - 1::per].view(torch.int32))
    # sampled heads against the oracle (float64, token by token)
    for b, h in ((0, 0), (3, 31)):
        qh = q[b:b + 1, :, h:h + 1].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        kh = k[b:b + 1, :, h:h + 1].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        vh = v[b:b + 1, :, h:h + 1].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        ah = a[b:b + 1, :, h:h + 1].contiguous().cpu().numpy()
        ro, rS, rck = oracle.gla(qh, kh, vh, ah, [0], [L], C_=C)
        assert maxnorm_err(o[b, :, h].cpu().numpy(), ro[0, :, 0], axes=(0, 1)) <= TOL
        assert maxnorm_err(state[b, h].cpu().numpy(), rS[0, 0], axes=(0, 1)) <= TOL
        got_ck = slots[b * per:(b + 1) * per, h].cpu().numpy()
        assert maxnorm_err(got_ck, rck[0][:, 0], axes=(1, 2)) <= TOL


@pytest.mark.parametrize("d", [64, 128])
def test_short_segments_match_across_kernels(d):
    """Calls whose tails are at most HS_SHORT_SEGMENT tokens: the tensor-core
    kernel's token-by-token path and the recurrent kernel agree bit for bit, so
    AUTO may send decode steps to either without changing results."""
    dev = device()
    B, nH, T = 6, 4, 8
    pos0 = [0, 5, 63, 64, 1000, 4095]
    n_tok = [8, 1, 2, 7, 3, 8]                       # some straddle a chunk boundary
    inp = gen_linear(13, 0, B, T, nH, d, d)
    S0 = gen_state(13, 0, B, nH, d, d)
    res = [run_prefill(inp, pos0, n_tok, S0, 64, dev, k)
           for k in (hs.HS_LINATTN_RECURRENT, hs.HS_LINATTN_CHUNKED_TC, hs.HS_LINATTN_AUTO)]
    for o, S, cks in res[1:]:
        for b, n in enumerate(n_tok):
            assert np.array_equal(o[b, :n].view(np.uint32), res[0][0][b, :n].view(np.uint32))
            assert np.array_equal(cks[b].view(np.uint32), res[0][2][b].view(np.uint32))
        assert np.array_equal(S.view(np.uint32), res[0][1].view(np.uint32))
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, pos0, n_tok, S0=S0, C_=64)
    _check(*res[0], ro, rS, rck, pos0, n_tok, "short")


@pytest.mark.parametrize("d", [64, 128])
def test_single_token_steps_match_across_kernels(d):
    """Decode steps (at most one token per problem): the single-token kernel, the
    recurrent kernel, the tensor-core kernel's token-by-token path and AUTO agree
    bit for bit over consecutive steps, including a step that ends on a checkpoint
    boundary and problems without a token; the result follows the oracle."""
    dev = device()
    B, nH, steps, C = 5, 4, 6, 64
    pos0 = [0, 61, 126, 4093, 700]      # problems 1-3 cross a 64-token boundary in these steps
    inp = gen_linear(21, d, B, steps, nH, d, d)
    S0 = gen_state(21, d, B, nH, d, d)
    kernels = [hs.HS_LINATTN_SINGLE_TOKEN, hs.HS_LINATTN_RECURRENT, hs.HS_LINATTN_AUTO,
               hs.HS_LINATTN_CHUNKED_TC]
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    tok_b, tok_f = nH * d * 2, nH * d * 4
    res = []
    for kern in kernels:
        state = to_dev(np.asarray(S0, np.float32), dev)
        o = torch.full((B, steps, nH, d), float("nan"), device=dev)
        slots = torch.full((B * steps, nH, d, d), float("nan"), device=dev)
        ptrs = hs.ptr_array([slots[i] for i in range(B * steps)], dev)
        err = torch.zeros(1, dtype=torch.int32, device=dev)
        shape = hs.make_shape(B, nH, d, d, steps, kern)
        for j in range(steps):
            n_tok = [0 if (b == 4 and j % 2) else 1 for b in range(B)]   # problem 4: every other step
            p0 = [pos0[b] + j for b in range(B)]
            # one checkpoint slot per problem and step (only boundary steps write theirs)
            base = [b * steps + j for b in range(B)]
            hs.hs_linattn_prefill_from_state(
                shape, q.data_ptr() + j * tok_b, k.data_ptr() + j * tok_b,
                v.data_ptr() + j * tok_b, a.data_ptr() + j * tok_f, o.data_ptr() + j * tok_f,
                state, p0, n_tok, C, _slots_for(p0, n_tok, C, slots, base, dev), err)
        torch.cuda.synchronize()
        assert err.item() == 0
        res.append((o.cpu().numpy(), state.cpu().numpy(), slots.cpu().numpy()))
    for o, S, sl in res[1:]:
        assert np.array_equal(o.view(np.uint32), res[0][0].view(np.uint32))
        assert np.array_equal(S.view(np.uint32), res[0][1].view(np.uint32))
        assert np.array_equal(sl.view(np.uint32), res[0][2].view(np.uint32))
    # oracle: problem 4 sees its tokens 0, 2, 4 (odd steps carry none)
    o0, S_end, sl0 = res[0]
    for b in range(B):
        js = [j for j in range(steps) if not (b == 4 and j % 2)]
        sub = type(inp)(*(x[b:b + 1, js] for x in (inp.q, inp.k, inp.v, inp.a)))
        ro, rS, rck = oracle.gla(sub.q, sub.k, sub.v, sub.a, [pos0[b]], [len(js)],
                                 S0=S0[b:b + 1], C_=C)
        assert maxnorm_err(o0[b, js], ro[0], axes=(0, 2)) <= TOL
        assert maxnorm_err(S_end[b:b + 1], rS, axes=(2, 3)) <= TOL
        jb = [j for j in js if (pos0[b] + j + 1) % C == 0]      # steps ending on the grid
        assert rck[0].shape[0] == len(jb) == (1 if b in (1, 2, 3) else 0)
        for m, j in enumerate(jb):
            assert maxnorm_err(sl0[b * steps + j], rck[0][m], axes=(1, 2)) <= TOL


def _slots_for(p0, n_tok, C, slots, base, dev):
    """Checkpoint-slot array of one call: one entry per checkpoint the call emits, in
    problem order (the layout hs_linattn_num_checkpoints counts)."""
    ptrs = [slots[base[b]] for b in range(len(p0))
            if n_tok[b] and (p0[b] + n_tok[b]) // C - p0[b] // C]
    return hs.ptr_array(ptrs, dev) if ptrs else None


@pytest.mark.parametrize("suffix", [1, 3, 4, 5, 8, 9, 64, 65, 127])
def test_table4_suffix_lengths_auto_resume_bitwise(suffix):
    """The repaired path recomputes suffixes of 1, 3, 4, 5 and 1,791-1,792 tokens
    (the paper's Table 4); with the default kernel choice a resumed tail of any
    length reproduces the full recomputation bit for bit."""
    dev = device()
    C, c, nH, d = 128, 256, 4, 128
    N = c + suffix
    inp = gen_linear(14, suffix, 1, N, nH, d, d)
    o_f, S_f, ck_f, = _resume_equals_recompute(inp, N, c, C, dev, hs.HS_LINATTN_AUTO)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, [0], [N], C_=C)
    _check(o_f, S_f, ck_f, ro, rS, rck, [0], [N], f"suffix={suffix}")


@pytest.mark.parametrize("kernel", KERNELS)
def test_offset_views_read_only_the_given_tokens(kernel):
    """Views that start mid-sequence (pointer offset by c tokens, batch stride kept)
    read and write only rows t < n_tokens: the last problem's rows end exactly at the
    end of the allocation, and results equal those of a contiguous copy, bitwise."""
    dev = device()
    B, T, nH, d, c = 3, 320, 2, 128, 192
    inp = gen_linear(15, 0, B, T, nH, d, d)
    S0 = gen_state(15, 0, B, nH, d, d)
    sub = type(inp)(*(np.ascontiguousarray(x[:, c:]) for x in (inp.q, inp.k, inp.v, inp.a)))
    o_ref, S_ref, _ = run_prefill(sub, [c] * B, [T - c] * B, S0, 0, dev, kernel, want_ckpts=False)
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    o = torch.full((B, T, nH, d), 7.0, device=dev)
    state = to_dev(S0, dev)
    off = c * nH * d
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_linattn_prefill_from_state(hs.make_shape(B, nH, d, d, T, kernel),
                                     q.data_ptr() + 2 * off, k.data_ptr() + 2 * off,
                                     v.data_ptr() + 2 * off, a.data_ptr() + 4 * off,
                                     o.data_ptr() + 4 * off, state, [c] * B, [T - c] * B, 0, None,
                                     err)
    torch.cuda.synchronize()
    assert err.item() == 0
    got = o.cpu().numpy()
    assert np.array_equal(got[:, c:].view(np.uint32), o_ref[:, :T - c].view(np.uint32))
    assert (got[:, :c] == 7.0).all()
    assert np.array_equal(state.cpu().numpy().view(np.uint32), S_ref.view(np.uint32))


@pytest.mark.parametrize("kernel", KERNELS + [pytest.param(hs.HS_LINATTN_AUTO, id="auto")])
def test_packed_layout_equals_padded_bitwise(kernel):
    """A batch of tails with different resume points and lengths (0, ragged, several chunks),
    packed back to back without padding, gives the padded layout's outputs, final states and
    checkpoints bit for bit, and those follow the oracle."""
    dev = device()
    nH, d, T, C = 4, 128, 200, 64
    pos0 = [64, 0, 4093, 700, 130]
    n_tok = [200, 0, 37, 129, 5]
    B = len(pos0)
    inp = gen_linear(31, 0, B, T, nH, d, d)
    S0 = gen_state(31, 0, B, nH, d, d)
    o_pad, S_pad, ck_pad = run_prefill(inp, pos0, n_tok, S0, C, dev, kernel)
    cu = [0]
    for n in n_tok:
        cu.append(cu[-1] + n)
    cat = lambda x: np.concatenate([x[b, :n_tok[b]] for b in range(B)], axis=0)[None]
    q, k, v, a = (to_dev(cat(x), dev) for x in (inp.q, inp.k, inp.v, inp.a))
    state = to_dev(np.asarray(S0, np.float32), dev)
    o = torch.full((cu[-1], nH, d), float("nan"), device=dev)
    nck = hs.hs_linattn_num_checkpoints(pos0, n_tok, C)
    slots = torch.full((nck, nH, d, d), float("nan"), device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    hs.hs_linattn_prefill_packed(hs.make_shape(B, nH, d, d, 0, kernel), q, k, v, a, o, state,
                                 pos0, n_tok, cu, C, hs.ptr_array([slots[i] for i in range(nck)], dev),
                                 err)
    torch.cuda.synchronize()
    assert err.item() == 0
    o_p = o.cpu().numpy()
    for b in range(B):
        assert np.array_equal(o_p[cu[b]:cu[b + 1]].view(np.uint32), o_pad[b, :n_tok[b]].view(np.uint32))
    assert np.array_equal(state.cpu().numpy().view(np.uint32), S_pad.view(np.uint32))
    assert np.array_equal(slots.cpu().numpy().view(np.uint32),
                          np.concatenate(ck_pad, axis=0).view(np.uint32))
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, pos0, n_tok, S0=S0, C_=C)
    _check(o_pad, S_pad, ck_pad, ro, rS, rck, pos0, n_tok, "packed")


def test_packed_decode_steps_match_padded():
    """One token per problem from a packed layout (cu_rows = 0..B) through the single-token
    kernel equals the padded call bit for bit."""
    dev = device()
    nH, d, B = 8, 128, 6
    inp = gen_linear(32, 0, B, 1, nH, d, d)
    S0 = gen_state(32, 0, B, nH, d, d)
    pos0 = [10, 63, 127, 4000, 2, 511]
    o_pad, S_pad, _ = run_prefill(inp, pos0, [1] * B, S0, 64, dev, hs.HS_LINATTN_SINGLE_TOKEN)
    q, k, v, a = (to_dev(x.reshape(1, B, nH, d), dev) for x in (inp.q, inp.k, inp.v, inp.a))
    state = to_dev(np.asarray(S0, np.float32), dev)
    o = torch.empty((B, nH, d), device=dev)
    hs.hs_linattn_prefill_packed(hs.make_shape(B, nH, d, d, 0, hs.HS_LINATTN_SINGLE_TOKEN), q, k,
                                 v, a, o, state, pos0, [1] * B, list(range(B + 1)), 0)
    torch.cuda.synchronize()
    assert np.array_equal(o.cpu().numpy().view(np.uint32), o_pad[:, 0].view(np.uint32))
    assert np.array_equal(state.cpu().numpy().view(np.uint32), S_pad.view(np.uint32))
