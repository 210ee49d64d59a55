"""Seeded stress calls of the prefill kernels against the float64 oracle.

Each call (``hs_inputs.gen_stress_case``) draws a random batch, resume points, tail lengths
and checkpoint interval, then plants stress on random token ranges: growing gates, strong
gates (-30, -1.2), a zero gate, v scaled by 2^17, q and k scaled by 64, starting states up to
2^16.  Every kernel that accepts the call (AUTO, the recurrent kernel, the tensor-core
kernel, the single-token kernel for calls of at most one token per problem) must stay
within the max-normalised error bound 2e-3 for outputs, final states and checkpoints.

The paper makes numerical control part of the method (Section 4, Table 3): these calls are
the committed part of that control for this library.  Seeds 90147, 100669 and 102867 are
calls where the tensor-core kernel once reached 2.02e-3, 2.12e-3 and 2.72e-3: in each, one
token whose own q . k cancels dominates its head's outputs.
"""
import numpy as np
import pytest

import oracle
import paper_2609_15030_gb300 as hs
from hs_inputs import gen_stress_case
from tests.gpu_helpers import TOL, device, maxnorm_err, run_prefill, run_scan_prefill

pytestmark = pytest.mark.gpu

KNOWN = [90147, 100669, 102867]
BLOCK = 25
BLOCKS = 12                 # 300 seeds from 200000
SCAN_BLOCKS = 4             # 100 seeds from 210000 through the segment-parallel prefill


def _kernels(case):
    ks = [hs.HS_LINATTN_AUTO, hs.HS_LINATTN_RECURRENT, hs.HS_LINATTN_CHUNKED_TC]
    if max(case.n_tokens) <= 1:
        ks.append(hs.HS_LINATTN_SINGLE_TOKEN)
    return ks


def _worst(seed, dev):
    """Largest error of any kernel on stress call `seed` (outputs, states, checkpoints)."""
    c = gen_stress_case(seed)
    x = c.inputs
    ro, rS, rck = oracle.gla(x.q, x.k, x.v, x.a, c.pos0, c.n_tokens, S0=c.S0,
                             C_=c.ckpt_interval, threads=16)
    worst = 0.0
    for kernel in _kernels(c):
        o, S, cks = run_prefill(x, c.pos0, c.n_tokens, c.S0, c.ckpt_interval, dev, kernel)
        errs = [maxnorm_err(S, rS, axes=(2, 3))]
        for b, n in enumerate(c.n_tokens):
            if n:
                errs.append(maxnorm_err(o[b, :n], ro[b, :n], axes=(0, 2)))
            assert cks[b].shape == rck[b].shape
            if cks[b].shape[0]:
                errs.append(maxnorm_err(cks[b], rck[b], axes=(2, 3)))
        e = max(errs)
        assert np.isfinite(e), (seed, kernel)
        worst = max(worst, e)
    return worst


@pytest.mark.parametrize("seed", KNOWN)
def test_known_worst_calls(seed):
    dev = device()
    e = _worst(seed, dev)
    assert e <= TOL, f"stress call {seed}: {e:.3g}"


@pytest.mark.parametrize("block", range(BLOCKS))
def test_seeded_stress_calls(block):
    dev = device()
    bad = []
    for seed in range(200000 + BLOCK * block, 200000 + BLOCK * (block + 1)):
        e = _worst(seed, dev)
        if not e <= TOL:
            bad.append((seed, round(e, 6)))
    assert not bad, f"calls above {TOL}: {bad}"


def _scan_error(seed, dev):
    """Largest error of the segment-parallel prefill on stress call `seed`."""
    c = gen_stress_case(seed)
    x = c.inputs
    ro, rS, rck = oracle.gla(x.q, x.k, x.v, x.a, c.pos0, c.n_tokens, S0=c.S0,
                             C_=c.ckpt_interval, threads=16)
    o, S, cks = run_scan_prefill(x, c.pos0, c.n_tokens, c.S0, c.ckpt_interval, dev)
    errs = [maxnorm_err(S, rS, axes=(2, 3))]
    for b, n in enumerate(c.n_tokens):
        if n:
            errs.append(maxnorm_err(o[b, :n], ro[b, :n], axes=(0, 2)))
        assert cks[b].shape == rck[b].shape
        if cks[b].shape[0]:
            errs.append(maxnorm_err(cks[b], rck[b], axes=(2, 3)))
    e = max(errs)
    assert np.isfinite(e), seed
    return e


@pytest.mark.parametrize("block", range(SCAN_BLOCKS))
def test_seeded_stress_calls_segment_parallel(block):
    """The same kind of calls through hs_linattn_prefill_scan: its segment-state pass (tf32
    products), the fp32 scan and the guarded output pass stay within the bar too."""
    dev = device()
    bad = []
    for seed in range(210000 + BLOCK * block, 210000 + BLOCK * (block + 1)):
        e = _scan_error(seed, dev)
        if not e <= TOL:
            bad.append((seed, round(e, 6)))
    assert not bad, f"calls above {TOL}: {bad}"

