"""Failure detection on the GPU without a fault: every wait of the tensor-core prefill is
bounded, and a wait that runs out ends the kernel through its abort path with a status the
host reads.  The hook hs_test_prefill_stalled (include/hs_test.h) makes one wait per CTA on
an mbarrier that nothing completes; the test checks the reported code, that nothing was
written, and that the same context then runs a normal call correctly."""
import time

import numpy as np
import pytest
import torch

import oracle
import paper_2609_15030_gb300 as hs
from hs_inputs import gen_linear, gen_state
from tests.gpu_helpers import TOL, device, maxnorm_err, run_prefill, to_dev

pytestmark = pytest.mark.gpu


def test_a_wait_that_runs_out_reports_timeout_and_leaves_the_context_usable():
    dev = device()
    B, nH, d, C = 2, 2, 128, 64
    pos0, n_tok = [64, 5], [130, 77]
    T = max(n_tok)
    inp = gen_linear(4242, 0, B, T, nH, d, d)
    S0 = gen_state(4242, 0, B, nH, d, d)
    q, k, v, a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
    state = to_dev(S0, dev)
    o = torch.full((B, T, nH, d), float("nan"), device=dev)
    nck = hs.hs_linattn_num_checkpoints(pos0, n_tok, C)
    slots = torch.full((nck, nH, d, d), float("nan"), device=dev)
    ptrs = hs.ptr_array([slots[i] for i in range(nck)], dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    shape = hs.make_shape(B, nH, d, d, T, hs.HS_LINATTN_CHUNKED_TC)
    t0 = time.perf_counter()
    hs.hs_test_prefill_stalled(shape, q, k, v, a, o, state, pos0, n_tok, C, ptrs, err)
    torch.cuda.synchronize()
    waited = time.perf_counter() - t0
    assert int(err.item()) == hs.HS_DEVERR_TIMEOUT
    assert 0.9 < waited < 30.0                       # the 1 s bound, not a hang
    # the CTAs left before any segment: nothing written
    assert torch.isnan(o).all()
    assert torch.isnan(slots).all()
    assert np.array_equal(state.cpu().numpy().view(np.uint32), S0.view(np.uint32))
    # the same context, the normal call, against the oracle
    o2, S2, cks = run_prefill(inp, pos0, n_tok, S0, C, dev, hs.HS_LINATTN_CHUNKED_TC)
    ro, rS, rck = oracle.gla(inp.q, inp.k, inp.v, inp.a, pos0, n_tok, S0=S0, C_=C)
    for b, n in enumerate(n_tok):
        assert maxnorm_err(o2[b, :n], ro[b, :n], axes=(0, 2)) <= TOL
    assert maxnorm_err(S2, rS, axes=(2, 3)) <= TOL
