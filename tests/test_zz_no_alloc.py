"""hs_linattn_prefill_scan_noalloc on the GPU, through the C ABI, against hs_linattn_prefill_scan.

The allocation-free entry point serves callers that cannot allocate device memory when they
resume a request: a serving engine that handed nearly all of its HBM to the KV-cache pool at
start-up, or a scheduler loop that must not take the device-wide synchronisation of cudaMalloc
or cudaFree.  It runs the segment-parallel prefill with the library's fixed 16 MiB per-device
workspace instead of a caller's.  Two calls in a row, of different shapes (the first at the
workspace's full size, the second a ragged batch that finds the first call's data in the
shared workspace), must each give the results of the entry point with a caller workspace,
within the parity bar the other prefill tests use.

The file is named so that pytest collects it last.  It passes alone in a fresh process, where
its first call does the entry point's one-time set-up on the device, and after the other tests.
"""
import numpy as np
import pytest
import torch

import paper_2609_15030_gb300 as hs
from hs_inputs import gen_linear, gen_state
from tests.gpu_helpers import TOL, device, maxnorm_err, to_dev

pytestmark = pytest.mark.gpu


class _Call:
    """Device inputs and result buffers of one prefill call (NaN-filled outputs)."""

    def __init__(self, dev, seed, B, nH, d, T, pos0, n_tokens, C):
        self.B, self.nH, self.d, self.T = B, nH, d, T
        self.pos0, self.n_tokens, self.C = pos0, n_tokens, C
        inp = gen_linear(seed, 0, B, T, nH, d, d, "uniform")
        self.q, self.k, self.v, self.a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
        self.S0 = torch.from_numpy(gen_state(seed, 1, B, nH, d, d)).to(dev)
        self.nck = hs.hs_linattn_num_checkpoints(pos0, n_tokens, C)
        self.shape = hs.make_shape(B, nH, d, d, T)
        self.err = torch.zeros(1, dtype=torch.int32, device=dev)

    def buffers(self, dev):
        state = self.S0.clone()
        o = torch.full((self.B, self.T, self.nH, self.d), float("nan"), device=dev)
        slots = torch.full((max(self.nck, 1), self.nH, self.d, self.d), float("nan"), device=dev)
        ptrs = hs.ptr_array([slots[i] for i in range(self.nck)], dev) if self.nck else None
        return state, o, slots, ptrs

    def args(self, state, o, ptrs):
        return (self.shape, self.q, self.k, self.v, self.a, o, state, self.pos0, self.n_tokens,
                self.C, ptrs)


def _compare(got, ref, n_tokens):
    (o, S, ck), (ro, rS, rck) = got, ref
    for b, n in enumerate(n_tokens):
        if n:
            assert maxnorm_err(o[b, :n], ro[b, :n], axes=(0, 2)) <= TOL, b
            assert np.isnan(o[b, n:]).all()
    assert maxnorm_err(S, rS, axes=(2, 3)) <= TOL
    assert ck.shape == rck.shape
    if ck.shape[0]:
        assert maxnorm_err(ck, rck, axes=(2, 3)) <= TOL


def test_noalloc_matches_the_workspace_entry_point_on_two_calls_in_a_row():
    dev = device()
    calls = [
        # one problem of 16 heads, 512 tokens from 4096: needs exactly the 16 MiB workspace
        _Call(dev, 71, B=1, nH=16, d=128, T=512, pos0=[4096], n_tokens=[512], C=512),
        # a ragged batch with off-grid resume points, a short tail, an empty one, checkpoints
        _Call(dev, 72, B=5, nH=3, d=128, T=200, pos0=[100, 0, 640, 64, 7],
              n_tokens=[37, 200, 5, 129, 0], C=128),
    ]
    assert hs.hs_linattn_scan_workspace_bytes(calls[0].shape, [4096], [512]) == \
        hs.HS_NOALLOC_SCRATCH_BYTES
    stream = torch.cuda.current_stream(dev)

    # the two allocation-free calls back to back on one stream
    got = []
    for i, c in enumerate(calls):
        state, o, slots, ptrs = c.buffers(dev)
        torch.cuda.synchronize()
        before = (torch.cuda.memory_allocated(dev), torch.cuda.mem_get_info(dev)[0])
        hs.hs_linattn_prefill_scan_noalloc(*c.args(state, o, ptrs), c.err, stream)
        torch.cuda.synchronize()
        if i > 0:       # after the first call's set-up, a call changes no device allocation
            assert (torch.cuda.memory_allocated(dev), torch.cuda.mem_get_info(dev)[0]) == before
        assert int(c.err.item()) == 0
        got.append((o.cpu().numpy(), state.cpu().numpy(), slots[:c.nck].cpu().numpy()))

    # the same calls through hs_linattn_prefill_scan with a caller workspace
    for c, g in zip(calls, got):
        state, o, slots, ptrs = c.buffers(dev)
        nb = hs.hs_linattn_scan_workspace_bytes(c.shape, c.pos0, c.n_tokens)
        ws = torch.full((nb // 4,), float("nan"), device=dev)
        hs.hs_linattn_prefill_scan(*c.args(state, o, ptrs), ws, nb, c.err, stream)
        torch.cuda.synchronize()
        assert int(c.err.item()) == 0
        ref = (o.cpu().numpy(), state.cpu().numpy(), slots[:c.nck].cpu().numpy())
        _compare(g, ref, c.n_tokens)
