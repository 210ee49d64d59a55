"""Parity at full size, in the launch configuration bench.py times.

Builds the benchmark's nine-length hybrid workload (9 linear layers x 16 heads
x d=128 folded into one batch, 3 full-attention layers), replays its CUDA
graphs for one request and checks:
  * KV pages of [0,c) in the paged cache are byte-equal to the staging pool;
  * the live state after restore + tail + 64 decode steps, and every output
    token, match the float64 oracle on sampled (layer, head) pairs, starting
    from the restored checkpoint;
  * the checkpoint emitted at L matches the oracle's state after the tail.
"""
import numpy as np
import pytest
import torch

import oracle
from tests.gpu_helpers import TOL, device, maxnorm_err

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("r", range(9))          # L = 512, 1024, ..., 4608
def test_hybrid_workload_request_matches_oracle(r):
    dev = device()
    import bench
    wl = bench.Hybrid12(dev, seeds=1, num_blocks=2048)
    wl.capture()
    R, I, O = wl.req[r], wl.inp[(0, r)], wl.out[r]
    O["live"].fill_(float("nan"))
    wl.cache.fill_(0xFF)
    wl.request(0, r)
    torch.cuda.synchronize()
    # KV restore: byte-exact
    n_pages, P = R["n_pages"], wl.page_bytes
    if n_pages:
        bt = I["bt"].long()
        for l in range(wl.nF):
            got = wl.cache[l].view(wl.NB, P)[bt]
            assert torch.equal(got, I["staging"][l].view(-1, P)[:n_pages])
    # linear layers: restored checkpoint -> tail (checkpoint at L) -> 64 decode steps
    c, L, T = R["c"], R["L"], wl.T
    for layer, h in ((0, 0), (4, 7), (8, 15)):
        q = _bits(I["q"][layer:layer + 1, :, h:h + 1])
        k = _bits(I["k"][layer:layer + 1, :, h:h + 1])
        v = _bits(I["v"][layer:layer + 1, :, h:h + 1])
        a = I["a"][layer:layer + 1, :, h:h + 1].contiguous().cpu().numpy()
        S0 = I["ck"][layer].view(wl.nH, wl.d, wl.d)[h].cpu().numpy()[None, None]
        ro, rS, _ = oracle.gla(q, k, v, a, [c], [T], S0=S0)
        _, rS_tail, _ = oracle.gla(q[:, :bench.TAIL], k[:, :bench.TAIL], v[:, :bench.TAIL],
                                   a[:, :bench.TAIL], [c], [bench.TAIL], S0=S0)
        got_o = O["o"][layer, :, h].cpu().numpy()
        assert maxnorm_err(got_o, ro[0, :, 0], axes=(0, 1)) <= TOL
        got_S = O["live"][layer].view(wl.nH, wl.d, wl.d)[h].cpu().numpy()
        assert maxnorm_err(got_S, rS[0, 0], axes=(0, 1)) <= TOL
        got_ck = O["emit"][layer].view(wl.nH, wl.d, wl.d)[h].cpu().numpy()
        assert maxnorm_err(got_ck, rS_tail[0, 0], axes=(0, 1)) <= TOL
    assert not torch.isnan(O["live"]).any()
