"""The library keeps no state between calls: work on two streams at once, and the same calls
captured in a CUDA graph and replayed, give the bytes of the same calls made one by one."""
import numpy as np
import pytest
import torch

import paper_2609_15030_gb300 as hs
from hs_inputs import gen_block_table, gen_kv_pages, gen_linear, gen_state
from tests.gpu_helpers import device, to_dev

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.contiguous().view(torch.int32).cpu().numpy()


class _Request:
    """One resumed request on the device: KV pages of [0,c) for 2 attention layers, the
    states at c for B linear problems, the tail and 4 decode tokens."""

    def __init__(self, dev, seed, B=3, nH=8, d=128, c=512, tail=200, steps=4, P=32768, nb=64):
        self.B, self.nH, self.d, self.c, self.tail, self.steps = B, nH, d, c, tail, steps
        self.P, self.nb, self.n_pages = P, nb, c // 16
        T = tail + steps
        inp = gen_linear(seed, 0, B, T, nH, d, d, "uniform")
        self.q, self.k, self.v, self.a = (to_dev(x, dev) for x in (inp.q, inp.k, inp.v, inp.a))
        self.ck = torch.from_numpy(gen_state(seed, 1, B, nH, d, d)).to(dev)
        self.staging = [torch.from_numpy(gen_kv_pages(seed, l, self.n_pages, P).reshape(-1)).to(dev)
                        for l in range(2)]
        self.bt = torch.from_numpy(gen_block_table(seed, 0, self.n_pages, nb)).to(dev)
        self.o = torch.empty((B, T, nH, d), device=dev)
        self.live = torch.empty((B, nH, d, d), device=dev)
        self.slots = torch.empty((B, nH, d, d), device=dev)
        self.cache = [torch.empty(nb * P, dtype=torch.uint8, device=dev) for _ in range(2)]
        self.stg_ptrs = hs.ptr_array(self.staging, dev)
        self.cache_ptrs = hs.ptr_array(self.cache, dev)
        self.src_ptrs = hs.ptr_array([self.ck[b] for b in range(B)], dev)
        self.live_ptrs = hs.ptr_array([self.live[b] for b in range(B)], dev)
        self.slot_ptrs = hs.ptr_array([self.slots[b] for b in range(B)], dev)

    def reset(self):
        self.o.fill_(float("nan"))
        self.live.fill_(float("nan"))
        self.slots.fill_(float("nan"))
        for c in self.cache:
            c.fill_(0xEE)

    def run(self, stream):
        """Restore, tail prefill, decode steps, then the live states snapshotted into slots."""
        B, nH, d, s = self.B, self.nH, self.d, stream.cuda_stream
        hs.hs_restore_request(self.stg_ptrs, self.cache_ptrs, 2, self.bt, self.n_pages, self.P,
                              self.nb, self.src_ptrs, self.live_ptrs, B, nH * d * d, None, s)
        shape = hs.make_shape(B, nH, d, d, self.tail + self.steps)
        hs.hs_linattn_prefill_from_state(shape, self.q, self.k, self.v, self.a, self.o, self.live,
                                         [self.c] * B, [self.tail] * B, 0, None, None, s)
        tb, tbf = nH * d * 2, nH * d * 4
        for j in range(self.steps):
            t = self.tail + j
            hs.hs_linattn_prefill_from_state(
                shape, self.q.data_ptr() + t * tb, self.k.data_ptr() + t * tb,
                self.v.data_ptr() + t * tb, self.a.data_ptr() + t * tbf,
                self.o.data_ptr() + t * tbf, self.live, [self.c + t] * B, [1] * B, 0, None, None, s)
        hs.hs_checkpoint_states(self.live_ptrs, self.slot_ptrs, B, nH * d * d, None, s)

    def result(self):
        return [_bits(self.o), _bits(self.live), _bits(self.slots)] + \
               [c.cpu().numpy() for c in self.cache]


def _same(x, y):
    assert len(x) == len(y)
    for a, b in zip(x, y):
        assert np.array_equal(a, b)


def test_two_streams_at_once_equal_one_by_one():
    dev = device()
    r1, r2 = _Request(dev, 31), _Request(dev, 32, B=2, c=1024, tail=130)
    s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ref = []
    for r in (r1, r2):
        r.reset()
        torch.cuda.synchronize()      # the fills run on the current stream
        r.run(s1)
        torch.cuda.synchronize()
        ref.append(r.result())
    for _ in range(3):
        r1.reset()
        r2.reset()
        torch.cuda.synchronize()
        r1.run(s1)
        r2.run(s2)
        torch.cuda.synchronize()
        _same(r1.result(), ref[0])
        _same(r2.result(), ref[1])


def test_graph_replay_equals_eager_calls():
    dev = device()
    r = _Request(dev, 33)
    s = torch.cuda.Stream(dev)
    r.reset()
    torch.cuda.synchronize()
    r.run(s)
    torch.cuda.synchronize()
    ref = r.result()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s, capture_error_mode="relaxed"):
        r.run(torch.cuda.current_stream(dev))
    for _ in range(2):
        r.reset()
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        _same(r.result(), ref)
