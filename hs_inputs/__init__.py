"""Seeded synthetic inputs shared by the oracle side and the CUDA side.

This module only draws random numbers and lays them out.  It holds none of
the method's arithmetic (no alignment, no recurrence, no copies): both the
float64 oracle (``oracle/``) and the CUDA library consume what it produces,
so it is the single place where the two sides meet.

Value recipes (the paper's prompts and weights are not public, so every
tensor is synthetic; the shapes follow the workloads described in the
paper's serial prompt-length sweep, Section 5.1 and Table 1):

* ``"sigmoid"`` gates (tiny hybrid stack): q, k, v ~ N(0,1)/8 rounded to
  bf16; log-gates a = log(sigmoid(x)), x ~ N(2, 0.5), computed in float64
  and rounded to float32, one per (token, head, d_k).
* ``"uniform"`` gates (sweep / hybrid / long-context stacks): q, k, v ~
  N(0,1)/sqrt(d), k L2-normalised per (token, head) in float32 before the
  bf16 cast; log-gates a ~ U(-0.1, 0) in float32.
* KV staging pages: N(0,1) rounded to bf16, viewed as raw bytes.
* Block tables: distinct block ids drawn uniformly without replacement.

Every draw uses ``numpy.random.default_rng([seed, layer, stream])`` so that
layer i of seed s is reproducible on its own.  Large workloads use the
torch generator on the device instead (``torch_*`` helpers).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

# streams inside one (seed, layer) key
_Q, _K, _V, _A, _KV, _BT, _S0 = range(7)


def rng_for(seed: int, layer: int, stream: int) -> np.random.Generator:
    return np.random.default_rng([int(seed), int(layer), int(stream)])


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (round to nearest, ties to even); uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16).astype(np.uint16)
    return r


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass
class LinearInputs:
    """One linear-attention layer's inputs for a batch of requests.

    q, k: uint16 bf16 bits [B, T, nH, d_k]; v: uint16 [B, T, nH, d_v];
    a: float32 log-gates [B, T, nH, d_k]; token t of request b is the
    absolute position pos0[b] + t.
    """
    q: np.ndarray
    k: np.ndarray
    v: np.ndarray
    a: np.ndarray


def gen_linear(seed: int, layer: int, batch: int, n_tokens: int, n_heads: int,
               d_k: int, d_v: int, gates: str = "uniform") -> LinearInputs:
    shp_k = (batch, n_tokens, n_heads, d_k)
    shp_v = (batch, n_tokens, n_heads, d_v)
    rq, rk, rv, ra = (rng_for(seed, layer, s) for s in (_Q, _K, _V, _A))
    if gates == "sigmoid":
        q = rq.standard_normal(shp_k) / 8.0
        k = rk.standard_normal(shp_k) / 8.0
        v = rv.standard_normal(shp_v) / 8.0
        x = ra.normal(2.0, 0.5, size=shp_k)
        a = -np.log1p(np.exp(-x))          # log(sigmoid(x)) in float64
        a = a.astype(np.float32)
        k32 = k.astype(np.float32)
    elif gates == "uniform":
        q = rq.standard_normal(shp_k) / math.sqrt(d_k)
        k = rk.standard_normal(shp_k) / math.sqrt(d_k)
        v = rv.standard_normal(shp_v) / math.sqrt(d_v)
        k32 = k.astype(np.float32)
        nrm = np.sqrt(np.sum(k32 * k32, axis=-1, keepdims=True, dtype=np.float32))
        k32 = (k32 / nrm).astype(np.float32)
        a = ra.uniform(-0.1, 0.0, size=shp_k).astype(np.float32)
    else:
        raise ValueError(gates)
    return LinearInputs(q=f32_to_bf16_bits(q.astype(np.float32)),
                        k=f32_to_bf16_bits(k32),
                        v=f32_to_bf16_bits(v.astype(np.float32)),
                        a=a)


def gen_state(seed: int, layer: int, batch: int, n_heads: int, d_k: int, d_v: int,
              scale: float = 0.5) -> np.ndarray:
    """A float32 state [B, nH, d_k, d_v] for tests that start off the zero state."""
    r = rng_for(seed, layer, _S0)
    return (r.standard_normal((batch, n_heads, d_k, d_v)) * scale).astype(np.float32)


def gen_kv_pages(seed: int, layer: int, n_pages: int, page_bytes: int) -> np.ndarray:
    """Staging pages [n_pages, page_bytes] uint8 holding N(0,1) bf16 values."""
    assert page_bytes % 2 == 0
    r = rng_for(seed, layer, _KV)
    x = r.standard_normal((n_pages, page_bytes // 2)).astype(np.float32)
    return f32_to_bf16_bits(x).view(np.uint8).reshape(n_pages, page_bytes)


def gen_block_table(seed: int, request: int, n_pages: int, num_blocks: int) -> np.ndarray:
    """n_pages distinct block ids, uniform without replacement over [0, num_blocks)."""
    r = rng_for(seed, request, _BT)
    if n_pages > num_blocks:
        raise ValueError("more pages than blocks")
    if num_blocks <= 4 * n_pages or num_blocks < 1 << 16:
        return r.permutation(num_blocks)[:n_pages].astype(np.int32)
    # sparse draw for very large pools: rejection on a set
    out, seen = [], set()
    while len(out) < n_pages:
        for b in r.integers(0, num_blocks, size=2 * (n_pages - len(out))):
            b = int(b)
            if b not in seen:
                seen.add(b)
                out.append(b)
                if len(out) == n_pages:
                    break
    return np.asarray(out, dtype=np.int32)


# ---------------------------------------------------------------------------
# device-side generation for workloads too large for numpy (torch plumbing)
# ---------------------------------------------------------------------------

def torch_gen_linear(seed: int, layer: int, batch: int, n_tokens: int, n_heads: int,
                     d: int, device, gates: str = "uniform"):
    """Same recipe as ``gen_linear`` ("uniform" gates) drawn by torch's
    generator on ``device``; returns (q, k, v, a) torch tensors (bf16 x3,
    float32).  Values differ from the numpy draw; tests that need the oracle
    copy slices back to the host."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1_000_003 + int(layer) * 7919 + 17) & 0x7FFFFFFFFFFF)
    shp = (batch, n_tokens, n_heads, d)
    if gates == "uniform":
        q = (torch.randn(shp, generator=g, device=device) / math.sqrt(d)).to(torch.bfloat16)
        k = torch.randn(shp, generator=g, device=device)
        k = (k / k.norm(dim=-1, keepdim=True)).to(torch.bfloat16)
        v = (torch.randn(shp, generator=g, device=device) / math.sqrt(d)).to(torch.bfloat16)
        a = torch.rand(shp, generator=g, device=device) * -0.1
    elif gates == "sigmoid":
        q = (torch.randn(shp, generator=g, device=device) / 8).to(torch.bfloat16)
        k = (torch.randn(shp, generator=g, device=device) / 8).to(torch.bfloat16)
        v = (torch.randn(shp, generator=g, device=device) / 8).to(torch.bfloat16)
        x = torch.randn(shp, generator=g, device=device, dtype=torch.float64) * 0.5 + 2.0
        a = torch.nn.functional.logsigmoid(x).to(torch.float32)
    else:
        raise ValueError(gates)
    return q, k, v, a


def torch_fill_bf16_normal(t, seed: int):
    """Fill a uint8/bf16 device buffer with N(0,1) bf16 values (seeded)."""
    import torch
    g = torch.Generator(device=t.device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFF)
    view = t.view(torch.bfloat16)
    view.normal_(generator=g)
    return t


# ---------------------------------------------------------------------------
# workload shapes (sizes only; every number here is a configuration choice)
# ---------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class HybridShape:
    name: str
    n_lin: int            # linear-attention layers
    n_full: int           # full-attention layers
    n_heads: int          # linear heads
    d: int                # d_k = d_v
    n_kv_heads: int
    head_dim: int
    page: int             # tokens per KV page
    ckpt: int             # state checkpoint interval C
    gates: str
    batch: int = 1

    @property
    def page_bytes(self) -> int:
        # one page of one full-attention layer: [2 (K,V), page, n_kv, head_dim] bf16
        return 2 * self.page * self.n_kv_heads * self.head_dim * 2

    @property
    def state_bytes_per_layer(self) -> int:
        return self.batch * self.n_heads * self.d * self.d * 4


TINY = HybridShape("tiny-hybrid-2L", n_lin=1, n_full=1, n_heads=2, d=64, n_kv_heads=2,
                   head_dim=64, page=16, ckpt=64, gates="sigmoid")
SWEEP = HybridShape("sweep-1L-16h-d128", n_lin=1, n_full=0, n_heads=16, d=128, n_kv_heads=0,
                    head_dim=0, page=16, ckpt=512, gates="uniform")
HYBRID12 = HybridShape("hybrid-12L-9lin-3full", n_lin=9, n_full=3, n_heads=16, d=128,
                       n_kv_heads=4, head_dim=128, page=16, ckpt=256, gates="uniform")
KVSTRESS = HybridShape("kv-stress-48full", n_lin=0, n_full=48, n_heads=0, d=0, n_kv_heads=8,
                       head_dim=128, page=16, ckpt=256, gates="uniform")
LONG24 = HybridShape("long-24L-18lin-6full", n_lin=18, n_full=6, n_heads=32, d=128,
                     n_kv_heads=8, head_dim=128, page=32, ckpt=512, gates="uniform", batch=4)

SWEEP_LENGTHS = tuple(range(512, 4608 + 1, 512))      # nine prompt lengths
LONG_LENGTHS = (16384, 32768, 65536)
PARTIAL_HIT_SHORTFALL = 37                              # partial hit: hit = L - 37
DECODE_STEPS = 64


# ---------------------------------------------------------------------------
# seeded stress calls (the accuracy campaign of the prefill kernels)
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class StressCase:
    """One seeded random prefill call built to stress the kernels' numerics."""
    seed: int
    d: int
    pos0: list
    n_tokens: list
    ckpt_interval: int
    inputs: LinearInputs
    S0: np.ndarray


def _scaled_bf16(bits: np.ndarray, factor: float) -> np.ndarray:
    return f32_to_bf16_bits(bf16_bits_to_f32(bits) * np.float32(factor))


def gen_stress_case(seed: int) -> StressCase:
    """Random batch (1-4 problems of 1-3 heads, d = 64 or 128), resume points in [0, 700),
    tails of 0-1, 0-11 or 0-599 tokens, checkpoint interval 0/64/128/256/512, and up to
    four random token ranges of one stress kind each: growing gates (+0.02), gates of -30
    or -1.2, one zero gate (-1e4), v scaled by 2^17, or q and k scaled by 64; the starting
    state N(0, 0.25) scaled by 1, 100 or 2^16."""
    rng = np.random.default_rng(seed)
    d = int(rng.choice([64, 128, 128, 128]))
    B, nH = int(rng.integers(1, 5)), int(rng.integers(1, 4))
    C = int(rng.choice([0, 64, 128, 256, 512]))
    pos0 = [int(x) for x in rng.integers(0, 700, B)]
    mode = int(rng.integers(4))
    if mode == 0:
        n_tok = [int(x) for x in rng.integers(0, 2, B)]
    elif mode == 1:
        n_tok = [int(x) for x in rng.integers(0, 12, B)]
    else:
        n_tok = [int(x) for x in rng.integers(0, 600, B)]
    T = max(max(n_tok), 1)
    inp = gen_linear(seed + 1000, 0, B, T, nH, d, d)
    for _ in range(int(rng.integers(0, 5))):
        b, t0 = int(rng.integers(B)), int(rng.integers(T))
        ln = int(rng.integers(1, 70))
        kind = int(rng.integers(6))
        if kind == 0:
            inp.a[b, t0:t0 + ln] = 0.02
        elif kind == 1:
            inp.a[b, t0:t0 + ln] = -30.0
        elif kind == 2:
            inp.a[b, t0] = -1e4
        elif kind == 3:
            inp.v[b, t0:t0 + ln] = _scaled_bf16(inp.v[b, t0:t0 + ln], 2.0 ** 17)
        elif kind == 4:
            inp.q[b, t0:t0 + ln] = _scaled_bf16(inp.q[b, t0:t0 + ln], 64.0)
            inp.k[b, t0:t0 + ln] = _scaled_bf16(inp.k[b, t0:t0 + ln], 64.0)
        else:
            inp.a[b, t0:t0 + ln] = -1.2
    S0 = gen_state(seed + 1000, 0, B, nH, d, d) * float(rng.choice([1.0, 1.0, 100.0, 2.0 ** 16]))
    return StressCase(seed=seed, d=d, pos0=pos0, n_tokens=n_tok, ckpt_interval=C, inputs=inp,
                      S0=S0.astype(np.float32))
