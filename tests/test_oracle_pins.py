"""Pins for the float64 oracle: checks against what the paper and the
mathematics fix, never against the oracle's own formulas.

Alignment: the paper's Table 4 worked example, the Section 2.2 closed form
B = C*floor((N-1)/C) on complete hits, a set-based maximum on random caches,
and the Section 3.2 pre-repair behaviour as a negative fixture.
Bytes: the per-rank byte counts of Section 5.2 and the Table 5 H2D total.
Recurrence: identity-gate, zero-gate and scalar-gate closed forms, an
explicit-sum expansion with per-dimension gates, a chunked matrix
restatement, resume-from-checkpoint == full recomputation, and checkpoint
positions.
"""
import os

import numpy as np
import pytest

import oracle
from hs_inputs import bf16_bits_to_f32, f32_to_bf16_bits, gen_linear

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    out = []
    for line in open(os.path.join(GOLD, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            out.append([int(x) for x in line.split()])
    return out


# ---------------------------------------------------------------- alignment

def test_table4_after_repair():
    C = 1792
    for N, _, _, B_after, suffix in _rows("table4_alignment.txt"):
        avail = list(range(C, N + 1, C))          # every checkpoint of the prompt is cached
        c, n_pages, tail = oracle.align_prefix(N, N, avail, page_size=16)
        assert c == B_after, N
        assert tail == suffix, N
        assert n_pages == c // 16


def test_table4_before_repair_negative_fixture():
    C = 1792
    mism = []
    for N, B_before, p_before, B_after, _ in _rows("table4_alignment.txt"):
        B, p = oracle.align_prerepair(N, C)
        assert (B, p) == (B_before, p_before), N
        if B != p:
            mism.append(N)
        c, _, _ = oracle.align_prefix(N, N, list(range(C, N + 1, C)), 16)
        assert (c != B) == (N in (3584, 5376))
    assert mism == [3584, 5376]                    # the two failing exact-boundary cases


@pytest.mark.parametrize("C", [16, 32, 64])
def test_complete_hit_closed_form(C):
    # Section 2.2: on a complete hit with every checkpoint available, B = C*floor((N-1)/C)
    for N in range(1, 301):
        avail = list(range(C, N + 1, C))
        c, _, tail = oracle.align_prefix(N, N, avail, page_size=16)
        assert c == C * ((N - 1) // C)
        assert tail >= 1                           # never credits N on a complete hit
        assert c < N


def test_random_caches_set_maximum():
    rng = np.random.default_rng(1234)
    for _ in range(3000):
        N = int(rng.integers(1, 300))
        hit = int(rng.integers(0, N + 1))
        P = int(rng.choice([1, 4, 16]))
        cand = rng.integers(1, N + 40, size=int(rng.integers(0, 12)))
        avail = sorted(set(int(x) for x in cand))
        ok = {0} | {b for b in avail if b <= min(hit, N - 1) and b % P == 0}
        c, n_pages, tail = oracle.align_prefix(N, hit, avail, P)
        assert c == max(ok)
        assert n_pages * P == c and tail == N - c and tail >= 1


def test_align_rejects_invalid():
    for args in [(0, 0, [], 16), (10, 11, [], 16), (10, -1, [], 16), (10, 5, [], 0)]:
        with pytest.raises(ValueError):
            oracle.align_prefix(*args)


def test_tiny_config_worked_example():
    # tiny hybrid stack: N = 256, checkpoints every 64, complete hit -> c = 192, 12 pages of 16
    c, n_pages, tail = oracle.align_prefix(256, 256, [64, 128, 192, 256], 16)
    assert (c, n_pages, tail) == (192, 12, 64)


# ---------------------------------------------------------------- bytes

def test_restore_bytes_affine_and_table5_total():
    rows = _rows("restore_bytes.txt")
    pts = [r for r in rows if len(r) == 2]
    (total,) = [r[0] for r in rows if len(r) == 1]
    (b0, y0), (b1, y1), (b2, y2) = pts
    slope = (y1 - y0) // (b1 - b0)
    icpt = y0 - slope * b0
    assert slope * (b1 - b0) == y1 - y0
    assert icpt + slope * b2 == y2                 # the three printed points are affine in B
    # the oracle's byte count is affine in the page count with the state as intercept:
    # express the paper's fit as one "layer" of slope bytes per token and a fixed part
    def bytes_at(B):
        fixed = icpt
        return oracle.restore_bytes(1, B, slope, 0, 0, 0, 0) + fixed
    assert [bytes_at(b) for b in (b0, b1, b2)] == [y0, y1, y2]
    # Table 5: the nine repaired reloads of Table 4, four ranks
    C = 1792
    Bs = [oracle.align_prefix(N, N, list(range(C, N + 1, C)), 16)[0]
          for N, *_ in _rows("table4_alignment.txt")]
    assert 4 * sum(bytes_at(B) for B in Bs) == total


def test_restore_bytes_of_the_workloads_derived_by_hand():
    """Pages and float32 states of one resumed request, derived by hand from the workload
    shapes in tests/golden/restore_bytes_configs.txt (the derivation is in its header): the
    tiny stack's 12 pages of 8 KiB plus two 64 x 64 states, the hybrid and long-context
    stacks at their longest prompts, and a states-only restore."""
    rows = _rows("restore_bytes_configs.txt")
    assert len(rows) == 4
    for n_full, n_pages, page_bytes, n_lin, heads, dk, dv, total in rows:
        assert oracle.restore_bytes(n_full, n_pages, page_bytes, n_lin, heads, dk, dv) == total


# ---------------------------------------------------------------- recurrence

def _inputs(seed, n, nH, dk, dv, gates="uniform", batch=1):
    x = gen_linear(seed, 0, batch, n, nH, dk, dv, gates=gates)
    return x.q, x.k, x.v, x.a


def _f64(bits):
    return bf16_bits_to_f32(bits).astype(np.float64)


def test_identity_gate_is_causal_masked_attention():
    n, dk, dv = 37, 8, 6
    q, k, v, a = _inputs(1, n, 1, dk, dv)
    a[:] = 0.0
    S0 = np.random.default_rng(5).standard_normal((1, 1, dk, dv))
    o, S, _ = oracle.gla(q, k, v, a, [0], [n], S0=S0)
    Q, K, V = _f64(q[0, :, 0]), _f64(k[0, :, 0]), _f64(v[0, :, 0])
    M = np.tril(np.ones((n, n)))
    ref = (Q @ K.T * M) @ V + Q @ S0[0, 0]
    np.testing.assert_allclose(o[0, :, 0], ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(S[0, 0], S0[0, 0] + K.T @ V, rtol=1e-12, atol=1e-12)


def test_zero_gate_forgets_everything():
    n, dk, dv = 19, 8, 8
    q, k, v, a = _inputs(2, n, 1, dk, dv)
    a[:] = -1e4                                    # exp underflows to exactly 0
    S0 = np.ones((1, 1, dk, dv))
    o, S, _ = oracle.gla(q, k, v, a, [0], [n], S0=S0)
    Q, K, V = _f64(q[0, :, 0]), _f64(k[0, :, 0]), _f64(v[0, :, 0])
    for t in range(n):
        np.testing.assert_allclose(o[0, t, 0], (Q[t] @ K[t]) * V[t], rtol=1e-14, atol=1e-15)
    np.testing.assert_array_equal(S[0, 0], np.outer(K[-1], V[-1]))


def test_scalar_gate_closed_form():
    n, dk, dv, gam = 41, 6, 5, 0.9
    q, k, v, a = _inputs(3, n, 1, dk, dv)
    a[:] = np.float32(np.log(gam))
    gam = float(np.exp(np.float64(np.float32(np.log(gam)))))
    S0 = np.random.default_rng(7).standard_normal((1, 1, dk, dv))
    o, S, _ = oracle.gla(q, k, v, a, [0], [n], S0=S0)
    Q, K, V = _f64(q[0, :, 0]), _f64(k[0, :, 0]), _f64(v[0, :, 0])
    t = np.arange(n)
    D = np.where(t[:, None] >= t[None, :], gam ** (t[:, None] - t[None, :]), 0.0)
    ref = (Q @ K.T * D) @ V + (gam ** (t + 1))[:, None] * (Q @ S0[0, 0])
    np.testing.assert_allclose(o[0, :, 0], ref, rtol=1e-11, atol=1e-12)


def test_per_dim_gates_explicit_sum():
    # S_t = diag(prod_{s<=t} g_s) S0 + sum_{j<=t} diag(prod_{j<s<=t} g_s) k_j v_j^T
    n, dk, dv = 12, 5, 4
    q, k, v, a = _inputs(4, n, 1, dk, dv, gates="sigmoid")
    S0 = np.random.default_rng(8).standard_normal((1, 1, dk, dv))
    o, S, _ = oracle.gla(q, k, v, a, [0], [n], S0=S0)
    Q, K, V = _f64(q[0, :, 0]), _f64(k[0, :, 0]), _f64(v[0, :, 0])
    g = np.exp(a[0, :, 0].astype(np.float64))
    for t in range(n):
        St = np.prod(g[:t + 1], axis=0)[:, None] * S0[0, 0]
        for j in range(t + 1):
            St = St + np.prod(g[j + 1:t + 1], axis=0)[:, None] * np.outer(K[j], V[j])
        np.testing.assert_allclose(o[0, t, 0], Q[t] @ St, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(S[0, 0], St, rtol=1e-12, atol=1e-13)


def _chunked_np(Q, K, V, A_, S0, chunk):
    """Chunked matrix form of the recurrence (second restatement, float64):
    within a chunk with cumulative log-decay G_i = sum_{s<=i} a_s,
      o_i = (q_i * exp(G_i)) S0 + sum_{j<=i} (sum_d q_id k_jd exp(G_id - G_jd)) v_j
      S'  = diag(exp(G_last)) S0 + sum_j (k_j * exp(G_last - G_j)) v_j^T"""
    n = Q.shape[0]
    S = np.array(S0)
    out = np.zeros((n, V.shape[1]))
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        q, k, v, a = Q[s:e], K[s:e], V[s:e], A_[s:e]
        G = np.cumsum(a, axis=0)
        Am = np.zeros((e - s, e - s))
        for i in range(e - s):
            for j in range(i + 1):
                Am[i, j] = np.sum(q[i] * k[j] * np.exp(G[i] - G[j]))
        out[s:e] = (q * np.exp(G)) @ S + Am @ v
        S = np.exp(G[-1])[:, None] * S + (k * np.exp(G[-1] - G)).T @ v
    return out, S


@pytest.mark.parametrize("chunk", [4, 16])
def test_chunked_restatement(chunk):
    n, dk, dv = 45, 8, 8
    q, k, v, a = _inputs(5, n, 1, dk, dv, gates="sigmoid")
    S0 = np.random.default_rng(9).standard_normal((1, 1, dk, dv))
    o, S, _ = oracle.gla(q, k, v, a, [0], [n], S0=S0)
    ref_o, ref_S = _chunked_np(_f64(q[0, :, 0]), _f64(k[0, :, 0]), _f64(v[0, :, 0]),
                               a[0, :, 0].astype(np.float64), S0[0, 0], chunk)
    np.testing.assert_allclose(o[0, :, 0], ref_o, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(S[0, 0], ref_S, rtol=1e-11, atol=1e-12)


def test_resume_from_checkpoint_equals_recompute_bitwise():
    N, C, nH, d = 256, 64, 2, 16
    q, k, v, a = _inputs(6, N, nH, d, d, gates="sigmoid")
    o_full, S_full, ck = oracle.gla(q, k, v, a, [0], [N], C_=C)
    assert ck[0].shape[0] == N // C
    for m, c in enumerate(range(C, N, C)):
        S_c = ck[0][m][None]
        o_r, S_r, ck_r = oracle.gla(q[:, c:], k[:, c:], v[:, c:], a[:, c:], [c], [N - c],
                                    S0=S_c, C_=C)
        np.testing.assert_array_equal(o_r[0], o_full[0, c:])
        np.testing.assert_array_equal(S_r, S_full)
        np.testing.assert_array_equal(ck_r[0], ck[0][m + 1:])


def test_checkpoints_are_prefix_states():
    N, C, d = 200, 48, 8
    q, k, v, a = _inputs(7, N, 1, d, d)
    _, _, ck = oracle.gla(q, k, v, a, [0], [N], C_=C)
    assert ck[0].shape[0] == N // C
    for m in range(N // C):
        b = (m + 1) * C
        _, S_b, _ = oracle.gla(q[:, :b], k[:, :b], v[:, :b], a[:, :b], [0], [b])
        np.testing.assert_array_equal(ck[0][m], S_b[0])
    # a run that starts mid-interval emits only the boundaries it crosses
    _, _, ck2 = oracle.gla(q[:, 30:], k[:, 30:], v[:, 30:], a[:, 30:], [30], [N - 30],
                           S0=None, C_=C)
    assert ck2[0].shape[0] == N // C - 30 // C


def test_batch_and_heads_are_independent():
    B, n, nH, d = 2, 23, 3, 8
    q, k, v, a = _inputs(8, n, nH, d, d, batch=B)
    o, S, _ = oracle.gla(q, k, v, a, [0, 5], [n, n - 4])
    for b, n_b in ((0, n), (1, n - 4)):
        for h in range(nH):
            o1, S1, _ = oracle.gla(q[b:b + 1, :, h:h + 1].copy(), k[b:b + 1, :, h:h + 1].copy(),
                                   v[b:b + 1, :, h:h + 1].copy(), a[b:b + 1, :, h:h + 1].copy(),
                                   [0], [n_b])
            np.testing.assert_array_equal(o1[0, :, 0], o[b, :, h])
            np.testing.assert_array_equal(S1[0, 0], S[b, h])
    assert not o[1, n - 4:].any()                  # tokens past n_tokens are untouched


def test_empty_tail_is_identity():
    q, k, v, a = _inputs(9, 4, 1, 8, 8)
    S0 = np.random.default_rng(3).standard_normal((1, 1, 8, 8))
    o, S, ck = oracle.gla(q, k, v, a, [64], [0], S0=S0, C_=64)
    np.testing.assert_array_equal(S, S0)
    assert not o.any() and ck[0].shape[0] == 0


# ---------------------------------------------------------------- copies

def test_scatter_pages_and_untouched_bytes():
    rng = np.random.default_rng(11)
    P, n_pages, nb, L = 64, 5, 12, 2
    staging = [rng.integers(1, 255, size=n_pages * P, dtype=np.uint8) for _ in range(L)]
    cache = [np.full(nb * P, 0xFF, np.uint8) for _ in range(L)]
    bt = np.array([7, 2, 11, 0, 5], np.int32)
    oracle.scatter_pages(staging, cache, bt, n_pages, P)
    for l in range(L):
        for j, b in enumerate(bt):
            assert bytes(cache[l][b * P:(b + 1) * P]) == bytes(staging[l][j * P:(j + 1) * P])
        untouched = sorted(set(range(nb)) - set(bt.tolist()))
        for b in untouched:
            assert (cache[l][b * P:(b + 1) * P] == 0xFF).all()


def test_gather_pages_reads_each_block_and_inverts_the_scatter():
    """The save path (Section 3.1): page j of the staging pool is cache block bt[j].
    Cache bytes encode (layer, block, offset), so a page landing from the wrong block
    or layer, or shifted, is caught; scatter after gather restores the cache blocks."""
    P, nb, L = 48, 10, 3
    cache = [np.array([(l * 37 + b * 5 + (i % 7)) % 251 for b in range(nb) for i in range(P)],
                      np.uint8) for l in range(L)]
    bt = np.array([9, 0, 4, 6], np.int32)
    staging = [np.zeros(len(bt) * P, np.uint8) for _ in range(L)]
    oracle.gather_pages(cache, staging, bt, len(bt), P)
    for l in range(L):
        for j, b in enumerate(bt):
            want = np.array([(l * 37 + int(b) * 5 + (i % 7)) % 251 for i in range(P)], np.uint8)
            assert np.array_equal(staging[l][j * P:(j + 1) * P], want)
    back = [np.full(nb * P, 0xFF, np.uint8) for _ in range(L)]
    oracle.scatter_pages(staging, back, bt, len(bt), P)
    for l in range(L):
        for b in bt:
            assert np.array_equal(back[l][b * P:(b + 1) * P], cache[l][b * P:(b + 1) * P])


def test_rank_slices_reassemble_the_full_page_transfer():
    """Four tensor-parallel ranks each move their bytes of every page row (Table 1: TP=4,
    FP8 pages; Section 5.2: per-rank transfers).  Restoring every rank's slice equals the
    full-page scatter; each rank's gathered slice is its columns of the full-page gather;
    each rank moves a quarter of the bytes."""
    rng = np.random.default_rng(13)
    tokens, heads, hd, TP, L, nb = 4, 8, 16, 4, 2, 7
    rows, row_bytes = 2 * tokens, heads * hd              # FP8: one byte per element
    P = rows * row_bytes
    cb = row_bytes // TP
    bt = np.array([5, 1, 3], np.int32)
    full = [rng.integers(0, 256, size=len(bt) * P, dtype=np.uint8) for _ in range(L)]
    want = [np.full(nb * P, 0xAB, np.uint8) for _ in range(L)]
    oracle.scatter_pages(full, want, bt, len(bt), P)
    got = [np.full(nb * P, 0xAB, np.uint8) for _ in range(L)]
    for r in range(TP):
        # rank r's staging: its bytes of every row, rows back to back
        st = [f.reshape(len(bt), rows, row_bytes)[:, :, r * cb:(r + 1) * cb].copy().reshape(-1)
              for f in full]
        assert sum(x.size for x in st) * TP == sum(x.size for x in full)
        oracle.scatter_slices(st, got, bt, len(bt), P, rows, r * cb, cb)
        back = [np.zeros_like(x) for x in st]
        oracle.gather_slices(want, back, bt, len(bt), P, rows, r * cb, cb)
        for a, b in zip(back, st):
            assert np.array_equal(a, b)
    for a, b in zip(got, want):
        assert np.array_equal(a, b)


# float32 bit patterns a state restore must carry through unchanged: quiet and signalling
# NaNs with payloads, both zeros, both infinities, the smallest and largest subnormals, the
# largest normal, and ordinary values
SPECIAL_F32 = np.array([0x7FC00000, 0xFFC12345, 0x7FA00001, 0xFF800001, 0x00000000, 0x80000000,
                        0x7F800000, 0xFF800000, 0x00000001, 0x807FFFFF, 0x7F7FFFFF, 0x3F800000,
                        0xC0490FDB, 0x00800000], np.uint32)


def _slot_bits(n, floats_each, tag):
    """n source slots whose words differ by slot and by position: the special patterns
    first, then words that encode (tag, slot, index)."""
    out = []
    for i in range(n):
        w = np.array([(tag << 24) ^ (i << 16) ^ x ^ 0x3C000000 for x in range(floats_each)],
                     np.uint32)
        m = min(len(SPECIAL_F32), floats_each)
        w[:m] = np.roll(SPECIAL_F32, i)[:m]
        out.append(w)
    return out


def test_copy_slots_bitwise_with_special_values():
    """The state restore and the checkpoint writer (Section 1: a recurrent state updated in
    place is restored, not recomputed; Section 2.2: the state at B) are copies of float32
    slots: every bit pattern arrives unchanged in the slot of the same index, and the
    destination past floats_each keeps its poison."""
    n, fe, guard = 5, 37, 11
    src_bits = _slot_bits(n, fe, 1)
    src = [b.view(np.float32) for b in src_bits]
    dst = [np.full(fe + guard, 0xDEADBEEF, np.uint32).view(np.float32) for _ in range(n)]
    oracle.copy_slots(src, dst, fe)
    for i in range(n):
        got = dst[i].view(np.uint32)
        assert np.array_equal(got[:fe], src_bits[i]), i
        assert (got[fe:] == 0xDEADBEEF).all(), i
    # the slots are distinct, so a copy from the wrong slot cannot pass the check above
    assert len({b.tobytes() for b in src_bits}) == n


def test_copy_slots_of_zero_slots_or_zero_floats_touch_nothing():
    src = [b.view(np.float32) for b in _slot_bits(3, 8, 2)]
    dst = [np.full(8, 0xDEADBEEF, np.uint32).view(np.float32) for _ in range(3)]
    oracle.copy_slots(src, dst, 0)
    oracle.copy_slots(src[:0], dst[:0], 8)
    for d in dst:
        assert (d.view(np.uint32) == 0xDEADBEEF).all()


def test_bf16_rounding_is_round_to_nearest_even():
    # 1 + 2^-8 is halfway between bf16 neighbours 1 and 1 + 2^-7: ties go to even (1.0)
    x = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -2.5, 0.0], np.float32)
    b = f32_to_bf16_bits(x)
    np.testing.assert_array_equal(bf16_bits_to_f32(b),
                                  np.array([1.0, 1.0 + 2.0 ** -6, -2.5, 0.0], np.float32))
