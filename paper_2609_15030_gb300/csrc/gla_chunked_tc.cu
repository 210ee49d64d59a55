// Chunked gated linear attention on tcgen05 tensor cores (sm_103a).
//
// Recurrence (per head):  S_t = diag(g_t) S_{t-1} + k_t v_t^T,  o_t = q_t S_t,
// g_t = exp(a_t).  The paper runs its linear layers on FLA kernels without
// printing their recurrence; this is the form the library implements, in
// the chunked matrix form.  For a segment of L <= 64 tokens inside one
// 64-token chunk of the absolute position grid, with cumulative log2-decay
// Lam_i = log2(e) * sum_{s<=i} a_s (per key dimension):
//
//   Q~_i = q_i * 2^{Lam_i}            K~_j = k_j * 2^{-Lam_j}
//   A_ij = [j <= i] * Q~_i . K~_j     (= sum_d q_id k_jd 2^{Lam_id - Lam_jd})
//   o_i  = Q~_i S + sum_j A_ij v_j
//   S'   = diag(2^{Lam_last}) (S + K~^T V)
//
// One CTA owns one (problem, head) and walks its segments in order; the
// float32 state lives in tensor memory (TMEM) for the whole call, stored
// transposed (lane = value dim e, column = key dim d).  (The RESTART
// instantiation, the output pass of the segment-parallel prefill, instead
// starts every segment from its own start state; see the kernel.)
//
// Fast chunks run kind::f16 MMA groups with fp16 operands and float32
// accumulators:  D_O = S^T Q~^T (A operand: an fp16 copy of S^T in TMEM),
// D_A = Q~ K~^T, then per 16 tokens D_O += V^T A^T (N = 64) and S^T += V^T K~
// (N = D, the K~ tile read MN-major), V^T in TMEM.  fp16 keeps the 10-bit
// mantissa of tf32 but halves the instructions (K = 16 per MMA).  The CTA's
// 16 warps form two groups in a pipeline over two alternating operand sets:
// while the eight state warps finish chunk c (the state pass, which applies
// the pending decay 2^{Lam_last}, writes a due checkpoint and refreshes the
// fp16 copy of S^T; the causal mask with each token's own score summed in
// float32 on the diagonal; the output epilogue) the eight builder warps stage
// chunk c+1 and build its operands (cumulative decay scan, Q~, K~, V^T).  The
// first builder thread issues the TMA copies and D_A, the first state thread
// the other MMAs.
//
// A chunk is fast only if every fp16 operand provably stays below 2^15 in
// magnitude (|q|, |v|, |K~|, the bound 128 max|q| max|k| on |A|, and a bound
// on |S| carried from the measured state) and its total decay factor
// 2^{Lam_last} stays >= 2^-10 in every key dim (so Q~ never nears fp16's
// subnormals).  Any other chunk (strong decay, huge values) runs the exact
// path: tf32 operands (the state split into two exact tf32 parts), the
// intra-chunk matrix computed elementwise in float32 with 2^{Lam_i - Lam_j} <= 1,
// and the state updated as
// diag(2^{Lam_last}) S + K^^T V with K^_j = k_j 2^{Lam_last - Lam_j}.  The
// choice depends only on the chunk's inputs and on the state it starts from,
// as does every operation order, so a resumed run reproduces a full
// recomputation bit for bit when it starts on the chunk grid.  Segments of at
// most 8 tokens run the per-token recurrence with the recurrent kernel's exact
// operation order.
//
// Every wait on an mbarrier is bounded (1 s) and is followed by a barrier that
// reduces the abort flag, so every thread of a group takes the same branch; on
// timeout the CTA reports HS_DEVERR_TIMEOUT, waits (bounded) for its own copies
// and MMAs in flight, frees its TMEM and returns.
#include "gla_chunk_common.cuh"

namespace hs {
namespace {

using namespace ptx;
using namespace gck;

// RESTART: the output pass of the segment-parallel prefill.  Every segment of a problem
// starts from its own start state (segment k of problem b from state slot ck_base[b] + k of
// p.state) instead of the state the previous segment leaves, and decides its path on that
// state as the first segment of a run does, so that a segment's outputs do not depend on
// which other segments share its CTA; no state or checkpoint is written.
template <int D, bool RESTART>
__global__ void __launch_bounds__(NT, 1)
gla_chunked_tc_kernel(const __grid_constant__ GlaParams p, const __grid_constant__ TmaMaps maps)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sb = smem_u32(smem);
    float *sRed = reinterpret_cast<float *>(smem + OFF_RED);
    // [0] TMEM base, [1] abort flag, [2] decision on the latest built segment (1 = fast),
    // [3] run result (1 = the segment at [4..5] needs the exact path), [4..5] position
    // where the run stopped, [6..7] its local token index
    volatile uint32_t *sMisc = reinterpret_cast<volatile uint32_t *>(smem + OFF_MISC);
    volatile int64_t *sRun = reinterpret_cast<volatile int64_t *>(smem + OFF_MISC + 16);
    const uint32_t bar_tma = sb + OFF_BAR, bar_a = sb + OFF_BAR + 8, bar_o = sb + OFF_BAR + 16,
                   bar_s = sb + OFF_BAR + 24, bar_built = sb + OFF_BAR + 32,
                   bar_go = sb + OFF_BAR + 40, bar_ld = sb + OFF_BAR + 48,
                   bar_a1 = sb + OFF_BAR + 56;

    const int tid = threadIdx.x, warp = tid >> 5;
    const int b = blockIdx.x / p.n_heads;
    const int h = blockIdx.x - b * p.n_heads;
    const int n = p.n_tokens[b];
    if (n <= 0)
        return;
    const int64_t pos0 = p.pos0[b];
    const int64_t end = pos0 + n;
    const int64_t tstride = (int64_t)p.n_heads * D;   // elements between consecutive tokens
    const int C = p.ckpt_interval;

    if (tid == 0) {
        mbar_init(bar_tma, 1);
        mbar_init(bar_a, 1);
        mbar_init(bar_o, 1);
        mbar_init(bar_s, 1);
        mbar_init(bar_built, 1);
        mbar_init(bar_go, 1);
        mbar_init(bar_ld, 1);
        mbar_init(bar_a1, 1);
        fence_mbar_init();
        sMisc[1] = 0;   // abort flag
    }
    if (warp == 0)
        tmem_alloc(sb + OFF_MISC, TMEM_COLS);
    if (tid == kLoader) {
        // the first segment's inputs into L2 while the previous kernel finishes: a
        // prefetch moves no data into this SM, and L2 holds the only copy any later write
        // updates, so it is safe even if that kernel writes those inputs
        const int32_t y = (int32_t)p.row0[b];
        tma_prefetch_2d(&maps.q, h * D, y);
        tma_prefetch_2d(&maps.k, h * D, y);
        tma_prefetch_2d(&maps.v, h * D, y);
        tma_prefetch_2d(&maps.g, h * D, y);
    }
    pdl_wait();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sMisc[0];
    const bool builder = warp < 8;
    const bool worker = !builder;                              // a state warp

    // bookkeeping of the loader (copies issued, one still in flight) and of the issuer,
    // for the waits and the abort path; every mbarrier is waited on by one thread only
    uint32_t n_tma = 0;
    bool tma_pending = false;
    uint32_t ph_tma = 0, ph_o = 0, ph_s = 0, ph_built = 0, ph_go = 0;
    uint32_t ph_a0 = 0, ph_a1 = 0;   // D_A products of even / odd segments (bar_a, bar_a1)
    bool aborted = false;

    // L2 prefetch of the 64 tokens from local position t (if any are this problem's)
    auto prefetch = [&](int64_t t) {
        if (t >= n)
            return;
        const int32_t y = (int32_t)((int64_t)p.row0[b] + t);
        const int32_t x = h * D;
        tma_prefetch_2d(&maps.q, x, y);
        tma_prefetch_2d(&maps.k, x, y);
        tma_prefetch_2d(&maps.v, x, y);
        tma_prefetch_2d(&maps.g, x, y);
    };
    // (loader) staged inputs of the segment at local position tok_local; segments after
    // the first start on the 64-token grid, so the segment kPrefetch ahead starts at
    // tok_local + 64 * kPrefetch and is requested into L2 now
    auto issue_tma = [&](int64_t tok_local) {
        const int32_t y = (int32_t)((int64_t)p.row0[b] + tok_local);
        const int32_t x = h * D;
        mbar_arrive_expect_tx(bar_tma, Geo<D>::STAGE);
        tma_load_2d(sb + OFF_SQ, &maps.q, x, y, bar_tma);
        tma_load_2d(sb + OFF_SK, &maps.k, x, y, bar_tma);
        tma_load_2d(sb + OFF_SV, &maps.v, x, y, bar_tma);
        tma_load_2d(sb + OFF_SG, &maps.g, x, y, bar_tma);
        ++n_tma;
        tma_pending = true;
        if (tok_local > 0)
            prefetch(tok_local + (int64_t)CH * kPrefetch);
    };
    // one thread (`who`) waits on an mbarrier; false (for every thread) if that wait ran
    // out or another thread raised the abort flag.  CTA-wide, or within the builder (id 1)
    // or state (id 2) warps; the barrier's OR reduction makes the answer uniform.
    auto wait_all = [&](int who, uint32_t bar, uint32_t &ph) -> bool {
        bool bad = false;
        if (tid == who)
            bad = !mbar_wait_bounded(bar, ph, kTimeoutNs);
        if (bad)
            sMisc[1] = 1;
        ph ^= 1;
        const bool stop = __syncthreads_or(bad || sMisc[1] != 0) != 0;
        tc_fence_after();
        if (stop)
            aborted = true;
        return !stop;
    };
    auto wait_tma = [&]() -> bool {
        tma_pending = false;
        return wait_all(kLoader, bar_tma, ph_tma);
    };
    auto wait_group = [&](int id, int who, uint32_t bar, uint32_t &ph) -> bool {
        bool bad = false;
        if (tid == who)
            bad = !mbar_wait_bounded(bar, ph, kTimeoutNs);
        if (bad)
            sMisc[1] = 1;
        ph ^= 1;
        const bool stop = bar_or(id, bad || sMisc[1] != 0);
        tc_fence_after();
        if (stop)
            aborted = true;
        return !stop;
    };
    // a group barrier that also reports the abort flag, uniformly
    auto sync_group = [&](int id) -> bool {
        const bool stop = bar_or(id, sMisc[1] != 0);
        if (stop)
            aborted = true;
        return !stop;
    };
    auto sync_all = [&]() -> bool {
        const bool stop = __syncthreads_or(sMisc[1] != 0) != 0;
        if (stop)
            aborted = true;
        return !stop;
    };
    auto seg_len = [&](int64_t at) -> int { return (int)(min(end, (at / CH + 1) * CH) - at); };
    auto is_long = [&](int64_t at) -> bool { return at < end && seg_len(at) > kShort; };
    auto ckpt_slot = [&](int64_t seg_end) -> float * {
        if (!(C > 0 && seg_end % C == 0 && p.ckpt_slots != nullptr))
            return nullptr;
        float *slot = p.ckpt_slots[p.ck_base[b] + (seg_end / C - pos0 / C - 1)];
        if (slot == nullptr || (reinterpret_cast<uintptr_t>(slot) & 15u) != 0) {
            if (tid == kIssuer)
                report(p.d_err, slot == nullptr ? HS_DEVERR_NULL : HS_DEVERR_MISALIGNED);
            return nullptr;
        }
        return slot + (int64_t)h * D * D;
    };
    // largest |S| recorded by the last state pass (valid after the barrier that follows it)
    auto state_max = [&]() -> float {
        float m = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w)
            m = fmaxf(m, sRed[w * 8 + 4]);
        return m;
    };

    if (tid == kLoader)
        issue_tma(0);
    bool prefetched = false;   // (loader) the segments after the first requested into L2

    // incoming state -> TMEM (state warps), transposed: S^T[e][d] = state[d][e]; its
    // largest magnitude.  The builders meanwhile stage and build the first segment.
    float *st_g = p.state + ((int64_t)(RESTART ? p.ck_base[b] : b) * p.n_heads + h) * D * D;
    if (worker) {
        state_load<D>(smem, tmem, st_g);
        tc_fence_before();
        bar_staters();
        tc_fence_after();
    }

    // the output rows from local token t
    auto outp = [&](int64_t t) { return p.o + (((int64_t)p.row0[b] + t) * p.n_heads + h) * D; };

    // ---- a short segment (<= kShort tokens, staged inputs already waited for, no decay
    // pending): the per-token recurrence with the recurrent kernel's exact operation order
    // (fma chains over groups of 16 key rows, group partials summed left to right)
    auto short_segment = [&](int64_t tok_s, int L, int64_t seg_end) {
        short_state<D>(smem, tmem, L, ckpt_slot(seg_end));
        if (tid == kLoader && seg_end < end)
            issue_tma(tok_s + L);
        short_outputs<D>(smem, L, outp(tok_s), tstride);
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    };

    // the guard of a built fast segment (state warps, after the wait for the builders): log-gates
    // <= 0, and every fp16 operand (Q~, K~, V, A, the fp16 copy of the state it starts from)
    // below 2^15 in magnitude.  Returns whether the segment's own inputs pass; `state_ok` says
    // whether the state (its measured magnitude, or a bound on it) passes too.
    float mk_new = 0.f, mv_new = 0.f;
    auto guard = [&](float s_mag, bool &state_ok) -> bool {
        float mq = 0.f, mk = 0.f, mv = 0.f;
        bool ok = true;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            mq = fmaxf(mq, sRed[w * 8 + 0]);
            ok = ok && sRed[w * 8 + 1] != 0.f;
            mk = fmaxf(mk, sRed[w * 8 + 2]);
            mv = fmaxf(mv, sRed[w * 8 + 3]);
        }
        mk_new = mk;
        mv_new = mv;
        state_ok = s_mag < kF16Lim;
        return ok && (float)D * mq * mk < kF16Lim;
    };

    // ---- one exact segment, from staged inputs, no decay pending and no MMA in flight;
    // leaves the final state in TMEM, writes its outputs and checkpoint
    auto exact_segment = [&](int64_t tok_s, int L, int par, int gslot, int64_t seg_end) -> bool {
        exact_build<D>(smem, tmem, L, gslot);
        exact_split_state<D>(tmem);
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == kIssuer) {
            tc_fence_after();
            exact_issue_sq<D>(tmem, sb);
        }
        exact_scores<D>(smem, L);
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == kIssuer) {
            tc_fence_after();
            exact_issue_av<D>(tmem, sb);
            tc_commit(bar_o);
        }
        if (!wait_all(kIssuer, bar_o, ph_o))
            return false;
        state_pass<D>(smem, tmem, gslot, nullptr, false);          // S <- diag(2^{Lam_last}) S
        tc_fence_before();
        __syncthreads();
        if (tid == kIssuer) {
            tc_fence_after();
            exact_issue_state<D>(tmem, sb);
            tc_commit(bar_s);
        }
        if (!wait_all(kIssuer, bar_s, ph_s))
            return false;
        state_pass<D>(smem, tmem, -1, ckpt_slot(seg_end), false);   // checkpoint and |S| of the final state
        out_epilogue<D>(tmem, outp(tok_s), tstride, L, par, false);
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        return true;
    };

    // ---- a run of long segments on the fast path, the two groups of warps in a pipeline:
    // the builders stage and build segment k+1 while the state warps finish segment k.
    // Handoffs (each mbarrier has one waiting thread and one arriving party):
    //   bar_built: builders -> state warps, segment k built (operands, V^T, guard maxima)
    //   bar_go:    state warps -> builders, the decision on segment k is made (sMisc[2]);
    //              when it is fast, it also means the operand set of segment k+1 is free
    //              (the products of segment k-1 are complete)
    // A run ends after the last long segment, before a segment whose own inputs the guard
    // sends to the exact path, or before a segment whose state bound fails: a decision inside a
    // run only has a bound on the state it starts from (that state is still being computed), so
    // such a segment starts a new run, whose first decision reads the measured state exactly as
    // a run resumed from a checkpoint at that segment does.  The groups then meet CTA-wide.
    // No MMA is in flight at either end.
    int kseq = 0;   // long segments of the current run so far (slot of 2^{Lam_last}: kseq mod 4)
    auto builder_run = [&](int64_t rpos, int64_t rtok) {
        int par = 0;
        while (true) {
            const int L = seg_len(rpos);
            if (!wait_group(1, kLoader, bar_tma, ph_tma))
                return;
            tma_pending = false;
            if (tid == kLoader && !prefetched) {
                // once the first segment has landed (the state and the first segment are
                // not queued behind these): the next kPrefetch segments into L2
                prefetched = true;
                for (int j = 1; j <= kPrefetch; ++j)
                    prefetch(rtok + L + (int64_t)CH * (j - 1));
            }
            build_fast<D>(smem, tmem, L, par, kseq & 3);
            fence_proxy_async_smem();
            tc_fence_before();
            if (!sync_group(1))
                return;
            const bool next_long = is_long(rpos + L);
            if (tid == kLoader) {
                mbar_arrive(bar_built);
                // the staged rows are consumed: stage the next segment (long or short) now;
                // an exact decision on this one reloads it
                if (rpos + L < end)
                    issue_tma(rtok + L);
                // D_A = Q~ K~^T of this segment, into its own buffer (the state warps wait on
                // bar_a / bar_a1 by parity before they read it)
                tc_fence_after();
                fast_issue_scores<D>(tmem, sb, par);
                tc_commit(par ? bar_a1 : bar_a);
            }
            if (!wait_group(1, kLoader, bar_go, ph_go))
                return;
            if (sMisc[2] == 0 || !next_long)
                return;
            rpos += L;
            rtok += L;
            par ^= 1;
            ++kseq;
        }
    };
    auto state_run = [&](int64_t rpos, int64_t rtok) {
        int par = 0;
        bool pend = false;
        uint32_t stop = 0;   // why the run ended: 0 done or short segment, 1 exact, 2 new run
        int pend_par = 0, pend_L = 0, pend_g = 0;
        int64_t pend_tok = 0, pend_end = 0;
        float mk_cur = 0.f, mv_cur = 0.f;
        if (!wait_group(2, kIssuer, bar_built, ph_built))
            return;
        // first segment of a run: the measured state (float32 maximum of the last state pass
        // or of the loaded state)
        bool state_ok;
        bool fast = guard(state_max(), state_ok) && state_ok;
        if (tid == kIssuer) {
            sMisc[2] = fast ? 1u : 0u;
            if (!fast)
                mbar_arrive(bar_go);
        }
        stop = fast ? 0u : 1u;
        // a segment sent to the exact path: its (unused) D_A product is drained first
        if (!fast && !wait_group(2, kIssuer, bar_a, ph_a0))
            return;
        while (fast) {
            const int L = seg_len(rpos);
            const int64_t seg_end = rpos + L;
            mk_cur = mk_new;
            mv_cur = mv_new;
            if (pend && !wait_group(2, kIssuer, bar_o, ph_o))
                return;
            // the products of the previous segment are complete: its operand set is free
            if (tid == kIssuer)
                mbar_arrive(bar_go);
            state_pass<D>(smem, tmem, pend ? pend_g : -1, pend ? ckpt_slot(pend_end) : nullptr, true);
            tc_fence_before();
            if (!sync_group(2))
                return;
            if (tid == kIssuer) {
                // D_O = S^T Q~^T (the N = 192 product below accumulates onto it in order)
                tc_fence_after();
                fast_issue_sq<D>(tmem, sb, par);
            }
            if (pend)
                out_epilogue<D>(tmem, outp(pend_tok), tstride, pend_L, pend_par, true);
            // D_A of this segment (issued by the builders' loader)
            if (!(par ? wait_group(2, kIssuer, bar_a1, ph_a1) : wait_group(2, kIssuer, bar_a, ph_a0)))
                return;
            a_build<D>(smem, tmem, par);
            fence_proxy_async_smem();
            tc_fence_before();
            if (!sync_group(2))
                return;
            if (tid == kIssuer) {
                tc_fence_after();
                fast_issue_update<D>(tmem, sb, par);
                tc_commit(bar_o);
            }
            pend = true;
            pend_par = par;
            pend_tok = rtok;
            pend_L = L;
            pend_end = seg_end;
            pend_g = kseq & 3;
            rpos = seg_end;
            rtok += L;
            par ^= 1;
            ++kseq;
            if (!is_long(rpos))
                break;
            // the builders' next segment, and the decision on it: the state it starts from is
            // bounded by the fp16 copy's largest |S| at this segment's start plus this segment's
            // largest update, 64 max|k| max|v| (the decay factors are <= 1)
            if (!wait_group(2, kIssuer, bar_built, ph_built))
                return;
            const bool inputs_ok =
                guard((state_max() + 64.0f * mk_cur * mv_cur) * kBoundMargin, state_ok);
            fast = inputs_ok && state_ok;
            if (tid == kIssuer) {
                sMisc[2] = fast ? 1u : 0u;
                if (!fast)
                    mbar_arrive(bar_go);
            }
            stop = fast ? 0u : (inputs_ok ? 2u : 1u);
            if (!fast && !(par ? wait_group(2, kIssuer, bar_a1, ph_a1) : wait_group(2, kIssuer, bar_a, ph_a0)))
                return;
        }
        if (pend) {
            if (!wait_group(2, kIssuer, bar_o, ph_o))
                return;
            state_pass<D>(smem, tmem, pend_g, ckpt_slot(pend_end), false);
            out_epilogue<D>(tmem, outp(pend_tok), tstride, pend_L, pend_par, false);
            tc_fence_before();
            if (!sync_group(2))
                return;
        }
        if (tid == kIssuer) {
            sMisc[3] = stop;
            sRun[0] = rpos;
            sRun[1] = rtok;
        }
    };

    // RESTART: the state warps' side of a run in which every segment decides on, and is
    // computed from, its own start state, loaded before its decision (the first segment's is
    // loaded before the run); the builders' side is builder_run, unchanged.  No product reads
    // the float32 state in TMEM here (the state update is skipped and D_O reads the fp16 copy),
    // so the next segment's state is loaded while the previous segment's products run.
    int loaded = 0;   // index of the segment whose start state is in TMEM (state warps)
    auto seg_idx = [&](int64_t at) -> int { return (int)(at / CH - pos0 / CH); };
    // (issuing thread) the start state of the segment at `at` into L2, one bulk request
    auto prefetch_state = [&](int64_t at) {
        const float *src = st_g + (int64_t)seg_idx(at) * p.n_heads * D * D;
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src),
                     "r"((uint32_t)(D * D * 4))
                     : "memory");
    };
    auto state_run_restart = [&](int64_t rpos, int64_t rtok) {
        int par = 0;
        bool pend = false;
        uint32_t stop = 0;   // 0 done or short segment, 1 exact
        int pend_par = 0, pend_L = 0;
        int64_t pend_tok = 0;
        while (true) {
            const int L = seg_len(rpos);
            if (!wait_group(2, kIssuer, bar_built, ph_built))
                return;
            if (loaded != seg_idx(rpos)) {
                state_load<D>(smem, tmem, st_g + (int64_t)seg_idx(rpos) * p.n_heads * D * D);
                loaded = seg_idx(rpos);
            }
            // the loaded state (its TMEM columns and its largest |S|) visible to the group
            tc_fence_before();
            if (!sync_group(2))
                return;
            tc_fence_after();
            bool state_ok;
            const bool fast = guard(state_max(), state_ok) && state_ok;
            if (tid == kIssuer) {
                sMisc[2] = fast ? 1u : 0u;
                if (!fast)
                    mbar_arrive(bar_go);
            }
            if (!fast) {
                // the exact path takes this segment: its (unused) D_A product drained first
                stop = 1;
                if (!(par ? wait_group(2, kIssuer, bar_a1, ph_a1) : wait_group(2, kIssuer, bar_a, ph_a0)))
                    return;
                break;
            }
            if (tid == kIssuer && is_long(rpos + L))
                prefetch_state(rpos + L);   // read by the load at the end of this segment
            if (pend && !wait_group(2, kIssuer, bar_o, ph_o))
                return;
            // the products of the previous segment are complete: its operand set is free
            if (tid == kIssuer)
                mbar_arrive(bar_go);
            state_pass<D>(smem, tmem, -1, nullptr, true);   // the fp16 copy of S for D_O
            tc_fence_before();
            if (!sync_group(2))
                return;
            if (tid == kIssuer) {
                tc_fence_after();
                fast_issue_sq<D>(tmem, sb, par);
            }
            if (pend)
                out_epilogue<D>(tmem, outp(pend_tok), tstride, pend_L, pend_par, true);
            if (!(par ? wait_group(2, kIssuer, bar_a1, ph_a1) : wait_group(2, kIssuer, bar_a, ph_a0)))
                return;
            a_build<D>(smem, tmem, par);
            fence_proxy_async_smem();
            tc_fence_before();
            if (!sync_group(2))
                return;
            if (tid == kIssuer) {
                tc_fence_after();
                fast_issue_update<D, false>(tmem, sb, par);   // D_O only: the state is discarded
                tc_commit(bar_o);
            }
            pend = true;
            pend_par = par;
            pend_tok = rtok;
            pend_L = L;
            rpos += L;
            rtok += L;
            par ^= 1;
            ++kseq;
            if (!is_long(rpos))
                break;
            // the next segment's start state, while this segment's products run and the
            // builders build it (this segment's fp16 copy is made: TMEM S is free)
            state_load<D>(smem, tmem, st_g + (int64_t)seg_idx(rpos) * p.n_heads * D * D);
            loaded = seg_idx(rpos);
        }
        if (pend) {
            if (!wait_group(2, kIssuer, bar_o, ph_o))
                return;
            out_epilogue<D>(tmem, outp(pend_tok), tstride, pend_L, pend_par, false);
            tc_fence_before();
            if (!sync_group(2))
                return;
        }
        if (tid == kIssuer) {
            sMisc[3] = stop;
            sRun[0] = rpos;
            sRun[1] = rtok;
        }
    };

    // failure-detection hook (tests only): every thread joins one CTA-wide wait on an
    // mbarrier that nothing completes before the first decision (bar_go, phase 0); the
    // loader's bounded wait runs out and raises the abort flag, and the CTA leaves through
    // the abort path below
    if (p.stall_for_test) {
        uint32_t ph_stall = 0;
        wait_all(kLoader, bar_go, ph_stall);
    }

    int64_t pos = pos0, tok = 0;
    while (!aborted && pos < end) {
        if (RESTART && worker && loaded != seg_idx(pos)) {
            // this segment's own start state (the previous segment's state is not used)
            state_load<D>(smem, tmem, st_g + (int64_t)seg_idx(pos) * p.n_heads * D * D);
            tc_fence_before();
            bar_staters();
            tc_fence_after();
            loaded = seg_idx(pos);
        }
        const int L = seg_len(pos);
        if (L <= kShort) {
            // a leading or trailing short segment (its inputs are staged or in flight)
            if (!wait_tma())
                break;
            short_segment(tok, L, pos + L);
            pos += L;
            tok += L;
            continue;
        }
        if (builder)
            builder_run(pos, tok);
        else if constexpr (RESTART)
            state_run_restart(pos, tok);
        else
            state_run(pos, tok);
        if (!sync_all())
            break;
        tc_fence_after();
        const uint32_t stop = sMisc[3];
        pos = sRun[0];
        tok = sRun[1];
        kseq = 0;
        if (stop != 0) {
            // the segment at pos takes the exact path (1) or starts a new run (2): restage its
            // inputs (the copy of the next segment may be in flight)
            const int Lx = seg_len(pos);
            if (tid == kLoader) {
                if (tma_pending && !mbar_wait_bounded(bar_tma, ph_tma, kTimeoutNs))
                    sMisc[1] = 1;
                if (tma_pending)
                    ph_tma ^= 1;
                issue_tma(tok);
            }
            if (stop == 2)
                continue;   // the new run waits for the copy
            // every thread runs the exact segment
            if (!wait_tma())
                break;
            if (!exact_segment(tok, Lx, 0, 0, pos + Lx))
                break;
            pos += Lx;
            tok += Lx;
            if (tid == kLoader && pos < end)
                issue_tma(tok);
        }
    }

    if (!aborted) {
        if (!p.no_state_out)
            state_store<D>(tmem, st_g);   // final state back to global memory, row = key dim
    } else {
        // let this CTA's own copies and MMAs drain (bounded) before its memory goes away
        if (tid == kLoader) {
            report(p.d_err, HS_DEVERR_TIMEOUT);
            if (n_tma > 0)
                mbar_wait_bounded(bar_tma, (n_tma - 1) & 1, kTimeoutNs);
            tc_commit(bar_ld);   // the D_A products this thread issued
            mbar_wait_bounded(bar_ld, 0, kTimeoutNs);
        }
        if (tid == kIssuer) {
            tc_commit(bar_s);
            mbar_wait_bounded(bar_s, ph_s, kTimeoutNs);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}


}  // namespace

bool gla_chunked_tc_supported(int d)
{
    return d == 64 || d == 128;
}

namespace {

template <int D, bool RESTART>
cudaError_t launch_tc(const GlaParams &p, cudaStream_t s)
{
    TmaMaps maps;
    const uint64_t inner = (uint64_t)p.n_heads * D;
    // rows up to the last token any problem has: copies never read beyond the tokens the
    // caller passed (boxes reaching further are zero-filled), so q/k/v/log_g may be
    // offset views whose last rows run past the end of the allocation
    uint64_t rows = 0;
    for (int32_t b = 0; b < p.batch; ++b) {
        const uint64_t r = (uint64_t)p.row0[b] + (uint64_t)p.n_tokens[b];
        rows = r > rows ? r : rows;
    }
    if (rows == 0)
        return cudaSuccess;
    if (!encode_rows<D>(&maps.q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, p.q, inner, rows, 2) ||
        !encode_rows<D>(&maps.k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, p.k, inner, rows, 2) ||
        !encode_rows<D>(&maps.v, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, p.v, inner, rows, 2) ||
        !encode_rows<D>(&maps.g, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, p.log_g, inner, rows, 4))
        return cudaErrorInvalidValue;
    static std::atomic<uint64_t> smem_set{0};
    const unsigned grid = (unsigned)p.batch * (unsigned)p.n_heads;
    return launch_pdl_big_smem(gla_chunked_tc_kernel<D, RESTART>, dim3(grid), dim3(NT), SMEM_BYTES, s,
                               smem_set, p, maps);
}

}  // namespace

cudaError_t launch_gla_chunked_tc(const GlaParams &p, int d, cudaStream_t s)
{
    if (d == 128)
        return launch_tc<128, false>(p, s);
    if (d == 64)
        return launch_tc<64, false>(p, s);
    return cudaErrorNotSupported;
}

cudaError_t launch_gla_chunked_tc_restart(const GlaParams &p, int d, cudaStream_t s)
{
    if (d == 128)
        return launch_tc<128, true>(p, s);
    if (d == 64)
        return launch_tc<64, true>(p, s);
    return cudaErrorNotSupported;
}

}  // namespace hs
