// Semantic fallback retrieval (Sec. 3.3, Eq. 4-5): for every selected
// sequence, cos(R[j], q) over all candidate rows j in [0, len-2], threshold
// tau, top-k under (score desc, j desc).
//
// This is a bandwidth-bound batched GEMV (each cached row is read once and
// used once), so it runs on the CUDA cores, not the tensor cores.  Design:
//
//  * Persistent grid, one CTA per SM.  The rows of all selected sequences are
//    concatenated into one global row space [0, G) (the plan holds the
//    per-sequence prefix sums) and split into equal contiguous ranges, one per
//    CTA, so a few very long sequences and many short ones balance alike.
//  * A producer warp streams each CTA's range through a shared-memory ring of
//    stages with bulk TMA copies (cp.async.bulk, mbarrier complete_tx, L2
//    evict-first); a stage holds SR whole rows (one contiguous block).
//  * 8 consumer warps own fixed column slices: thread t holds the query
//    columns [8(t + 256c), +8) for c < MAXC in registers, so a row costs one
//    16-byte shared load and packed f32x2 FMAs for <R, q> and |R|^2.  The
//    2*SR partial sums of a stage are reduced across each warp with a
//    reduce-scatter, then across warps through shared memory; warps 1-7
//    signal them on a per-stage mbarrier that warp 0 waits on.
//  * Warp 0 finishes the cosines and keeps a register-resident top-k (one
//    entry per lane) that it updates with ballots.  At the end of each
//    sequence segment it publishes its partial list; the last CTA to publish
//    for a sequence (atomic counter) merges all partial lists, so the result
//    does not depend on CTA timing.
//  * Every wait inside the streaming loop is a bounded mbarrier wait; on
//    expiry the CTA raises ADAPLD_DEV_TIMEOUT, stops issuing copies, drains
//    the copies in flight, skips all further waits and exits without
//    publishing.  The only named barriers are the full-CTA ones at the start
//    and end of each sequence segment, which every consumer warp reaches in
//    the same order whatever happened in between.
#include <cstdio>
#include <cstdlib>

#include "common.cuh"

namespace adapld {

namespace {

constexpr int kProducerWarp = kConsumers2 / 32;  // warp 8
constexpr int kBarQ = 15;                        // named barrier for |q|^2
constexpr int kBarMerge = 14;                    // named barrier for the final merge
constexpr int kPlanCache = kConsumers2 + 32;     // plan entries kept in shared memory
static_assert(kPlanCache == kPlanInKernelB, "the lexical kernel leaves small plans to this one");

struct SemArgs {
    SemLaunch p;
    Workspace ws;
    int nstages;
    int stage_bytes;
    uint64_t wait_limit_ns;  // bound of every mbarrier wait
    int stall;               // test switch: the producer issues no copy
    const int64_t *plan;     // row prefix sums over the (virtual) sequences
    int32_t *done;           // per-sequence count of CTAs that published
    int32_t *slots;          // partial top-k lists
};

// The real sequence, the query token and the output row of (virtual)
// sequence p.
__device__ __forceinline__ int real_seq(const SemLaunch &a, int p) {
    return a.vseq_b ? a.vseq_b[p] : p;
}
__device__ __forceinline__ int out_row(const SemLaunch &a, int p) {
    return a.vseq_out ? a.vseq_out[p] : p;
}

// Token id of position j of real sequence b, clamped into the table (an
// out-of-range id reads row 0 and marks the sequence).
__device__ __forceinline__ int table_row(const SemLaunch &a, int b, int tok) {
    if (tok >= 0 && tok < a.vocab) return tok;
    if (a.status) atomicOr(a.status + b, ADAPLD_SEQ_BAD_TOKEN);
    return 0;
}

// Reduce-scatter of N values across a warp (N a power of two <= 32): after
// the call, lanes with lane % (32/N) == 0 hold in v[0] the warp total of
// value index lane / (32/N).
template <int N, int O>
struct ReduceScatter {
    static __device__ __forceinline__ void run(float *v, int lane) {
        if constexpr (O > 0) {
            if constexpr (N > 1) {
                constexpr int H = N / 2;
                const bool up = (lane & O) != 0;
#pragma unroll
                for (int i = 0; i < H; ++i) {
                    const float send = up ? v[i] : v[i + H];
                    const float keep = up ? v[i + H] : v[i];
                    v[i] = keep + __shfl_xor_sync(0xffffffffu, send, O);
                }
                ReduceScatter<H, O / 2>::run(v, lane);
            } else {
                v[0] += __shfl_xor_sync(0xffffffffu, v[0], O);
                ReduceScatter<1, O / 2>::run(v, lane);
            }
        }
    }
};

// Index of the CTA whose row range [c*G/grid, (c+1)*G/grid) holds row g.
__device__ __forceinline__ int cta_of(int64_t g, int64_t G, int grid) {
    return (int)(((g + 1) * grid - 1) / G);
}

__device__ __forceinline__ bool cta_nonempty(int c, int64_t G, int grid) {
    return ((int64_t)(c + 1) * G) / grid > ((int64_t)c * G) / grid;
}

// Largest b in [0, B) with plan[b] <= g (plan is non-decreasing, plan[0] = 0).
__device__ __forceinline__ int seq_of(const int64_t *plan, int B, int64_t g) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (plan[mid] <= g)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

// Two fp32 values in one 64-bit register, for the packed f32x2 FMA.
__device__ __forceinline__ uint64_t bf16x2_to_f32x2(uint32_t w) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(w << 16), "r"(w & 0xffff0000u));
    return r;
}

__device__ __forceinline__ uint64_t f32x2(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

__device__ __forceinline__ float sum_f32x2(uint64_t v) {
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
    return lo + hi;
}

// c += a * b on both halves (two fp32 FMAs, round to nearest).
__device__ __forceinline__ void fma2(uint64_t &c, uint64_t a, uint64_t b) {
    asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(c) : "l"(a), "l"(b));
}

// Variants whose per-thread state (query slice plus one stage of loads) is
// large get the register budget of one CTA per SM.
template <int MAXC, int SR>
constexpr int semantic_min_blocks() {
    return MAXC * (SR * 4 + 8) > 72 ? 1 : 2;
}

template <int MAXC, int SR, bool GATHER>
__global__ void __launch_bounds__(kConsumers2 + 32, (semantic_min_blocks<MAXC, SR>()))
    semantic_kernel(SemArgs args) {
    static_assert(32 % SR == 0, "a stage never straddles a 32-row id window");
    const SemLaunch &a = args.p;
    const Workspace &ws = args.ws;
    extern __shared__ __align__(128) uint8_t smem[];
    const int NS = args.nstages;
    const int stage_bytes = args.stage_bytes;
    uint8_t *ring = smem;
    float *red = (float *)(smem + (size_t)NS * stage_bytes);  // [max(NS,3)][32][8]
    float *qred = red + (NS > 3 ? NS : 3) * 32 * 8;            // [2][8]
    uint64_t *full = (uint64_t *)(qred + 16);                  // [NS] stage landed
    uint64_t *empty = full + kMaxStages2;                      // [NS] stage consumed
    uint64_t *redbar = empty + kMaxStages2;                    // [NS] partial sums written
    volatile int *abort_flag = (volatile int *)(redbar + kMaxStages2);
    int64_t *s_plan = (int64_t *)(abort_flag + 4);            // [kPlanCache]

    pdl_wait_then_release();  // the plan and the lexical outcomes come from the previous kernel
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int grid = gridDim.x, c = blockIdx.x;
    const int B = a.nvseq ? *a.nvseq : a.B, d = a.d, k = a.k;
    const int ostride = a.out_stride ? a.out_stride : k;
    if (B <= 0) return;
    // A plan of up to kPlanCache entries is read once, one entry per thread
    // (one memory round trip), and searched in shared memory; a longer one is
    // searched in global memory.  On the step path with B < kPlanCache the
    // CTA derives the plan itself from the lexical outcomes and the lengths
    // (one round trip and a block scan): a sequence without a lexical hit
    // and with a valid length contributes its len-1 rows.  hit_kind may
    // already read SEM or NONE for a sequence another CTA has finished; both
    // mean "no lexical hit", so every CTA derives the same plan.
    const bool cached = B < kPlanCache;
    if (a.plan_from_outcome) {
        int64_t rows = 0;
        if (t < B) {
            const int len = a.lengths[t];
            if (a.hit_kind[t] != ADAPLD_HIT_LEX && len >= 1 && (int64_t)len <= a.ld) rows = len - 1;
        }
        int64_t total;
        const int64_t ex = block_exclusive_scan(rows, &total, (int64_t *)red);
        if (t < B) s_plan[t] = ex;
        if (t == 0) s_plan[B] = total;
        __syncthreads();
    } else if (cached) {
        if (t <= B) s_plan[t] = args.plan[t];
        __syncthreads();
    }
    const int64_t *plan = cached ? s_plan : args.plan;
    const int64_t G = plan[B];
    if (G < 0 || G > (int64_t)B * a.ld) {  // never expected: the plan is corrupt
        if (t == 0 && c == 0) atomicOr(ws.dev_status, ADAPLD_DEV_INTERNAL);
        return;
    }
    const int64_t g0 = (int64_t)c * G / grid, g1 = (int64_t)(c + 1) * G / grid;
    if (g0 >= g1) return;

    if (t == 0) {
        for (int s = 0; s < NS; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kConsumers2 / 32);
            mbar_init(&redbar[s], kConsumers2 / 32 - 1);
        }
        *abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();

    const int b_first = seq_of(plan, B, g0);
    const size_t row_bytes = (size_t)d * 2;

    // ------------------------------------------------------------ producer
    if (warp == kProducerWarp) {
        // Gathered rows need their token ids: the whole warp keeps a window
        // of 32 upcoming ids; lane 0 issues the copies.
        if (!GATHER && lane != 0) return;
        // streamed cache rows are read once; embedding rows of frequent
        // tokens come back, so they stay ordinary L2 citizens
        const uint64_t pol = GATHER ? l2_evict_normal_policy() : l2_evict_first_policy();
        int it = 0;
        bool failed = false;
        int p = b_first;
        int64_t g = g0;
        while (g < g1 && !failed) {
            while (p < B - 1 && plan[p + 1] <= g) ++p;
            const int64_t seg_end = min(plan[p + 1], g1);
            if (seg_end <= g) {  // never expected: a corrupt plan
                if (lane == 0) atomicOr(ws.dev_status, ADAPLD_DEV_INTERNAL);
                break;
            }
            const int b = real_seq(a, p);
            const int jend = (int)(seg_end - plan[p]);
            // (checked build: the segment lies inside the sequence's rows)
            if (!idx_ok(jend, 1, a.ld + 1, ws.dev_status) || !idx_ok(b, 0, a.B, ws.dev_status))
                break;
            const uint8_t *base = (const uint8_t *)(a.reps + (int64_t)b * a.ld * d);
            const int32_t *Mb = GATHER ? a.tokens + (int64_t)b * a.ld : nullptr;
            // row ids in windows of 32 (SR divides 32, so a window starts on
            // a stage); the next window is loaded one window ahead
            const int jstart = (int)(g - plan[p]);
            int win = jstart, wtok = 0, wnext = 0;
            if (GATHER) {
                wtok = jstart + lane < jend ? Mb[jstart + lane] : 0;
                wnext = jstart + 32 + lane < jend ? Mb[jstart + 32 + lane] : 0;
            }
            for (int j = jstart; j < jend; j += SR) {
                const int nrows = min(SR, jend - j);
                const int s = it % NS, r = it / NS;
                int ok = 1;
                if (lane == 0) {
                    if (r > 0 && !mbar_wait_bounded(&empty[s], (r - 1) & 1, args.wait_limit_ns))
                        ok = 0;
                    if (*abort_flag || args.stall) ok = 0;
                }
                if (GATHER) ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) {
                    failed = true;
                    break;
                }
                const uint32_t bytes = (uint32_t)(nrows * row_bytes);
                uint8_t *dst = ring + (size_t)s * stage_bytes;
                if (GATHER) {
                    if (j >= win + 32) {
                        win += 32;
                        wtok = wnext;
                        wnext = win + 32 + lane < jend ? Mb[win + 32 + lane] : 0;
                    }
                    int rowtok[SR];
#pragma unroll
                    for (int rr = 0; rr < SR; ++rr)
                        rowtok[rr] = __shfl_sync(0xffffffffu, wtok, (j - win + rr) & 31);
                    if (lane == 0) {
                        mbar_arrive_expect_tx(&full[s], bytes);
#pragma unroll
                        for (int rr = 0; rr < SR; ++rr)
                            if (rr < nrows)
                                bulk_g2s(dst + (size_t)rr * row_bytes,
                                         a.reps + (int64_t)table_row(a, b, rowtok[rr]) * d,
                                         (uint32_t)row_bytes, &full[s], pol);
                    }
                } else {
                    mbar_arrive_expect_tx(&full[s], bytes);
                    bulk_g2s(dst, base + (size_t)j * row_bytes, bytes, &full[s], pol);
                }
                ++it;
            }
            g = seg_end;
        }
        if (failed && lane == 0) {
            *abort_flag = 1;
            atomicOr(ws.dev_status, ADAPLD_DEV_TIMEOUT);
            // drain the copies still in flight before the CTA may exit
            for (int i = max(0, it - NS); i < it; ++i)
                (void)mbar_wait_bounded(&full[i % NS], (uint32_t)(i / NS) & 1, args.wait_limit_ns);
        }
        return;
    }

    // ------------------------------------------------------------ consumers
    // column slice of this thread: 16-byte chunks t + 256*cc, cc < MAXC
    bool colok[MAXC];
#pragma unroll
    for (int cc = 0; cc < MAXC; ++cc) colok[cc] = (t + kConsumers2 * cc) * 8 < d;
    uint64_t q2[MAXC][4];
    WarpTopK tk;
    tk.reset();
    bool aborted = false;
    int it = 0, segno = 0;
    int p = b_first;
    int64_t g = g0;
    const float tau = a.tau;
    while (g < g1) {
        while (p < B - 1 && plan[p + 1] <= g) ++p;
        const int64_t seg_end = min(plan[p + 1], g1);
        if (seg_end <= g) break;  // never expected: a corrupt plan (flagged by the producer)
        const int jbeg = (int)(g - plan[p]);
        const int jend = (int)(seg_end - plan[p]);

        // query slice of this sequence (registers) and |q|^2
        float qpart = 0.f;
        const uint16_t *q;
        if (GATHER) {
            const int b = real_seq(a, p);
            const int qt = a.vseq_tok ? a.vseq_tok[p]
                                      : a.tokens[(int64_t)b * a.ld + a.lengths[b] - 1];
            q = a.reps + (int64_t)table_row(a, b, qt) * d;
        } else {
            q = a.query + (int64_t)p * d;
        }
#pragma unroll
        for (int cc = 0; cc < MAXC; ++cc) {
            const uint4 w = colok[cc] ? ldg_nc_v4(q + (t + kConsumers2 * cc) * 8)
                                      : make_uint4(0, 0, 0, 0);
            const uint32_t ws4[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float lo = bf16lo(ws4[e]), hi = bf16hi(ws4[e]);
                q2[cc][e] = f32x2(lo, hi);
                qpart = fmaf(lo, lo, qpart);
                qpart = fmaf(hi, hi, qpart);
            }
        }
        qpart = warp_sum(qpart);
        if (lane == 0) qred[(segno & 1) * 8 + warp] = qpart;
        named_bar_sync(kBarQ, kConsumers2);
        float qss = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) qss += qred[(segno & 1) * 8 + w];
        if (warp == 0) tk.reset();

        for (int j = jbeg; j < jend; j += SR) {
            const int nrows = min(SR, jend - j);
            const int s = it % NS;
            const uint32_t ph = (uint32_t)(it / NS) & 1;
            if (!aborted && !mbar_wait_bounded(&full[s], ph, args.wait_limit_ns)) {
                aborted = true;
                *abort_flag = 1;
                atomicOr(ws.dev_status, ADAPLD_DEV_TIMEOUT);
            }
            // all shared loads of this stage first, then the packed FMAs
            const uint8_t *st = ring + (size_t)s * stage_bytes + (size_t)t * 16;
            uint4 wv[SR][MAXC];
#pragma unroll
            for (int r = 0; r < SR; ++r)
#pragma unroll
                for (int cc = 0; cc < MAXC; ++cc)
                    wv[r][cc] = (r < nrows && colok[cc])
                                    ? *(const uint4 *)(st + (size_t)r * row_bytes +
                                                       (size_t)cc * kConsumers2 * 16)
                                    : make_uint4(0, 0, 0, 0);
            float acc[2 * SR];
#pragma unroll
            for (int r = 0; r < SR; ++r) {
                uint64_t dacc[2] = {0ull, 0ull}, sacc[2] = {0ull, 0ull};
#pragma unroll
                for (int cc = 0; cc < MAXC; ++cc) {
                    const uint32_t w4[4] = {wv[r][cc].x, wv[r][cc].y, wv[r][cc].z, wv[r][cc].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const uint64_t x = bf16x2_to_f32x2(w4[e]);
                        fma2(dacc[e & 1], x, q2[cc][e]);
                        fma2(sacc[e & 1], x, x);
                    }
                }
                acc[2 * r] = sum_f32x2(dacc[0]) + sum_f32x2(dacc[1]);
                acc[2 * r + 1] = sum_f32x2(sacc[0]) + sum_f32x2(sacc[1]);
            }
            ReduceScatter<2 * SR, 16>::run(acc, lane);
            constexpr int GRP = 32 / (2 * SR);
            if (lane % GRP == 0) red[(s * 32 + lane / GRP) * 8 + warp] = acc[0];
            __syncwarp();
            if (warp != 0) {
                if (lane == 0) {
                    mbar_arrive(&redbar[s]);
                    mbar_arrive(&empty[s]);
                }
            } else {
                // the other warps' partial sums of this stage (bounded; once
                // aborted the results are discarded and nothing is waited for)
                if (*abort_flag) aborted = true;
                if (!aborted && !mbar_wait_bounded(&redbar[s], ph, args.wait_limit_ns)) {
                    aborted = true;
                    *abort_flag = 1;
                    atomicOr(ws.dev_status, ADAPLD_DEV_TIMEOUT);
                }
                float dot = 0.f, ss = 0.f;
                if (lane < nrows) {
#pragma unroll
                    for (int w = 0; w < 8; ++w) {
                        dot += red[(s * 32 + 2 * lane) * 8 + w];
                        ss += red[(s * 32 + 2 * lane + 1) * 8 + w];
                    }
                }
                const float cs = cosine_from(dot, ss, qss);
                const bool want = lane < nrows && !aborted && cs >= tau;
                tk.insert(want, cs, j + lane, k);
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[s]);
            }
            ++it;
        }

        // ---- end of this CTA's segment of sequence b: publish; the CTA that
        // publishes last for b merges every partial list, with all 8 warps
        const int cfirst = cta_of(plan[p], G, grid);
        const int clast = cta_of(plan[p + 1] - 1, G, grid);
        volatile int *s_flag = (volatile int *)abort_flag + 1;  // the merge decision
        if (warp == 0) {
            int last = 0;
            if (!aborted && !*abort_flag && idx_ok(p + c, 0, B + grid, ws.dev_status)) {
                int32_t *sp = args.slots + (int64_t)(p + c) * kSlotInts;
                if (lane == 0) sp[0] = tk.n;
                if (lane < tk.n) {
                    sp[1 + lane] = tk.j;
                    sp[1 + kMaxK + lane] = __float_as_int(tk.s);
                }
                __threadfence();
                __syncwarp();
                int expected = clast - cfirst + 1;
                if (G < grid) {
                    expected = 0;
                    for (int cc = cfirst; cc <= clast; ++cc) expected += cta_nonempty(cc, G, grid);
                }
                if (lane == 0) last = atomicAdd(args.done + p, 1) == expected - 1;
                last = __shfl_sync(0xffffffffu, last, 0);
            }
            if (lane == 0) *s_flag = last;
        }
        named_bar_sync(kBarMerge, kConsumers2);
        const bool merge = *s_flag != 0;
        if (merge) {
            __threadfence();
            // each warp merges every 8th contributing CTA's list, 4 lists per
            // round of independent loads
            WarpTopK m;
            m.reset();
            for (int cc0 = cfirst + warp * 4; cc0 <= clast; cc0 += 8 * 4) {
                int n[4], xj[4];
                float xs[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int cc = cc0 + u;
                    const bool ok = cc <= clast && cta_nonempty(cc, G, grid);
                    const int32_t *op = args.slots + (int64_t)(p + (ok ? cc : c)) * kSlotInts;
                    n[u] = ok ? __ldcg(op) : 0;
                    xj[u] = ok ? __ldcg(op + 1 + lane) : -1;
                    xs[u] = ok ? __int_as_float(__ldcg(op + 1 + kMaxK + lane)) : 0.f;
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) m.insert(lane < n[u], xs[u], xj[u], k);
            }
            float *wl_s = red;                          // [8][32] per-warp lists
            int *wl_j = (int *)(red + 8 * 32);          // [8][32]
            int *wl_n = (int *)(red + 16 * 32);         // [8]
            wl_s[warp * 32 + lane] = m.s;
            wl_j[warp * 32 + lane] = m.j;
            if (lane == 0) wl_n[warp] = m.n;
            named_bar_sync(kBarMerge, kConsumers2);
            if (warp == 0) {
                WarpTopK f;
                f.reset();
                for (int w = 0; w < 8; ++w)
                    f.insert(lane < wl_n[w], wl_s[w * 32 + lane], wl_j[w * 32 + lane], k);
                const int64_t orow = out_row(a, p);
                if (lane < k) {
                    a.cand[orow * ostride + lane] = lane < f.n ? f.j : -1;
                    a.score[orow * ostride + lane] = lane < f.n ? f.s : 0.f;
                }
                if (lane == 0) {
                    a.n_cand[orow] = f.n;
                    if (a.hit_kind) a.hit_kind[orow] = f.n > 0 ? ADAPLD_HIT_SEM : ADAPLD_HIT_NONE;
                }
            }
            named_bar_sync(kBarMerge, kConsumers2);  // before red is reused by the next stage
        }
        g = seg_end;
        ++segno;
    }
}

// Shared memory per CTA: the ring, the per-stage reduction buffers (at least
// three, which the final merge reuses for the per-warp lists), |q|^2
// partials, the barriers, the abort flag and the merge decision.
inline size_t semantic_smem(int ns, int stage) {
    return (size_t)ns * stage + (size_t)(ns > 3 ? ns : 3) * 32 * 8 * 4 + 16 * 4 +
           3 * kMaxStages2 * 8 + 16 + (size_t)kPlanCache * 8;
}

template <int MAXC, int SR, bool GATHER>
cudaError_t launch_variant(const SemArgs &args0, int sms, int ctas_per_sm, int stages,
                           cudaStream_t s) {
    SemArgs args = args0;
    auto kern = semantic_kernel<MAXC, SR, GATHER>;
    const int stage = (int)align_up((size_t)SR * args.p.d * 2, 128);
    // shared memory budget per CTA for the requested CTAs per SM
    const size_t per_sm = 227 * 1024;
    int cps = ctas_per_sm < 1 ? 1 : ctas_per_sm;
    int ns = 0;
    for (; cps >= 1; --cps) {
        const size_t budget = (per_sm - (size_t)(cps - 1) * 1024) / cps;
        ns = 0;
        while (ns < kMaxStages2 && (stages <= 0 || ns < stages) &&
               semantic_smem(ns + 1, stage) <= budget)
            ++ns;
        if (ns >= 2) break;
    }
    if (cps < 1 || ns < 2) return cudaErrorInvalidConfiguration;
    args.nstages = ns;
    args.stage_bytes = stage;
    const size_t smem = semantic_smem(ns, stage);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    int fit = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&fit, kern, kConsumers2 + 32, smem);
    if (e != cudaSuccess) return e;
    if (fit < 1) return cudaErrorInvalidConfiguration;
    if (cps > fit) cps = fit;
    int grid = sms * cps;
    if (grid > kMaxGrid2) grid = kMaxGrid2;
    if (std::getenv("ADAPLD_SEMANTIC_TUNING"))
        std::fprintf(stderr, "adapld semantic: d=%d rows/stage=%d stages=%d stage_bytes=%d "
                     "ctas/SM=%d grid=%d smem=%zu\n", args.p.d, SR, ns, stage, cps, grid, smem);
    return launch_dependent(kern, dim3(grid), dim3(kConsumers2 + 32), smem, s, args);
}

// Launch shape: CTAs per SM, rows per stage and stages per CTA.  The defaults
// come from sweeps on GB300: about 128 KB of bulk copies in flight per SM, in
// 32-64 KB copies, is fastest (deeper rings lose bandwidth, 16 KB copies too),
// i.e. 2 CTAs/SM with 2 stages of ~32-48 KB for d <= 8192.
// ADAPLD_SEMANTIC_TUNING="<ctas_per_sm>,<rows_per_stage>[,<stages>]" overrides
// them for tuning sweeps (0 keeps the default; the launch shape chosen is then
// printed to stderr).
struct SemTuning {
    int ctas_per_sm = 0;
    int rows = 0;
    int stages = 0;
};

SemTuning semantic_tuning() {
    SemTuning t;
    if (const char *e = std::getenv("ADAPLD_SEMANTIC_TUNING")) {
        int a = 0, b = 0, c = 0;
        if (std::sscanf(e, "%d,%d,%d", &a, &b, &c) >= 1 && a >= 1 && a <= 4) t.ctas_per_sm = a;
        if (b == 1 || b == 2 || b == 4 || b == 8 || b == 16) t.rows = b;
        if (c >= 2 && c <= kMaxStages2) t.stages = c;
    }
    return t;
}

}  // namespace

int device_sms() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return sms;
}

cudaError_t launch_semantic(const SemLaunch &a, const Workspace &ws, cudaStream_t s) {
    if (!a.plan_ready) {
        cudaError_t e = launch_plan(a.lengths, a.ld, a.B, a.active, a.k, a.cand, a.score,
                                    a.n_cand, ws, s);
        if (e != cudaSuccess) return e;
    }
    const int sms = device_sms();
    if (sms <= 0) return cudaErrorInvalidDevice;
    const SemTuning tun = semantic_tuning();
    SemArgs args{a, ws, 0, 0, kWaitLimitNs, 0, ws.plan, ws.done2, ws.slots2};
    if (a.nvseq) {  // the successor backoff pass has its own plan, counters and slots
        args.plan = ws.plan3;
        args.done = ws.done3;
        args.slots = ws.slots3;
    }
    // Test switch for the timeout path: the producer issues nothing, every
    // consumer wait runs out after 20 ms, the call reports ADAPLD_DEV_TIMEOUT
    // and publishes no result.  Never set in normal use.
    if (const char *e = std::getenv("ADAPLD_TEST_SEMANTIC_STALL")) {
        if (e[0] == '1') {
            args.stall = 1;
            args.wait_limit_ns = 20000000ull;
        }
    }
    const int d = a.d, R = tun.rows;
    // gathered rows (scattered table rows) want more bytes in flight than
    // streamed ones: a third stage where it fits at 2 CTAs/SM (measured on
    // GB300 in two-representation steps: 3-7% less time per step at d = 4096
    // and d = 8192; streamed rows lose bandwidth with it)
    const int gs = a.tokens ? 3 : 2;
#define ADAPLD_SEM(MAXC, SR, CPS, NS)                                                       \
    return (a.tokens ? launch_variant<MAXC, SR, true> : launch_variant<MAXC, SR, false>)(    \
        args, sms, tun.ctas_per_sm ? tun.ctas_per_sm : CPS, tun.stages ? tun.stages : NS, s)
    if (d <= 2048) {
        if (R == 4) ADAPLD_SEM(1, 4, 2, 2);
        if (R == 16) ADAPLD_SEM(1, 16, 2, 2);
        ADAPLD_SEM(1, 8, 2, gs);
    }
    if (d <= 4096) {
        if (R == 2) ADAPLD_SEM(2, 2, 2, 2);
        if (R == 8) ADAPLD_SEM(2, 8, 2, 2);
        ADAPLD_SEM(2, 4, 2, gs);
    }
    if (d <= 6144) {
        if (R == 2) ADAPLD_SEM(3, 2, 2, 2);
        ADAPLD_SEM(3, 4, 2, 2);
    }
    if (d <= 8192) {
        if (R == 1) ADAPLD_SEM(4, 1, 2, 4);
        if (R == 4) ADAPLD_SEM(4, 4, 1, 2);
        ADAPLD_SEM(4, 2, 2, gs);
    }
    if (d <= 12288) {
        if (R == 2) ADAPLD_SEM(6, 2, 1, 2);
        ADAPLD_SEM(6, 1, 2, 3);
    }
    if (R == 2) ADAPLD_SEM(8, 2, 1, 2);
    ADAPLD_SEM(8, 1, 1, 4);
#undef ADAPLD_SEM
}

}  // namespace adapld
