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
//    16-byte shared load, 8 FMAs for <R, q> and 8 for |R|^2 per slice.  The
//    2*SR partial sums of a stage are reduced across each warp with a
//    reduce-scatter, then across warps through shared memory.
//  * Warp 0 finishes the cosines and keeps a register-resident top-k (one
//    entry per lane) that it updates with ballots.  At the end of each
//    sequence segment it publishes its partial list; the last CTA to publish
//    for a sequence (atomic counter) merges all partial lists, so the result
//    does not depend on CTA timing.
//  * Every mbarrier wait is bounded; on expiry the CTA raises
//    ADAPLD_DEV_TIMEOUT, stops issuing copies, drains the copies in flight and
//    exits without publishing.
#include "common.cuh"

namespace adapld {

namespace {

constexpr int kRingBytes = 192 * 1024;
constexpr int kProducerWarp = kConsumers2 / 32;  // warp 8
constexpr int kBarQ = 15;                        // named barrier for |q|^2

struct SemArgs {
    SemLaunch p;
    Workspace ws;
    int nstages;
    int stage_bytes;
};

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

template <int MAXC, int SR>
__global__ void __launch_bounds__(kConsumers2 + 32, 1) semantic_kernel(SemArgs args) {
    const SemLaunch &a = args.p;
    const Workspace &ws = args.ws;
    extern __shared__ __align__(128) uint8_t smem[];
    const int NS = args.nstages;
    const int stage_bytes = args.stage_bytes;
    uint8_t *ring = smem;
    float *red = (float *)(smem + (size_t)NS * stage_bytes);  // [kMaxStages2][32][8]
    float *qred = red + kMaxStages2 * 32 * 8;                  // [2][8]
    uint64_t *full = (uint64_t *)(qred + 16);                  // [kMaxStages2]
    uint64_t *empty = full + kMaxStages2;                      // [kMaxStages2]
    volatile int *abort_flag = (volatile int *)(empty + kMaxStages2);

    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int grid = gridDim.x, c = blockIdx.x;
    const int B = a.B, d = a.d, k = a.k;
    const int64_t *plan = ws.plan;
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
        }
        *abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();

    const int b_first = seq_of(plan, B, g0);
    const size_t row_bytes = (size_t)d * 2;

    // ------------------------------------------------------------ producer
    if (warp == kProducerWarp) {
        if (lane != 0) return;
        const uint64_t pol = l2_evict_first_policy();
        int it = 0;
        bool failed = false;
        int b = b_first;
        int64_t g = g0;
        while (g < g1 && !failed) {
            while (b < B - 1 && plan[b + 1] <= g) ++b;
            const int64_t seg_end = min(plan[b + 1], g1);
            if (seg_end <= g) {  // never expected: a corrupt plan
                atomicOr(ws.dev_status, ADAPLD_DEV_INTERNAL);
                break;
            }
            const int jend = (int)(seg_end - plan[b]);
            const uint8_t *base = (const uint8_t *)(a.reps + (int64_t)b * a.ld * d);
            for (int j = (int)(g - plan[b]); j < jend; j += SR) {
                const int nrows = min(SR, jend - j);
                const int s = it % NS, r = it / NS;
                if (r > 0 && !mbar_wait_bounded(&empty[s], (r - 1) & 1)) {
                    failed = true;
                    break;
                }
                if (*abort_flag) {
                    failed = true;
                    break;
                }
                const uint32_t bytes = (uint32_t)(nrows * row_bytes);
                mbar_arrive_expect_tx(&full[s], bytes);
                bulk_g2s(ring + (size_t)s * stage_bytes, base + (size_t)j * row_bytes, bytes,
                         &full[s], pol);
                ++it;
            }
            g = seg_end;
        }
        if (failed) {
            *abort_flag = 1;
            atomicOr(ws.dev_status, ADAPLD_DEV_TIMEOUT);
            // drain the copies still in flight before the CTA may exit
            for (int i = max(0, it - NS); i < it; ++i)
                (void)mbar_wait_bounded(&full[i % NS], (uint32_t)(i / NS) & 1);
        }
        return;
    }

    // ------------------------------------------------------------ consumers
    float qf[MAXC][8];
    WarpTopK tk;
    tk.reset();
    bool aborted = false;
    int it = 0, segno = 0;
    int b = b_first;
    int64_t g = g0;
    const float tau = a.tau;
    while (g < g1) {
        while (b < B - 1 && plan[b + 1] <= g) ++b;
        const int64_t seg_end = min(plan[b + 1], g1);
        if (seg_end <= g) break;  // never expected: a corrupt plan (flagged by the producer)
        const int jbeg = (int)(g - plan[b]);
        const int jend = (int)(seg_end - plan[b]);

        // query slice of this sequence and |q|^2
        float qpart = 0.f;
        const uint16_t *q = a.query + (int64_t)b * d;
#pragma unroll
        for (int cc = 0; cc < MAXC; ++cc) {
            const int col8 = t + kConsumers2 * cc;
            if (col8 * 8 < d) {
                const uint4 w = ldg_nc_v4(q + col8 * 8);
                qf[cc][0] = bf16lo(w.x);
                qf[cc][1] = bf16hi(w.x);
                qf[cc][2] = bf16lo(w.y);
                qf[cc][3] = bf16hi(w.y);
                qf[cc][4] = bf16lo(w.z);
                qf[cc][5] = bf16hi(w.z);
                qf[cc][6] = bf16lo(w.w);
                qf[cc][7] = bf16hi(w.w);
#pragma unroll
                for (int e = 0; e < 8; ++e) qpart = fmaf(qf[cc][e], qf[cc][e], qpart);
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) qf[cc][e] = 0.f;
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
            if (!aborted && !mbar_wait_bounded(&full[s], ph)) {
                aborted = true;
                *abort_flag = 1;
                atomicOr(ws.dev_status, ADAPLD_DEV_TIMEOUT);
            }
            if (*abort_flag) aborted = true;

            float acc[2 * SR];
#pragma unroll
            for (int i = 0; i < 2 * SR; ++i) acc[i] = 0.f;
            const uint8_t *st = ring + (size_t)s * stage_bytes;
#pragma unroll
            for (int r = 0; r < SR; ++r) {
                if (r < nrows) {
#pragma unroll
                    for (int cc = 0; cc < MAXC; ++cc) {
                        const int col8 = t + kConsumers2 * cc;
                        if (col8 * 8 < d) {
                            const uint4 w =
                                *(const uint4 *)(st + (size_t)r * row_bytes + (size_t)col8 * 16);
                            const float x0 = bf16lo(w.x), x1 = bf16hi(w.x);
                            const float x2 = bf16lo(w.y), x3 = bf16hi(w.y);
                            const float x4 = bf16lo(w.z), x5 = bf16hi(w.z);
                            const float x6 = bf16lo(w.w), x7 = bf16hi(w.w);
                            float dt = acc[2 * r], ss = acc[2 * r + 1];
                            dt = fmaf(x0, qf[cc][0], dt);
                            dt = fmaf(x1, qf[cc][1], dt);
                            dt = fmaf(x2, qf[cc][2], dt);
                            dt = fmaf(x3, qf[cc][3], dt);
                            dt = fmaf(x4, qf[cc][4], dt);
                            dt = fmaf(x5, qf[cc][5], dt);
                            dt = fmaf(x6, qf[cc][6], dt);
                            dt = fmaf(x7, qf[cc][7], dt);
                            ss = fmaf(x0, x0, ss);
                            ss = fmaf(x1, x1, ss);
                            ss = fmaf(x2, x2, ss);
                            ss = fmaf(x3, x3, ss);
                            ss = fmaf(x4, x4, ss);
                            ss = fmaf(x5, x5, ss);
                            ss = fmaf(x6, x6, ss);
                            ss = fmaf(x7, x7, ss);
                            acc[2 * r] = dt;
                            acc[2 * r + 1] = ss;
                        }
                    }
                }
            }
            ReduceScatter<2 * SR, 16>::run(acc, lane);
            constexpr int GRP = 32 / (2 * SR);
            if (lane % GRP == 0) red[(s * 32 + lane / GRP) * 8 + warp] = acc[0];
            __syncwarp();
            if (warp != 0) {
                if (lane == 0) mbar_arrive(&empty[s]);
                named_bar_arrive(1 + s, kConsumers2);
            } else {
                named_bar_sync(1 + s, kConsumers2);
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

        // ---- end of this CTA's segment of sequence b: publish, maybe merge
        if (warp == 0 && !aborted) {
            const int slot = b + c;
            int32_t *sp = ws.slots2 + (int64_t)slot * kSlotInts;
            if (lane == 0) sp[0] = tk.n;
            if (lane < tk.n) {
                sp[1 + lane] = tk.j;
                sp[1 + kMaxK + lane] = __float_as_int(tk.s);
            }
            __threadfence();
            __syncwarp();
            const int cfirst = cta_of(plan[b], G, grid);
            const int clast = cta_of(plan[b + 1] - 1, G, grid);
            int expected = clast - cfirst + 1;
            if (G < grid) {
                expected = 0;
                for (int cc = cfirst; cc <= clast; ++cc) expected += cta_nonempty(cc, G, grid);
            }
            int last = 0;
            if (lane == 0) last = atomicAdd(ws.done2 + b, 1) == expected - 1;
            last = __shfl_sync(0xffffffffu, last, 0);
            if (last) {
                __threadfence();
                WarpTopK m;
                m.reset();
                for (int cc = cfirst; cc <= clast; ++cc) {
                    if (!cta_nonempty(cc, G, grid)) continue;
                    const int32_t *op = ws.slots2 + (int64_t)(b + cc) * kSlotInts;
                    const int n = __ldcg(op);
                    float xs = 0.f;
                    int xj = -1;
                    if (lane < n) {
                        xj = __ldcg(op + 1 + lane);
                        xs = __int_as_float(__ldcg(op + 1 + kMaxK + lane));
                    }
                    m.insert(lane < n, xs, xj, k);
                }
                if (lane < k) {
                    a.cand[(int64_t)b * k + lane] = lane < m.n ? m.j : -1;
                    a.score[(int64_t)b * k + lane] = lane < m.n ? m.s : 0.f;
                }
                if (lane == 0) {
                    a.n_cand[b] = m.n;
                    if (a.hit_kind) a.hit_kind[b] = m.n > 0 ? ADAPLD_HIT_SEM : ADAPLD_HIT_NONE;
                }
            }
        }
        g = seg_end;
        ++segno;
    }
}

template <int MAXC, int SR>
cudaError_t launch_variant(const SemArgs &args0, int grid, cudaStream_t s) {
    SemArgs args = args0;
    const int stage = (int)align_up((size_t)SR * args.p.d * 2, 128);
    int ns = kRingBytes / stage;
    ns = ns > kMaxStages2 ? kMaxStages2 : (ns < 2 ? 2 : ns);
    args.nstages = ns;
    args.stage_bytes = stage;
    const size_t smem = (size_t)ns * stage + kMaxStages2 * 32 * 8 * 4 + 16 * 4 +
                        2 * kMaxStages2 * 8 + 16;
    auto kern = semantic_kernel<MAXC, SR>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, kConsumers2 + 32, smem, s>>>(args);
    return cudaGetLastError();
}

}  // namespace

int semantic_grid() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return sms < kMaxGrid2 ? sms : kMaxGrid2;
}

cudaError_t launch_semantic(const SemLaunch &a, const Workspace &ws, cudaStream_t s) {
    if (!a.plan_ready) {
        cudaError_t e = launch_plan(a.lengths, a.ld, a.B, a.active, a.k, a.cand, a.score,
                                    a.n_cand, ws, s);
        if (e != cudaSuccess) return e;
    }
    const int grid = semantic_grid();
    if (grid <= 0) return cudaErrorInvalidDevice;
    SemArgs args{a, ws, 0, 0};
    const int d = a.d;
    if (d <= 2048) return launch_variant<1, 16>(args, grid, s);
    if (d <= 4096) return launch_variant<2, 4>(args, grid, s);
    if (d <= 6144) return launch_variant<3, 4>(args, grid, s);
    if (d <= 8192) return launch_variant<4, 2>(args, grid, s);
    if (d <= 12288) return launch_variant<6, 2>(args, grid, s);
    return launch_variant<8, 1>(args, grid, s);
}

}  // namespace adapld
