// Lexical anchoring (Sec. 3.3, Eq. 3, generalised to the longest suffix
// n-gram).
//
// Grid (X, B), 512 threads; the X CTAs of a sequence form one thread-block
// cluster (X <= 8, or 16 for a few long sequences).  CTA x scans a contiguous
// range of 8192-position chunks, most recent chunk first; thread t of a chunk
// owns the 16 consecutive positions j0 + 16 t .. j0 + 16 t + 15.  Each thread
// loads its window -- its 16 tokens and the 8 before them -- from global
// memory into registers (16-byte loads where the row is aligned); the window
// of the CTA's most recent chunk is requested before the sequence length
// arrives (it is at the same place whatever the length), so the two round
// trips overlap.  For each position j the backward match length
// m(j) = #{i : M[j-i'] == M[len-1-i'] for all i' <= i}, capped at
// min(n_max, len-1), is built as bit masks over the thread's 16 positions:
// the positions matching the anchor token, then those of them whose next
// older token matches too, and so on while any is left.  A warp reduces its
// maximum and the count of its positions reaching it, scanned from the top
// lane; after one CTA barrier every thread knows the chunk maximum and where
// its own hits rank, most recent first, and writes them straight into the
// CTA's running result (a longer match replaces it, an equal one appends).
// With several CTAs each one then pushes its result into the shared memory
// of CTA rank 0 (distributed shared memory), and after one cluster barrier
// rank 0 merges them locally: n* = max m, candidates = the k most recent
// positions with m(j) = n* (higher ranks hold more recent chunks).
//
// On the step path the kernel also zeroes the workspace counters of the
// step's later kernels, so a step needs no memset, and it is launched as a
// programmatic dependent of whatever kernel precedes it in the stream.  For
// B < 288 the semantic kernel derives its row plan from the outcomes itself;
// for larger batches outcome_plan_kernel writes it.
#include <cstdlib>

#include "common.cuh"

namespace adapld {

namespace {

constexpr int kWarpsL = kThreadsL / 32;
constexpr int kPerThreadL = kChunkL / kThreadsL;  // consecutive positions per thread (16)
constexpr int kHaloL = 8;                         // tokens before them (n_max - 1 <= 7 used)
constexpr int kWinL = kHaloL + kPerThreadL;       // window of a thread (24 tokens)
constexpr int kResL = 2 + kMaxK;                  // a CTA's result: m, count, positions
static_assert(kPerThreadL == 16 && kWinL % 4 == 0, "16 positions, whole 16-byte groups");

struct LexArgs {
    LexLaunch p;
    Workspace ws;
    int q;  // chunks per CTA
};

// W[w] = M[base - kHaloL + w] for w < kWinL; entries outside the row [0, lim)
// read as -1 (positions are bounded separately, so they are never compared).
__device__ __forceinline__ void load_window(int (&W)[kWinL], const int32_t *M, int base, int lim,
                                            bool vec) {
#pragma unroll
    for (int g = 0; g < kWinL / 4; ++g) {
        const int i0 = base - kHaloL + 4 * g;
        if (vec && i0 >= 0 && i0 + 4 <= lim) {
            const int4 v = __ldg(reinterpret_cast<const int4 *>(M + i0));
            W[4 * g] = v.x;
            W[4 * g + 1] = v.y;
            W[4 * g + 2] = v.z;
            W[4 * g + 3] = v.w;
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u)
                W[4 * g + u] = (i0 + u >= 0 && i0 + u < lim) ? __ldg(M + i0 + u) : -1;
        }
    }
}

__global__ void __launch_bounds__(kThreadsL, 2) lexical_kernel(LexArgs args) {
    const LexLaunch &a = args.p;
    __shared__ int wmax_s[kWarpsL];            // per warp: its longest match in the chunk
    __shared__ int wtot_s[kWarpsL];            // ... and its positions reaching it
    __shared__ int res[kResL];                 // this CTA's result
    __shared__ int mres[kWideClusterL][kResL]; // rank 0: every CTA's result

    pdl_wait_then_release();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int b = blockIdx.y, x = blockIdx.x, X = gridDim.x;
    // every CTA of the cluster has started before results are pushed (the
    // matching wait comes after the scan)
    if (X > 1) cluster_arrive_relaxed();
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const bool vec = ((uintptr_t)M & 15) == 0;
    const int lim = (int)a.ld;
    // the most recent chunk of this CTA were the sequence full: its window
    // is requested together with the length
    const int c_spec = min(x * args.q + args.q, chunks_of(a.ld - 1, kChunkL)) - 1;
    int W[kWinL];
    int loaded = -1;
    if (c_spec >= x * args.q) {
        load_window(W, M, c_spec * kChunkL + kPerThreadL * t, lim, vec);
        loaded = c_spec;
    }
    const int len = a.lengths[b];
    const bool valid = len >= 1 && (int64_t)len <= a.ld;
    const int nj = valid ? len - 1 : 0;  // candidates j in [0, len-2]
    const int top = valid ? min(a.n_max, len - 1) : 0;
    const int nchunks = (nj + kChunkL - 1) / kChunkL;
    const int c_lo = x * args.q, c_hi = min(c_lo + args.q, nchunks);

    if (a.zero) {  // the later kernels' counters (grid-stride over every thread)
        const size_t nthreads = (size_t)gridDim.x * gridDim.y * kThreadsL;
        for (size_t i = ((size_t)b * X + x) * kThreadsL + t; i < a.zero_words; i += nthreads)
            a.zero[i] = 0;
    }
    if (a.stats && b == 0 && x == 0 && t < 4) a.stats[t] = 0;
    int suf[8];  // the suffix, most recent token first (broadcast loads)
#pragma unroll
    for (int i = 0; i < 8; ++i) suf[i] = i < top ? __ldg(M + len - 1 - i) : 0;

    int rm = 0, rn = 0;  // the CTA's best length so far and its positions (same in every thread)
    for (int c = c_hi - 1; c >= c_lo && top > 0; --c) {
        const int base = c * kChunkL + kPerThreadL * t;
        if (c != loaded) {
            load_window(W, M, base, lim, vec);
            loaded = c;
        }
        // al: positions whose last i + 1 tokens match the suffix; hits: the
        // longest such set met, of length mymax
        uint32_t al = 0;
#pragma unroll
        for (int e = 0; e < kPerThreadL; ++e)
            al |= (uint32_t)(base + e < nj && W[kHaloL + e] == suf[0]) << e;
        uint32_t hits = al;
        int mymax = al ? 1 : 0;
#pragma unroll
        for (int i = 1; i < 8; ++i) {
            if (i >= top || al == 0) break;
            uint32_t eq = 0;
#pragma unroll
            for (int e = 0; e < kPerThreadL; ++e)
                eq |= (uint32_t)(W[kHaloL + e - i] == suf[i]) << e;
            if (base == 0) eq &= ~((1u << i) - 1u);  // positions j < i have no token j - i
            al &= eq;
            if (al) {
                hits = al;
                mymax = i + 1;
            }
        }
        // rank most recent first: higher warps, then higher lanes, then
        // higher positions of a thread
        const int wmax = warp_max_i(mymax);
        const int mine = (wmax > 0 && mymax == wmax) ? __popc(hits) : 0;
        int incl = mine;  // over this lane and the higher ones
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_down_sync(0xffffffffu, incl, o);
            if (lane + o < 32) incl += u;
        }
        if (lane == 0) {
            wmax_s[warp] = wmax;
            wtot_s[warp] = incl;
        }
        __syncthreads();
        int cmax = 0;
#pragma unroll
        for (int w = 0; w < kWarpsL; ++w) cmax = max(cmax, wmax_s[w]);
        int before = 0, total = 0;  // the chunk's hits in higher warps / in all
#pragma unroll
        for (int w = 0; w < kWarpsL; ++w) {
            const int n = wmax_s[w] == cmax ? wtot_s[w] : 0;
            total += n;
            before += w > warp ? n : 0;
        }
        if (cmax > 0 && cmax >= rm) {  // a longer match replaces the result, an equal one appends
            const int off = cmax > rm ? 0 : rn;
            const int room = a.k - off;
            if (wmax == cmax && mine > 0) {
                int r = before + incl - mine;
                for (uint32_t h = hits; h && r < room; ++r) {
                    const int e = 31 - __clz(h);
                    h &= ~(1u << e);
                    res[2 + off + r] = base + e;
                }
            }
            rn = off + min(total, room);
            rm = cmax;
        }
        __syncthreads();  // res is complete; wmax_s and wtot_s may be rewritten
    }

    // ---- the sequence's result ------------------------------------------------
    int32_t *cb = a.cand + (int64_t)b * a.k;
    int best = rm, total = rm > 0 ? rn : 0;
    if (X > 1) {
        cluster_wait();  // every CTA has started
        if (warp == 0) {
            if (lane == 0) st_cluster_i32(&mres[x][0], 0, rm);
            if (lane == 1) st_cluster_i32(&mres[x][1], 0, rn);
            if (lane < rn) st_cluster_i32(&mres[x][2 + lane], 0, res[2 + lane]);
        }
        cluster_sync_all();  // the pushes are visible to rank 0
        if (x != 0) return;
        if (warp == 0) {
            best = lane < X ? mres[lane][0] : 0;
            best = warp_max_i(best);
            total = 0;
            if (best > 0)
                total = warp_merge_desc(
                    X, a.k, [&](int r) { return mres[r][0] == best ? mres[r][1] : 0; },
                    [&](int r, int i) { return mres[r][2 + i]; }, cb);
        }
    } else if (warp == 0 && lane < total) {
        cb[lane] = res[2 + lane];
    }
    if (warp == 0) {
        if (lane >= total && lane < a.k) cb[lane] = -1;
        if (a.score && lane < a.k) a.score[(int64_t)b * a.k + lane] = 0.f;
        if (lane == 0) {
            a.match_n[b] = best;
            a.n_cand[b] = total;
            a.hit_kind[b] = best > 0 ? ADAPLD_HIT_LEX : ADAPLD_HIT_NONE;
            if (a.status) a.status[b] = valid ? 0 : ADAPLD_SEQ_BAD_LENGTH;
        }
    }
}

struct PlanArgs {
    const int32_t *lengths;
    int64_t ld;
    int32_t B;
    const int32_t *hit_kind;  // selection by outcome (then active is unused)
    const uint8_t *active;
    int32_t k;
    int32_t *cand;
    float *score;
    int32_t *n_cand;
    int64_t *plan;
};

__global__ void __launch_bounds__(kThreads1) plan_kernel(PlanArgs a) {
    build_plan_cta(a.lengths, a.ld, a.B, nullptr, a.active, a.plan, true, a.k, a.cand, a.score,
                   a.n_cand);
}

__global__ void __launch_bounds__(kThreads1) outcome_plan_kernel(PlanArgs a) {
    pdl_wait_then_release();  // the outcomes come from the lexical kernel
    build_plan_cta(a.lengths, a.ld, a.B, a.hit_kind, nullptr, a.plan, false, 0, nullptr, nullptr,
                   nullptr);
}

// CTAs per sequence at most (one cluster): 8 (a portable cluster), or 16 (a
// non-portable one) when the grid then still fits one CTA per SM -- at most 14
// clusters of 16 are resident at once on GB300, so wide clusters pay only for
// few long sequences (config 5: 10.9 instead of 14.4 us per call).
// ADAPLD_LEXICAL_CLUSTER=<1..16> overrides it for tuning sweeps.
int lexical_cluster_max(int chunks, int B) {
    if (const char *e = std::getenv("ADAPLD_LEXICAL_CLUSTER")) {
        const int v = std::atoi(e);
        if (v >= 1 && v <= 16) return v;
    }
    const int wide = chunks < kWideClusterL ? chunks : kWideClusterL;
    if (chunks > kMaxClusterL && (int64_t)B * wide <= device_sms()) return kWideClusterL;
    return kMaxClusterL;
}

}  // namespace

cudaError_t launch_lexical(const LexLaunch &a, const Workspace &ws, cudaStream_t s) {
    const int chunks = chunks_of(a.ld - 1, kChunkL);
    const int xmax = lexical_cluster_max(chunks, a.B);
    const int X = chunks < xmax ? chunks : xmax;
    const int q = (chunks + X - 1) / X;
    LexArgs args{a, ws, q};
    cudaError_t e = cudaSuccess;
    if (X > 8) {
        e = cudaFuncSetAttribute(lexical_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(X, a.B);
    cfg.blockDim = dim3(kThreadsL);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (X > 1) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = X;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
    }
    return counted(cudaLaunchKernelEx(&cfg, lexical_kernel, args));
}

cudaError_t launch_outcome_plan(const int32_t *lengths, int64_t ld, int32_t B,
                                const int32_t *hit_kind, const Workspace &ws, cudaStream_t s) {
    PlanArgs a{lengths, ld, B, hit_kind, nullptr, 0, nullptr, nullptr, nullptr, ws.plan};
    return launch_dependent(outcome_plan_kernel, dim3(1), dim3(kThreads1), 0, s, a);
}

cudaError_t launch_plan(const int32_t *lengths, int64_t ld, int32_t B, const uint8_t *active,
                        int32_t k, int32_t *cand, float *score, int32_t *n_cand,
                        const Workspace &ws, cudaStream_t s) {
    PlanArgs a{lengths, ld, B, nullptr, active, k, cand, score, n_cand, ws.plan};
    plan_kernel<<<1, kThreads1, 0, s>>>(a);
    return counted(cudaGetLastError());
}

}  // namespace adapld
