// Lexical anchoring (Sec. 3.3, Eq. 3, generalised to the longest suffix
// n-gram).
//
// Grid (X, B), 512 threads; the X CTAs of a sequence form one thread-block
// cluster (X <= 8, or 16 for a few long sequences).  CTA x scans a contiguous range of
// 8192-position chunks, most recent chunk first.  A chunk and its n_max-1
// token halo are staged in shared memory with 16-byte cp.async copies (4-byte
// copies for the unaligned head and tail), the next chunk's copies in flight
// while the current one is scanned.  For each position j the backward match
// length m(j) = #{i : M[j-i'] == M[len-1-i'] for all i' <= i}, capped at
// min(n_max, len-1), is computed: one comparison with the anchor token for
// every position, extended only where it matches.  The chunk maximum and the
// positions reaching it, most recent first, are ranked with warp ballots and
// one scan over (block, warp) cells.  The CTA keeps the best length over its
// chunks and its k most recent positions.  The cluster then merges its CTAs'
// results through distributed shared memory (CTA rank 0 reads them; ranks hold
// contiguous ranges, higher ranks more recent): n* = max m, candidates = the
// k most recent positions with m(j) = n*.  No global ticket, no counters.
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
constexpr int kPerThreadL = kChunkL / kThreadsL;  // positions per thread and chunk (16)
constexpr int kBufL = kChunkL + 16;               // chunk + halo (<= 7) + alignment (<= 3)

struct LexArgs {
    LexLaunch p;
    Workspace ws;
    int q;  // chunks per CTA
};

// Stages tokens M[j0-h .. j1) (indices below 0 are never read and are not
// copied) into buf, global index i at buf[i - (j0-h) + off], where `off`
// makes 16-byte aligned global addresses land on 16-byte aligned slots.
__device__ __forceinline__ int stage_chunk(int *buf, const int32_t *M, int j0, int j1, int h) {
    const int t = threadIdx.x;
    const int b0 = j0 - h;
    const int off = (int)((((uintptr_t)M >> 2) & 3) + b0) & 3;
    const int gs = max(b0, 0);
    int f = gs + ((4 - ((gs - b0 + off) & 3)) & 3);  // first 16-byte boundary >= gs
    int l = j1 - ((j1 - b0 + off) & 3);             // last 16-byte boundary <= j1
    if (f > j1) f = j1;
    if (l < f) l = f;
    const int shift = off - b0;  // buf index of global index i: i + shift
    for (int v = t; v < (l - f) >> 2; v += kThreadsL)
        cp_async16(buf + (f + 4 * v + shift), M + f + 4 * v);
    if (t < f - gs) cp_async4(buf + (gs + t + shift), M + gs + t);
    if (t >= 32 && t - 32 < j1 - l) cp_async4(buf + (l + (t - 32) + shift), M + l + (t - 32));
    return off;
}

__global__ void __launch_bounds__(kThreadsL, 2) lexical_kernel(LexArgs args) {
    const LexLaunch &a = args.p;
    extern __shared__ __align__(16) int dyn[];  // [1 or 2][kBufL] staged chunks
    __shared__ int suf[8];
    __shared__ int wval[kWarpsL];
    __shared__ int wcnt[kPerThreadL * kWarpsL];  // hits per (block, warp)
    __shared__ int wbase[kPerThreadL * kWarpsL]; // hits ranked before each (block, warp)
    __shared__ int clist[kMaxK];                 // this chunk's ranked positions
    __shared__ int res[2 + kMaxK];               // this CTA's result: m, count, positions

    pdl_wait_then_release();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int b = blockIdx.y, x = blockIdx.x, X = gridDim.x;
    const int len = a.lengths[b];
    const bool valid = len >= 1 && (int64_t)len <= a.ld;
    const int nj = valid ? len - 1 : 0;  // candidates j in [0, len-2]
    const int top = valid ? min(a.n_max, len - 1) : 0;
    const int h = top > 0 ? top - 1 : 0;  // halo before a chunk
    const int nchunks = (nj + kChunkL - 1) / kChunkL;
    const int c_lo = x * args.q, c_hi = min(c_lo + args.q, nchunks);
    const int32_t *M = a.tokens + (int64_t)b * a.ld;

    if (a.zero) {  // the later kernels' counters (grid-stride over every thread)
        const size_t nthreads = (size_t)gridDim.x * gridDim.y * kThreadsL;
        for (size_t i = ((size_t)b * X + x) * kThreadsL + t; i < a.zero_words; i += nthreads)
            a.zero[i] = 0;
    }
    if (a.stats && b == 0 && x == 0 && t < 4) a.stats[t] = 0;
    if (t == 0) {
        res[0] = 0;
        res[1] = 0;
    }
    if (t < top) suf[t] = M[len - 1 - t];

    int off = 0;
    if (c_hi > c_lo && top > 0) {
        const int jc = (c_hi - 1) * kChunkL;
        off = stage_chunk(dyn, M, jc, min(jc + kChunkL, nj), h);
        cp_async_commit();
    }
    for (int c = c_hi - 1, i = 0; c >= c_lo && top > 0; --c, ++i) {
        const int j0 = c * kChunkL, j1 = min(j0 + kChunkL, nj);
        const int *tok = dyn + (i & 1) * kBufL;
        const int shift = off - (j0 - h);  // tok[p + shift] = M[p]
        int next_off = 0;
        if (c - 1 >= c_lo) {  // the next (older) chunk's copies fly during this scan
            const int jn = (c - 1) * kChunkL;
            next_off = stage_chunk(dyn + ((i + 1) & 1) * kBufL, M, jn, jn + kChunkL, h);
            cp_async_commit();
            cp_async_wait_group<1>();
        } else {
            cp_async_wait_group<0>();
        }
        __syncthreads();  // the staged chunk and the suffix are visible

        // match lengths (<= 8) of this thread's 16 positions, 4 bits each: one
        // comparison with the anchor token per position, extended backwards
        // only where it matches
        const int s0 = suf[0];
        uint32_t first = 0;
#pragma unroll
        for (int e = 0; e < kPerThreadL; ++e) {
            const int p = j0 + e * kThreadsL + t;
            if (p < j1 && tok[p + shift] == s0) first |= 1u << e;
        }
        uint64_t mpack = 0;
        int mymax = 0;
        for (uint32_t f = first; f; f &= f - 1) {
            const int e = __ffs(f) - 1;
            const int p = j0 + e * kThreadsL + t;
            int mm = 1;
            while (mm < top && p - mm >= 0 && tok[p - mm + shift] == suf[mm]) ++mm;
            mpack |= (uint64_t)mm << (4 * e);
            mymax = max(mymax, mm);
        }
        mymax = warp_max_i(mymax);
        if (lane == 0) wval[warp] = mymax;
        __syncthreads();
        int cmax = 0;
#pragma unroll
        for (int w = 0; w < kWarpsL; ++w) cmax = max(cmax, wval[w]);
        int ccnt = 0;
        if (cmax > 0) {
            uint32_t hits = 0;
            for (uint32_t f = first; f; f &= f - 1) {
                const int e = __ffs(f) - 1;
                if ((int)((mpack >> (4 * e)) & 15u) == cmax) hits |= 1u << e;
            }
            auto hit = [&](int e) { return ((hits >> e) & 1u) != 0; };
            // most recent first: position blocks e from the top, within a
            // block higher warps and then higher lanes first.  The hits per
            // (block, warp) are counted, scanned once in that order, and each
            // hit's rank is its (block, warp) offset plus the hits of the
            // higher lanes of its warp.
#pragma unroll
            for (int e = 0; e < kPerThreadL; ++e) {
                const unsigned bal = __ballot_sync(0xffffffffu, hit(e));
                if (lane == 0) wcnt[e * kWarpsL + warp] = __popc(bal);
            }
            __syncthreads();
            constexpr int kCells = kPerThreadL * kWarpsL;  // 256 (block, warp) cells
            static_assert(kCells <= kThreadsL && kCells % 32 == 0, "one cell per thread");
            int v = 0, cell = 0;
            if (t < kCells) {
                const int e = kPerThreadL - 1 - t / kWarpsL, w = kWarpsL - 1 - t % kWarpsL;
                cell = e * kWarpsL + w;
                v = wcnt[cell];
            }
            int incl = v;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += u;
            }
            if (t < kCells && lane == 31) wval[warp] = incl;  // (cmax is already read)
            __syncthreads();
            int before = 0, total = 0;
#pragma unroll
            for (int w = 0; w < kCells / 32; ++w) {
                const int x = wval[w];
                before += w < warp ? x : 0;
                total += x;
            }
            if (t < kCells) wbase[cell] = before + incl - v;
            __syncthreads();
#pragma unroll
            for (int e = 0; e < kPerThreadL; ++e) {
                const bool mine = hit(e);
                const unsigned bal = __ballot_sync(0xffffffffu, mine);
                const unsigned higher = lane == 31 ? 0u : (bal & (0xffffffffu << (lane + 1)));
                const int rank = wbase[e * kWarpsL + warp] + __popc(higher);
                if (mine && rank < a.k) clist[rank] = j0 + e * kThreadsL + t;
            }
            ccnt = min(total, a.k);
        }
        __syncthreads();  // clist complete
        // fold the chunk into the CTA's result (chunks arrive most recent first)
        if (warp == 0 && cmax > 0) {
            const int rm = res[0], rn = res[1];
            __syncwarp();
            if (cmax > rm) {
                if (lane < ccnt) res[2 + lane] = clist[lane];
                if (lane == 0) {
                    res[0] = cmax;
                    res[1] = ccnt;
                }
            } else if (cmax == rm) {
                const int add = min(ccnt, a.k - rn);
                if (lane < add) res[2 + rn + lane] = clist[lane];
                if (lane == 0) res[1] = rn + add;
            }
        }
        __syncthreads();  // before the buffers, wval, wcnt and clist are reused
        off = next_off;
    }

    // ---- the sequence's result: CTA rank 0 merges the cluster's CTAs ---------
    int32_t *cb = a.cand + (int64_t)b * a.k;
    if (X == 1) {
        __syncthreads();
        if (warp == 0) {
            const int best = res[0];
            const int total = best > 0 ? res[1] : 0;
            if (lane < a.k) cb[lane] = lane < total ? res[2 + lane] : -1;
            if (a.score && lane < a.k) a.score[(int64_t)b * a.k + lane] = 0.f;
            if (lane == 0) {
                a.match_n[b] = best;
                a.n_cand[b] = total;
                a.hit_kind[b] = best > 0 ? ADAPLD_HIT_LEX : ADAPLD_HIT_NONE;
                if (a.status) a.status[b] = valid ? 0 : ADAPLD_SEQ_BAD_LENGTH;
            }
        }
    } else {
        // every CTA's result is in its shared memory (warp 0 wrote it)
        if (warp == 0)
            cluster_sync_all();
        else
            cluster_sync_relaxed();
        if (x == 0 && warp == 0) {
            int best = lane < X ? ld_cluster_i32(&res[0], lane) : 0;
            best = warp_max_i(best);
            int total = 0;
            if (best > 0) {
                total = warp_merge_desc(
                    X, a.k,
                    [&](int r) {
                        return ld_cluster_i32(&res[0], r) == best ? ld_cluster_i32(&res[1], r)
                                                                  : 0;
                    },
                    [&](int r, int i) { return ld_cluster_i32(&res[2 + i], r); }, cb);
            }
            if (lane >= total && lane < a.k) cb[lane] = -1;
            if (a.score && lane < a.k) a.score[(int64_t)b * a.k + lane] = 0.f;
            if (lane == 0) {
                a.match_n[b] = best;
                a.n_cand[b] = total;
                a.hit_kind[b] = best > 0 ? ADAPLD_HIT_LEX : ADAPLD_HIT_NONE;
                if (a.status) a.status[b] = valid ? 0 : ADAPLD_SEQ_BAD_LENGTH;
            }
        }
        cluster_sync_relaxed();  // the CTAs' shared memory stays until rank 0 has read it
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
    const size_t smem = sizeof(int) * (size_t)kBufL * (q > 1 ? 2 : 1);
    cudaError_t e = cudaFuncSetAttribute(lexical_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (X > 8) {
        e = cudaFuncSetAttribute(lexical_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(X, a.B);
    cfg.blockDim = dim3(kThreadsL);
    cfg.dynamicSmemBytes = smem;
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
    return cudaLaunchKernelEx(&cfg, lexical_kernel, args);
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
    return cudaGetLastError();
}

}  // namespace adapld
