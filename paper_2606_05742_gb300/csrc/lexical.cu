// Lexical anchoring (Sec. 3.3, Eq. 3, generalised to the longest suffix
// n-gram) and the semantic work plan.
//
// Grid (C1 chunks, B sequences), 256 threads.  A CTA stages one chunk of
// 4096 candidate positions (plus an n_max-1 token halo) in shared memory,
// computes for each position j the length m(j) of the backward match
// M[j-i] == M[len-1-i], i < m(j) <= min(n_max, len-1), reduces the chunk
// maximum and ranks the positions reaching it, most recent first, with warp
// ballots and one barrier.  A history of one chunk writes its result
// directly; otherwise the last CTA of a sequence (atomic ticket) merges the
// chunk results: n* = max m, candidates = the k most recent positions with
// m(j) = n*.  On the step path the last sequence to finish also writes the
// prefix sums of the semantic fallback's rows (the plan), so the semantic
// kernel can balance rows over the whole GPU without a host round trip.
#include "common.cuh"

namespace adapld {

namespace {

struct LexArgs {
    LexLaunch p;
    Workspace ws;
};

__global__ void __launch_bounds__(kThreads1) lexical_kernel(LexArgs args) {
    const LexLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ int tok[kChunk1 + 8];
    __shared__ int suf[8];
    __shared__ int wval[kThreads1 / 32];
    __shared__ int wcnt[(kChunk1 / kThreads1) * (kThreads1 / 32)];  // hits per (block, warp)
    __shared__ int list[kMaxK];
    __shared__ int flag;

    pdl_wait_then_release();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int b = blockIdx.y, c = blockIdx.x;
    const int len = a.lengths[b];
    const bool valid = len >= 1 && (int64_t)len <= a.ld;
    const int nj = valid ? len - 1 : 0;               // candidates j in [0, len-2]
    const int top = valid ? min(a.n_max, len - 1) : 0;
    const int j0 = c * kChunk1;
    const int j1 = min(j0 + kChunk1, nj);
    const int32_t *M = a.tokens + (int64_t)b * a.ld;

    if (a.stats && b == 0 && c == 0 && t < 4) a.stats[t] = 0;

    int cmax = 0, cnt = 0;
    if (j0 < j1 && top > 0) {
        const int h = top - 1;  // halo before the chunk
        for (int i = t; i < j1 - j0 + h; i += kThreads1) {
            const int p = j0 - h + i;
            tok[i] = p >= 0 ? M[p] : 0;
        }
        if (t < top) suf[t] = M[len - 1 - t];
        __syncthreads();
        int m[kChunk1 / kThreads1];
        int mymax = 0;
#pragma unroll
        for (int e = 0; e < kChunk1 / kThreads1; ++e) {
            const int p = j0 + e * kThreads1 + t;
            int mm = 0;
            if (p < j1) {
                while (mm < top && p - mm >= 0 && tok[p - mm - j0 + h] == suf[mm]) ++mm;
            }
            m[e] = mm;
            mymax = max(mymax, mm);
        }
        mymax = warp_max_i(mymax);
        if (lane == 0) wval[warp] = mymax;
        __syncthreads();
        for (int w = 0; w < kThreads1 / 32; ++w) cmax = max(cmax, wval[w]);
        __syncthreads();
        if (cmax > 0) {
            // most recent first: position blocks e from the top, within a
            // block higher warps and then higher lanes first.  Every
            // (block, warp) count goes to shared memory at once, so one
            // barrier ranks all positions.
            constexpr int E = kChunk1 / kThreads1, NW = kThreads1 / 32;
            unsigned bal[E];
#pragma unroll
            for (int e = 0; e < E; ++e) {
                const int p = j0 + e * kThreads1 + t;
                bal[e] = __ballot_sync(0xffffffffu, p < j1 && m[e] == cmax);
                if (lane == 0) wcnt[e * NW + warp] = __popc(bal[e]);
            }
            __syncthreads();
            // ranks: positions of higher blocks, then of higher warps and
            // lanes in this block, come first
            int before = 0;  // hits in blocks above e (filled from the top)
#pragma unroll
            for (int e = E - 1; e >= 0; --e) {
                int above = 0, all = 0;
#pragma unroll
                for (int w = 0; w < NW; ++w) {
                    const int cw = wcnt[e * NW + w];
                    above += w > warp ? cw : 0;
                    all += cw;
                }
                const unsigned higher = lane == 31 ? 0u : (bal[e] & (0xffffffffu << (lane + 1)));
                const int rank = before + above + __popc(higher);
                if (((bal[e] >> lane) & 1u) && rank < a.k) list[rank] = j0 + e * kThreads1 + t;
                before += all;
            }
            cnt = min(before, a.k);
        }
    }

    __syncthreads();
    if (gridDim.x == 1) {
        // ---- the history is one chunk: its list is the result (no merge)
        if (warp == 0) {
            const int total = cmax > 0 ? cnt : 0;
            if (lane < a.k) a.cand[(int64_t)b * a.k + lane] = lane < total ? list[lane] : -1;
            if (a.score && lane < a.k) a.score[(int64_t)b * a.k + lane] = 0.f;
            if (lane == 0) {
                a.match_n[b] = cmax;
                a.n_cand[b] = total;
                a.hit_kind[b] = cmax > 0 ? ADAPLD_HIT_LEX : ADAPLD_HIT_NONE;
                if (a.status) a.status[b] = valid ? 0 : ADAPLD_SEQ_BAD_LENGTH;
            }
        }
    } else {
        int32_t *part = ws.part1 + ((int64_t)b * ws.C1 + c) * kPart1Ints;
        if (t == 0) {
            part[0] = cmax;
            part[1] = cnt;
        }
        if (t < cnt) part[2 + t] = list[t];
        __threadfence();
        __syncthreads();
        if (t == 0) flag = atomicAdd(ws.ticket1 + b, 1) == (int)gridDim.x - 1;
        __syncthreads();
        if (!flag) return;
        __threadfence();

        // ---- last chunk of sequence b: merge --------------------------------
        if (warp == 0) {
            const int nchunks = (int)gridDim.x;
            const int32_t *pb = ws.part1 + (int64_t)b * ws.C1 * kPart1Ints;
            int best = 0;
            for (int cc = lane; cc < nchunks; cc += 32)
                best = max(best, __ldcg(pb + cc * kPart1Ints));
            best = warp_max_i(best);
            int32_t *cb = a.cand + (int64_t)b * a.k;
            int total = 0;
            if (best > 0) {
                total = warp_merge_desc(
                    nchunks, a.k,
                    [&](int cc) {
                        const int32_t *pp = pb + cc * kPart1Ints;
                        return __ldcg(pp) == best ? __ldcg(pp + 1) : 0;
                    },
                    [&](int cc, int i) { return __ldcg(pb + cc * kPart1Ints + 2 + i); }, cb);
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
    }
    if (!a.build_plan) return;

    // ---- last sequence overall: semantic plan ---------------------------------
    // (a grid of one CTA is last by construction: no ticket)
    if (gridDim.x * gridDim.y > 1) {
        __threadfence();
        __syncthreads();
        if (t == 0) flag = atomicAdd(ws.global_ticket, 1) == a.B - 1;
        __syncthreads();
        if (!flag) return;
        __threadfence();
    } else {
        __syncthreads();  // this CTA's outcome writes are visible to the block
    }
    build_plan_cta(a.lengths, a.ld, a.B, a.hit_kind, nullptr, ws.plan, false, a.k, nullptr,
                   nullptr, nullptr);
}

struct PlanArgs {
    const int32_t *lengths;
    int64_t ld;
    int32_t B;
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

}  // namespace

cudaError_t launch_lexical(const LexLaunch &a, const Workspace &ws, cudaStream_t s) {
    LexArgs args{a, ws};
    dim3 grid(ws.C1, a.B);
    lexical_kernel<<<grid, kThreads1, 0, s>>>(args);
    return cudaGetLastError();
}

cudaError_t launch_plan(const int32_t *lengths, int64_t ld, int32_t B, const uint8_t *active,
                        int32_t k, int32_t *cand, float *score, int32_t *n_cand,
                        const Workspace &ws, cudaStream_t s) {
    PlanArgs a{lengths, ld, B, active, k, cand, score, n_cand, ws.plan};
    plan_kernel<<<1, kThreads1, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace adapld
