// Rerank and draft-tree construction (Sec. 3.4-3.6, Eq. 6-15, Algorithm 1).
//
// With at most 16 successor rows per sequence (W*k <= 16) the stage is one
// kernel: succ_scan_kernel<U, true>, where the CTA that completes a
// sequence's scan (or CTA 0 of a sequence without successors) goes on to
// build its tree (tree_body, every row in that CTA, one per warp).
// With more rows, or in two-representation mode (the successor backoff runs
// in between), it is two kernels so that every gathered row is read by its
// own warp somewhere on the GPU instead of queueing behind one CTA:
//
// succ_scan_kernel, grid (S4 slices, B), 512 threads -- only for sequences
// that draft successors (Algorithm 1: semantic hits; every hit under
// ADAPLD_SUCC_ON_STRICT).  Each CTA rebuilds the anchor and the branch set
// (lexical hits are reranked here in that mode), then scans its slice of
// 8192 positions for the branch tokens, a warp per branch, backwards with
// ballots, keeping the k most recent occurrences.  The last slice CTA
// (atomic ticket; none with one slice) merges the slices, most recent first,
// into the successor candidate lists.
//
// tree_kernel, grid (R5, B), 512 threads.  Every sequence has a list of rows
// to score: the lexical candidates against the query (Eq. 6), or every
// successor candidate against R[j*+1] (Eq. 13).  CTA r scores rows
// [16r, 16r+16), one warp per row against the reference vector staged once
// per CTA in shared memory, with 16 (or 8) 16-byte row loads per lane in
// flight.  The last CTA of the sequence
// then ranks the lexical candidates (Eq. 7), picks each branch's successor
// (Eq. 14), lays out the tree (root, main chain, branch paths with their
// successors) and writes tokens, parents, position ids and the ancestor mask.
#include "common.cuh"

namespace adapld {

namespace {

constexpr int kRowsPerCta5 = kThreads4 / 32;  // one warp per scored row

struct TreeArgs {
    TreeLaunch p;
    Workspace ws;
    int rows_ctas;  // gridDim.x of tree_kernel
};

// Shared state of the tree stage (the candidates, the branch set and the
// node layout of one sequence).
struct TreeSmem {
    int cand[kMaxK];
    float score[kMaxK];
    int next[kMaxW];
    int br[kMaxW];
    int succ[kMaxW];
    int misc[4];
    int node_par[kMaxNodes];
    short node_depth[kMaxNodes];
    short node_path[kMaxNodes];
    int node_src[kMaxNodes];
    float red[32];
};

// <row, ref> and |row|^2 of one bf16 row in global memory against an fp32
// vector in shared memory (one warp, U independent 16-byte loads per lane in
// flight).  A lane sums its chunks lane, lane + 32, ... in the same order
// whatever U, so the result does not depend on U.
template <int U = 16>
__device__ __forceinline__ void warp_row_dot(const uint16_t *row, const float *ref, int d,
                                             float &dot_out, float &ss_out) {
    const int lane = threadIdx.x & 31;
    const int nch = d >> 3;
    float dot = 0.f, ss = 0.f;
    for (int base = 0; base < nch; base += 32 * U) {
        uint4 w[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int ch = base + u * 32 + lane;
            w[u] = ch < nch ? ldg_nc_v4(row + (size_t)ch * 8) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int ch = base + u * 32 + lane;
            if (ch < nch) {
                const float4 r0 = *(const float4 *)(ref + ch * 8);
                const float4 r1 = *(const float4 *)(ref + ch * 8 + 4);
                const float x0 = bf16lo(w[u].x), x1 = bf16hi(w[u].x);
                const float x2 = bf16lo(w[u].y), x3 = bf16hi(w[u].y);
                const float x4 = bf16lo(w[u].z), x5 = bf16hi(w[u].z);
                const float x6 = bf16lo(w[u].w), x7 = bf16hi(w[u].w);
                dot = fmaf(x0, r0.x, dot);
                dot = fmaf(x1, r0.y, dot);
                dot = fmaf(x2, r0.z, dot);
                dot = fmaf(x3, r0.w, dot);
                dot = fmaf(x4, r1.x, dot);
                dot = fmaf(x5, r1.y, dot);
                dot = fmaf(x6, r1.z, dot);
                dot = fmaf(x7, r1.w, dot);
                ss = fmaf(x0, x0, ss);
                ss = fmaf(x1, x1, ss);
                ss = fmaf(x2, x2, ss);
                ss = fmaf(x3, x3, ss);
                ss = fmaf(x4, x4, ss);
                ss = fmaf(x5, x5, ss);
                ss = fmaf(x6, x6, ss);
                ss = fmaf(x7, x7, ss);
            }
        }
    }
    dot_out = warp_sum(dot);
    ss_out = warp_sum(ss);
}

// Loads a bf16 vector into shared memory as fp32 and returns its squared
// norm (block-wide; every thread gets the same value).
__device__ float block_load_vec(const uint16_t *v, float *dst, int d, float *scratch) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float part = 0.f;
    for (int ch = threadIdx.x; ch < (d >> 3); ch += blockDim.x) {
        const uint4 w = ldg_nc_v4(v + (size_t)ch * 8);
        const float x[8] = {bf16lo(w.x), bf16hi(w.x), bf16lo(w.y), bf16hi(w.y),
                            bf16lo(w.z), bf16hi(w.z), bf16lo(w.w), bf16hi(w.w)};
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            dst[ch * 8 + e] = x[e];
            part = fmaf(x[e], x[e], part);
        }
    }
    part = warp_sum(part);
    if (lane == 0) scratch[warp] = part;
    __syncthreads();
    float tot = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += scratch[w];
    __syncthreads();
    return tot;
}

// Per-sequence facts every kernel of the tree stage derives the same way.
struct SeqView {
    int len;
    bool valid, cand_ok, lex, sem, branch_on, need_succ;
    bool rr;  // the candidates are (re)ranked by Eq. 6 in this stage
    int nc;
    int cand_t;      // this thread's candidate cand[b][t] (t < k) and its score
    float score_t;
};

// Block-wide (every thread must call, before any early exit).
__device__ __forceinline__ SeqView view_of(const TreeLaunch &a, int b) {
    SeqView v;
    const int k = a.p.k, W = a.p.branch_width, t = threadIdx.x;
    const uint32_t flags = a.p.flags;
    // independent loads first (one memory round trip), then the checks
    v.len = a.lengths[b];
    const int nc_raw = a.n_cand[b];
    const int hk_raw = a.hit_kind[b];
    const int c = t < k ? a.cand[(int64_t)b * k + t] : 0;
    v.score_t = t < k ? a.score[(int64_t)b * k + t] : 0.f;
    v.cand_t = c;
    v.valid = v.len >= 1 && (int64_t)v.len <= a.ld;
    // candidates come from the caller on the standalone path: check the range
    const int nc0 = v.valid ? min(nc_raw, k) : 0;
    const bool ok = t >= nc0 || (c >= 0 && c <= v.len - 2);
    v.cand_ok = __syncthreads_and(ok) != 0;
    const int hk = (v.valid && v.cand_ok) ? hk_raw : ADAPLD_HIT_NONE;
    v.nc = v.cand_ok ? max(nc0, 0) : 0;
    v.lex = hk == ADAPLD_HIT_LEX && v.nc > 0;
    v.sem = hk == ADAPLD_HIT_SEM && v.nc > 0;
    v.branch_on = !(flags & ADAPLD_NO_BRANCH) && W > 0 && (v.lex || v.sem);
    v.need_succ = v.branch_on && !(flags & ADAPLD_NO_SUCC) &&
                  (v.sem || (v.lex && (flags & ADAPLD_SUCC_ON_STRICT)));
    // lexical hits are reranked unless switched off; semantic hits only in
    // the two-representation mode (otherwise their retrieval scores already
    // are the rerank scores)
    v.rr = (v.lex && !(flags & ADAPLD_NO_LEX_RERANK)) || (v.sem && a.emb.table != nullptr);
    return v;
}

// Branch set (Eq. 10-11) into s_br, count returned; s_cand holds the ranked
// candidates (s_cand[0] = j*).  Block-wide: every thread must call.
__device__ __forceinline__ int branch_set(const TreeLaunch &a, int b, const SeqView &v,
                                          const int *s_cand,
                          int *s_next, int *s_br, int *s_misc) {
    const int t = threadIdx.x, W = a.p.branch_width;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const int js = s_cand[0];
    if (a.next_topk) {
        const int32_t *row = a.next_topk + ((int64_t)b * a.ld + js) * a.Kn;
        if (t < a.Kn) s_next[t] = row[t];
    } else if (t < v.nc) {
        s_next[t] = M[s_cand[t] + 1];
    }
    if (t == kThreads4 - 1) s_misc[0] = v.lex ? M[js + 1] : -1;
    __syncthreads();
    if (t == 0) {
        int nb = 0;
        if (a.next_topk) {
            for (int r = 0; r < a.Kn && nb < W; ++r)
                if (s_next[r] >= 0) s_br[nb++] = s_next[r];
        } else {
            for (int r = 0; r < v.nc && nb < W; ++r) {
                const int tkn = s_next[r];
                bool dup = false;
                for (int e = 0; e < nb; ++e) dup |= s_br[e] == tkn;
                if (!dup) s_br[nb++] = tkn;
            }
        }
        if (v.lex) {  // Eq. 11
            int m = 0;
            for (int e = 0; e < nb; ++e)
                if (s_br[e] != s_misc[0]) s_br[m++] = s_br[e];
            nb = m;
        }
        s_misc[1] = nb;
    }
    __syncthreads();
    return s_misc[1];
}

// Warp 0 sorts n <= 32 (score, position) pairs in place by (score desc,
// position desc).
__device__ __forceinline__ void warp_sort_desc(int *s_cand, float *s_score, int n) {
    const int lane = threadIdx.x & 31;
    const float sc = lane < n ? s_score[lane] : -INFINITY;
    const int cj = lane < n ? s_cand[lane] : -1;
    int rank = 0;
    for (int m = 0; m < n; ++m) {
        const float os = __shfl_sync(0xffffffffu, sc, m);
        const int oj = __shfl_sync(0xffffffffu, cj, m);
        rank += better(os, oj, sc, cj) ? 1 : 0;
    }
    __syncwarp();
    if (lane < n) {
        s_cand[rank] = cj;
        s_score[rank] = sc;
    }
    __syncwarp();
}

// ---------------------------------------------------------------------------
// Publishes the successor-candidate count of branch w of sequence b.  A
// branch token that never occurs earlier backs off (Sec. 3.5) to the
// embedding fallback with the branch token as the anchor: with a table, the
// (sequence, branch) pair is registered for the gathered pass.
__device__ __forceinline__ void register_successors(const TreeLaunch &a, const Workspace &ws,
                                                    int b, int w, int total, int token) {
    ws.succ_n[(int64_t)b * ws.W + w] = total;
    if (total == 0 && a.emb.table) {
        const int idx = atomicAdd(ws.npairs, 1);
        ws.pair_b[idx] = b;
        ws.pair_tok[idx] = token;
        ws.pair_out[idx] = b * ws.W + w;
    }
}

template <int U>
__device__ void tree_body(const TreeLaunch &a, const Workspace &ws, int b, const SeqView &v,
                          int r5, bool fused, TreeSmem &sm, float *s_ref);

// FUSED: the CTA that completes a sequence's scan (or CTA 0 of a sequence
// without successors) then builds that sequence's tree itself (tree_body,
// all scored rows in this CTA), so the tree stage is one kernel.  U: row
// loads in flight in tree_body.
template <int U, bool FUSED>
__global__ void __launch_bounds__(kThreads4, U == 8 ? 2 : 1) succ_scan_kernel(TreeArgs args) {
    const TreeLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ int s_tok[kSlice4];
    __shared__ TreeSmem sm;
    int *s_cand = sm.cand;
    float *s_score = sm.score;
    int *s_next = sm.next;
    int *s_br = sm.br;
    int *s_misc = sm.misc;
    float *s_red = sm.red;
    extern __shared__ __align__(16) float s_q[];  // [d] the query (fp32) for a rerank here

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nwarps = kThreads4 / 32;
    const int b = blockIdx.y, sl = blockIdx.x;
    const int k = a.p.k, d = a.d;
    pdl_wait_then_release();
    const SeqView v = view_of(a, b);
    if (!v.need_succ) {
        if (FUSED && sl == 0) tree_body<U>(a, ws, b, v, 0, true, sm, s_q);
        return;
    }
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const uint16_t *R = a.reps + (int64_t)b * a.ld * d;

    if (t < v.nc) {
        s_cand[t] = v.cand_t;
        s_score[t] = v.score_t;
    }
    __syncthreads();
    if (v.rr) {  // the ranking the branches depend on (each slice alike; the
                 // arithmetic of the tree kernel's rerank, so the scores agree)
        const float qss = block_load_vec(a.query + (int64_t)b * d, s_q, d, s_red);
        for (int ci = warp; ci < v.nc; ci += nwarps) {
            float dot, ss;
            warp_row_dot<8>(R + (int64_t)s_cand[ci] * d, s_q, d, dot, ss);
            if (lane == 0) s_score[ci] = cosine_from(dot, ss, qss);
        }
        __syncthreads();
        if (warp == 0) warp_sort_desc(s_cand, s_score, v.nc);
        __syncthreads();
    } else if (v.lex) {
        if (t < v.nc) s_score[t] = __int_as_float(0x7fc00000);  // NaN: not computed
        __syncthreads();
    }
    const int nb = branch_set(a, b, v, s_cand, s_next, s_br, s_misc);

    const int p0 = sl * kSlice4;
    const int p1 = min(p0 + kSlice4, v.len - 1);  // positions t <= len-2
    for (int i = t; i < p1 - p0; i += kThreads4) s_tok[i] = M[p0 + i];
    __syncthreads();
    constexpr int G = 8;  // 32-position groups tested per pass (independent loads)
    // one slice: its lists are the merged result, written in place (no merge)
    const bool single = gridDim.x == 1;
    for (int w = warp; w < nb; w += nwarps) {
        const int bt = s_br[w];
        int32_t *part =
            single ? nullptr : ws.part4 + (((int64_t)b * ws.S4 + sl) * ws.W + w) * kPart4Ints;
        int32_t *lst = single ? ws.succ + ((int64_t)b * ws.W + w) * kMaxK : part + 1;
        int cnt = 0;
        for (int top = p1 - 1; top >= p0 && cnt < k; top -= 32 * G) {
            unsigned m[G];
#pragma unroll
            for (int u = 0; u < G; ++u) {
                const int p = top - 32 * u - lane;
                m[u] = __ballot_sync(0xffffffffu, p >= p0 && s_tok[p - p0] == bt);
            }
#pragma unroll
            for (int u = 0; u < G; ++u) {
                const int p = top - 32 * u - lane;
                const int rank = cnt + __popc(m[u] & ((1u << lane) - 1u));
                if (((m[u] >> lane) & 1u) && rank < k) lst[rank] = p;
                cnt += __popc(m[u]);
            }
        }
        if (lane == 0) {
            if (single)
                register_successors(a, ws, b, w, min(cnt, k), s_br[w]);
            else
                part[0] = min(cnt, k);
        }
    }
    if (!single) {
        __threadfence();
        __syncthreads();
        if (t == 0) s_misc[2] = atomicAdd(ws.ticket4 + b, 1) == (int)gridDim.x - 1;
        __syncthreads();
        if (!s_misc[2]) return;
        __threadfence();
        // last slice: merge, most recent first
        for (int w = warp; w < nb; w += nwarps) {
            const int32_t *pw = ws.part4 + ((int64_t)b * ws.S4 * ws.W + w) * kPart4Ints;
            const int64_t stride = (int64_t)ws.W * kPart4Ints;  // next slice, same branch
            const int total = warp_merge_desc(
                (int)gridDim.x, k, [&](int s2) { return __ldcg(pw + s2 * stride); },
                [&](int s2, int i) { return __ldcg(pw + s2 * stride + 1 + i); },
                ws.succ + ((int64_t)b * ws.W + w) * kMaxK);
            if (lane == 0) register_successors(a, ws, b, w, total, s_br[w]);
        }
    }
    if ((v.lex || v.rr) && t < v.nc) {
        ws.rr_cand[(int64_t)b * kMaxK + t] = s_cand[t];
        ws.rr_score[(int64_t)b * kMaxK + t] = s_score[t];
    }
    if (FUSED) {
        __syncthreads();  // the lists and the ranking above are visible to the block
        tree_body<U>(a, ws, b, v, 0, true, sm, s_q);
    }
}

// The plan of the successor backoff pass: row prefix sums over the
// (sequence, branch) pairs registered by succ_scan_kernel (one CTA).
__global__ void __launch_bounds__(256) backoff_plan_kernel(TreeArgs args) {
    const TreeLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ int64_t scratch[8];
    pdl_wait_then_release();
    const int n = *ws.npairs;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int64_t carry = 0;
    for (int base = 0; base < n; base += 256) {
        const int p = base + threadIdx.x;
        int64_t rows = 0;
        if (p < n) {  // the pair scores its sequence's distinct tokens
            const int len = __ldcg(ws.rep_len + ws.pair_b[p]);
            rows = len >= 2 ? len - 1 : 0;
        }
        int64_t incl = rows;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t u = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += u;
        }
        if (lane == 31) scratch[warp] = incl;
        __syncthreads();
        int64_t before = 0, all = 0;
        for (int w = 0; w < 8; ++w) {
            if (w < warp) before += scratch[w];
            all += scratch[w];
        }
        if (p < n) ws.plan3[p] = carry + before + incl - rows;
        carry += all;
        __syncthreads();
    }
    if (threadIdx.x == 0) ws.plan3[n] = carry;
}

// ---------------------------------------------------------------------------
// The tree stage of sequence b for one CTA (all threads): CTA r5 of the
// sequence scores its share of rows (every row when `fused`); the CTA that
// completes the sequence ranks, picks successors and emits the tree.  s_ref:
// d floats of shared memory.
template <int U>
__device__ void tree_body(const TreeLaunch &a, const Workspace &ws, int b, const SeqView &v,
                          int r5, bool fused, TreeSmem &sm, float *s_ref) {
    int *s_cand = sm.cand;
    float *s_score = sm.score;
    int *s_next = sm.next;
    int *s_br = sm.br;
    int *s_succ = sm.succ;
    int *s_misc = sm.misc;
    int *node_par = sm.node_par;
    short *node_depth = sm.node_depth;
    short *node_path = sm.node_path;
    int *node_src = sm.node_src;
    float *s_red = sm.red;

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nwarps = kThreads4 / 32;
    const int k = a.p.k, d = a.d, W = a.p.branch_width, D = a.p.draft_len;
    const int succ_len = a.p.succ_len;
    const uint32_t flags = a.p.flags;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const uint16_t *R = a.reps + (int64_t)b * a.ld * d;
    // the status word is rewritten at the end; its token bit comes from
    // earlier kernels, so it is read now, off the tail's critical path
    const int status0 = (a.status && t == 0) ? a.status[b] : 0;

    // ---- ranked candidates (the successor scan reranked a strict hit already)
    if (t < v.nc) {
        if (v.need_succ && (v.lex || v.rr)) {
            s_cand[t] = __ldcg(ws.rr_cand + (int64_t)b * kMaxK + t);
            s_score[t] = __ldcg(ws.rr_score + (int64_t)b * kMaxK + t);
        } else {
            s_cand[t] = v.cand_t;
            s_score[t] = v.score_t;
        }
    }
    __syncthreads();
    // with successors the ranking is final here, so the branch set is known
    int nb = v.need_succ ? branch_set(a, b, v, s_cand, s_next, s_br, s_misc) : 0;

    // the rows this sequence scores, and the CTAs that share them: lexical
    // candidates against the query, or successor candidate (w, i) at w*k + i
    const bool rerank = v.rr && !v.need_succ;
    const int ntasks = v.need_succ ? nb * k : (rerank ? v.nc : 0);
    const int nctas = fused ? 1 : max(1, (ntasks + kRowsPerCta5 - 1) / kRowsPerCta5);
    if (r5 >= nctas) return;
    const int js0 = (v.lex || v.sem) ? s_cand[0] : -1;
    float *score5 = ws.score5 + (int64_t)b * ws.W * kMaxK;

    // ---- this CTA's share of the scored rows
    if (ntasks > 0) {
        // this CTA's tasks: 16 (one per warp), or all of them when fused
        const int task0 = fused ? 0 : r5 * kRowsPerCta5;
        const int task1 = fused ? ntasks : min(ntasks, task0 + kRowsPerCta5);
        const uint16_t *ref = v.need_succ ? R + (int64_t)(js0 + 1) * d : a.query + (int64_t)b * d;
        const float rss = block_load_vec(ref, s_ref, d, s_red);  // syncs the block
        for (int task = task0 + warp; task < task1; task += nwarps) {
            int row;
            if (v.need_succ) {
                const int w = task / k, i = task % k;
                const int n = __ldcg(ws.succ_n + (int64_t)b * ws.W + w);
                const int pos = __ldcg(ws.succ + ((int64_t)b * ws.W + w) * kMaxK + i);
                row = i < n ? pos : -1;
            } else {
                row = s_cand[task];
            }
            if (row >= 0) {
                float dot, ss;
                warp_row_dot<U>(R + (int64_t)row * d, s_ref, d, dot, ss);
                if (lane == 0) score5[task] = cosine_from(dot, ss, rss);
            }
        }
        if (nctas > 1) {
            __threadfence();
            __syncthreads();
            if (t == 0) s_misc[2] = atomicAdd(ws.ticket5 + b, 1) == nctas - 1;
            __syncthreads();
            if (!s_misc[2]) return;
            __threadfence();
        } else {
            __syncthreads();
        }
    }

    // ---- the last CTA of the sequence: rank, branch, pick successors, emit
    if (rerank) {
        if (warp == 0) {
            if (lane < v.nc) s_score[lane] = __ldcg(score5 + lane);
            __syncwarp();
            warp_sort_desc(s_cand, s_score, v.nc);
        }
        __syncthreads();
    } else if (v.lex && (flags & ADAPLD_NO_LEX_RERANK)) {
        if (t < v.nc) s_score[t] = __int_as_float(0x7fc00000);  // NaN: not computed
        __syncthreads();
    }
    const int js = (v.lex || v.sem) ? s_cand[0] : -1;
    if (v.branch_on && !v.need_succ) nb = branch_set(a, b, v, s_cand, s_next, s_br, s_misc);
    if (v.need_succ) {
        for (int w = warp; w < nb; w += nwarps) {  // Eq. 14: argmax per branch
            // all three loads at once (lanes past the count are masked after)
            const int n = __ldcg(ws.succ_n + (int64_t)b * ws.W + w);
            const float sl = __ldcg(score5 + w * k + lane);
            const int pl = __ldcg(ws.succ + ((int64_t)b * ws.W + w) * kMaxK + lane);
            float bs = lane < n ? sl : -INFINITY;
            int bj = lane < n ? pl : -1;
#pragma unroll
            for (int o = 16; o; o >>= 1) {
                const float os = __shfl_xor_sync(0xffffffffu, bs, o);
                const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
                if (better(os, oj, bs, bj)) {
                    bs = os;
                    bj = oj;
                }
            }
            if (lane == 0) s_succ[w] = n > 0 ? bj : -1;
        }
        __syncthreads();
    }

    const int N = 1 + D + W * (1 + succ_len);
    if (t == 0) {
        int n = 0, ext = 0;
        if (v.valid) {
            node_par[0] = -1;
            node_depth[0] = 0;
            node_path[0] = 0;
            node_src[0] = v.len - 1;
            n = 1;
            if (v.lex) {
                const int l = min(D, v.len - 1 - js);
                for (int i = 0; i < l; ++i, ++n) {
                    node_par[n] = i == 0 ? 0 : n - 1;
                    node_depth[n] = (short)(i + 1);
                    node_path[n] = 1;
                    node_src[n] = js + 1 + i;
                }
            }
            for (int w = 0; w < nb; ++w) {
                node_par[n] = 0;
                node_depth[n] = 1;
                node_path[n] = (short)(2 + w);
                node_src[n] = -2 - w;  // the branch token itself
                ++n;
                if (v.need_succ && s_succ[w] >= 0) {
                    const int tb = s_succ[w];
                    int added = 0;
                    for (int i = 1; i <= succ_len && tb + i <= v.len - 1; ++i, ++n, ++added) {
                        node_par[n] = n - 1;
                        node_depth[n] = (short)(1 + i);
                        node_path[n] = (short)(2 + w);
                        node_src[n] = tb + i;
                    }
                    if (added > 0) ++ext;
                }
            }
        }
        s_misc[0] = n;
        s_misc[3] = ext;
    }
    __syncthreads();
    const int n = s_misc[0];
    const int64_t ob = (int64_t)b * N;
    for (int i = t; i < N; i += kThreads4) {
        int tok = -1, par = -1, pos = -1;
        if (i < n) {
            const int src = node_src[i];
            tok = src >= 0 ? M[src] : s_br[-2 - src];
            par = node_par[i];
            pos = v.len - 1 + node_depth[i];
        }
        a.out.draft_tokens[ob + i] = tok;
        a.out.parents[ob + i] = par;
        a.out.positions[ob + i] = pos;
    }
    uint8_t *mk = a.out.mask + (int64_t)b * N * N;
    for (int idx = t; idx < N * N; idx += kThreads4) {
        const int i = idx / N, j = idx % N;
        const bool anc = i < n && j < n &&
                         (j == i || j == 0 ||
                          (node_path[i] == node_path[j] && j <= i && node_path[i] != 0));
        mk[idx] = anc ? 1 : 0;
    }
    if ((v.lex || v.rr) && t < k) {
        a.cand[(int64_t)b * k + t] = t < v.nc ? s_cand[t] : -1;
        a.score[(int64_t)b * k + t] = t < v.nc ? s_score[t] : 0.f;
    }
    if (t == 0) {
        a.out.anchor[b] = js;
        a.out.n_nodes[b] = n;
        if (a.out.stats) {
            atomicAdd(a.out.stats + (v.lex ? 0 : (v.sem ? 1 : 2)), 1);
            if (s_misc[3]) atomicAdd(a.out.stats + 3, s_misc[3]);
        }
        if (a.status)  // the embedding fallback may have flagged a token id
            a.status[b] = (status0 & ADAPLD_SEQ_BAD_TOKEN) |
                          (v.valid ? 0 : ADAPLD_SEQ_BAD_LENGTH) |
                          (v.cand_ok ? 0 : ADAPLD_SEQ_BAD_CANDIDATE);
    }
}

// U: row loads in flight per lane.  U = 16 (one CTA per SM by registers)
// when the grid fits one wave, U = 8 (two CTAs per SM) otherwise; the
// scores are the same either way (see warp_row_dot).
template <int U>
__global__ void __launch_bounds__(kThreads4, U == 8 ? 2 : 1) tree_kernel(TreeArgs args) {
    __shared__ TreeSmem sm;
    extern __shared__ __align__(16) float s_ref[];  // [d] reference vector (fp32)
    pdl_wait_then_release();
    const SeqView v = view_of(args.p, blockIdx.y);
    tree_body<U>(args.p, args.ws, blockIdx.y, v, blockIdx.x, false, sm, s_ref);
}

}  // namespace

// Successor rows per sequence up to which the fused kernel scores them in the
// CTA that completes the scan (one row per warp, as a tree-kernel CTA would)
// instead of a tree kernel spreading them over CTAs.  Measured on GB300: with
// 16 rows (configs 1 and 4) fusing saves 2.4-2.7 us per step; with 24 or 64
// rows (configs 2 and 3) the second kernel's parallel rows win by 4-14 us.
constexpr int kMaxFusedTasks = kRowsPerCta5;

cudaError_t launch_tree(const TreeLaunch &a, const Workspace &ws, cudaStream_t s) {
    const int W = a.p.branch_width, k = a.p.k;
    const bool succ_possible =
        W > 0 && !(a.p.flags & (ADAPLD_NO_SUCC | ADAPLD_NO_BRANCH));
    const int tasks = succ_possible ? (W * k > k ? W * k : k) : k;
    TreeArgs args{a, ws, (tasks + kRowsPerCta5 - 1) / kRowsPerCta5};
    int sms = 0, dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return cudaErrorInvalidDevice;
    const size_t vsmem = (size_t)a.d * sizeof(float);  // the staged query / reference row
    if (succ_possible) {
        cudaError_t e;
        if (!a.emb.table && W * k <= kMaxFusedTasks) {  // scan and tree in one kernel
            auto kern = (int64_t)ws.S4 * a.B <= sms ? succ_scan_kernel<16, true>
                                                    : succ_scan_kernel<8, true>;
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)vsmem);
            if (e != cudaSuccess) return e;
            return launch_dependent(kern, dim3(ws.S4, a.B), dim3(kThreads4), vsmem, s, args);
        }
        if (a.emb.table && !a.lists_ready) {  // distinct-token lists for the backoff
            DedupeLaunch da{a.tokens, a.ld,  a.lengths, a.B,     a.emb.vocab, nullptr, nullptr,
                            a.status, true, false,     nullptr, false,       k,       nullptr,
                            nullptr,  nullptr};
            e = launch_dedupe(da, ws, s);
            if (e != cudaSuccess) return e;
        }
        e = cudaFuncSetAttribute(succ_scan_kernel<8, false>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)vsmem);
        if (e != cudaSuccess) return e;
        e = launch_dependent(succ_scan_kernel<8, false>, dim3(ws.S4, a.B), dim3(kThreads4), vsmem,
                             s, args);
        if (e != cudaSuccess) return e;
        if (a.emb.table) {  // successor backoff over token embeddings
            e = launch_dependent(backoff_plan_kernel, dim3(1), dim3(256), 0, s, args);
            if (e != cudaSuccess) return e;
            SemLaunch sl{a.emb.table, a.ld, a.emb.dim, nullptr, ws.rep_len, nullptr, a.B, k,
                         a.p.tau, ws.succ, ws.succ_es, ws.succ_n, nullptr, true};
            sl.tokens = ws.rep_tok;
            sl.vocab = a.emb.vocab;
            sl.vseq_b = ws.pair_b;
            sl.vseq_tok = ws.pair_tok;
            sl.vseq_out = ws.pair_out;
            sl.nvseq = ws.npairs;
            sl.out_stride = kMaxK;
            sl.status = a.status;
            e = launch_semantic(sl, ws, s);
            if (e != cudaSuccess) return e;
            // the best distinct tokens back to their k most recent positions
            ExpandLaunch ea{a.tokens, a.ld,     a.lengths, a.emb.vocab, a.B * ws.W, ws.npairs,
                            ws.pair_b, ws.pair_out, ws.succ,  ws.succ_es,  ws.succ_n, kMaxK,
                            k,         nullptr,     nullptr,  ws.xticket2};
            e = launch_expand(ea, ws, s);
            if (e != cudaSuccess) return e;
        }
    }
    auto kern = (int64_t)args.rows_ctas * a.B <= sms ? tree_kernel<16> : tree_kernel<8>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)vsmem);
    if (e != cudaSuccess) return e;
    return launch_dependent(kern, dim3(args.rows_ctas, a.B), dim3(kThreads4), vsmem, s, args);
}

}  // namespace adapld
