// Rerank and draft-tree construction (Sec. 3.4-3.6, Eq. 6-15, Algorithm 1).
//
// In single-cache mode with histories of at most 16 slices of 8192 positions
// (every workload shape here) the stage is one kernel of thread-block
// clusters, tree_cluster_kernel (see its comment below): the CTAs of a
// sequence scan slices, score rows and hand their results to CTA rank 0
// through distributed shared memory.  The kernels below serve the other
// cases (token-embedding mode, whose successor backoff runs between the scan
// and the scoring, and longer histories).
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
// ADAPLD_SUCC_ON_STRICT).  Each CTA stages its slice of 8192 positions (and
// the one after it) while it reads the sequence's outcome, rebuilds the
// anchor and the branch set (lexical hits are reranked here in that mode),
// then scans the slice for the branch tokens, a warp per branch, backwards
// with ballots, keeping the k most recent occurrences.  The last slice CTA
// (atomic ticket; none with one slice) merges the slices, most recent first,
// into the successor candidate lists; slice 0 publishes the branch set.
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
//
// Each of these CTAs moves a few KB, so its time is the number of dependent
// memory round trips.  Loads that do not depend on one another are issued
// together: the branch set, the ranked candidates and each warp's list entry
// with the sequence's outcome; each warp's first row with the reference
// vector, the candidates' continuation tokens and the token after each scored
// row.  With one slice the fused kernel reads every history token it needs
// from the staged slice.
#include <cstdlib>

#include "common.cuh"

namespace adapld {

namespace {

constexpr int kRowsPerCta5 = kThreads4 / 32;  // one warp per scored row
constexpr int kWin = 16;  // continuation tokens staged per lexical candidate
constexpr int kVecPer = 16384 / 8 / kThreads4;  // 16-byte chunks per thread of a staged vector
static_assert(kMaxK * kWin == kThreads4, "one continuation token per thread");

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
    int slot[kMaxK];  // window row (win) of each ranked candidate
    int next[kMaxW];
    int br[kMaxW];
    int succ[kMaxW];  // the successor picked for each branch (Eq. 14)
    int stok[kMaxW];  // and the token after it
    int misc[4];
    int lpos[kMaxK];  // rows of a CTA that scores all of its sequence's rows:
    float lsc[kMaxK];  //   position, score and the token after the position
    int ltok[kMaxK];
    int win[kMaxK][kWin];  // M[c+1 .. c+kWin] of each lexical candidate c (-1 past len-1)
    int node_par[kMaxNodes];
    short node_depth[kMaxNodes];
    short node_path[kMaxNodes];
    int node_src[kMaxNodes];
    float red[32];
};

// Where a CTA reads history tokens: the staged history (s_tok: positions
// [0, ld) of the sequence), or global memory; wsm, when set, holds the
// continuation windows of the candidates (M[s_cand[q]+1] = win[slot[q]][0]).
__device__ __forceinline__ float *s_red_of(TreeSmem &sm) { return sm.red; }

struct TokSrc {
    const int *s_tok;
    const TreeSmem *wsm;
};

// One warp's dot product of a bf16 row in global memory with a bf16 vector
// in shared memory (both widened exactly to fp32), in batches of U 16-byte
// chunks per lane: chunk
// base + 32u + lane for u < U.  A lane sums its chunks lane, lane + 32, ... in
// increasing order whatever U, so the result does not depend on U or on where
// the first batch was loaded.
template <int U>
__device__ __forceinline__ void row_batch_load(const uint16_t *row, int nch, int base,
                                               uint4 (&w)[U]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int u = 0; u < U; ++u) {
        const int ch = base + u * 32 + lane;
        w[u] = ch < nch ? ldg_nc_v4(row + (size_t)ch * 8) : make_uint4(0, 0, 0, 0);
    }
}

template <int U>
__device__ __forceinline__ void row_batch_acc(const uint4 (&w)[U], const uint16_t *ref, int nch,
                                              int base, float &dot, float &ss) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int u = 0; u < U; ++u) {
        const int ch = base + u * 32 + lane;
        if (ch < nch) {
            const uint4 rv = *(const uint4 *)(ref + ch * 8);
            const float4 r0 = make_float4(bf16lo(rv.x), bf16hi(rv.x), bf16lo(rv.y), bf16hi(rv.y));
            const float4 r1 = make_float4(bf16lo(rv.z), bf16hi(rv.z), bf16lo(rv.w), bf16hi(rv.w));
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

// <row, ref> and |row|^2 (warp totals); w holds the row's first batch.
template <int U>
__device__ __forceinline__ void warp_row_dot_from(const uint16_t *row, const uint16_t *ref, int d,
                                                  uint4 (&w)[U], float &dot_out, float &ss_out) {
    const int nch = d >> 3;
    float dot = 0.f, ss = 0.f;
    row_batch_acc<U>(w, ref, nch, 0, dot, ss);
    for (int base = 32 * U; base < nch; base += 32 * U) {
        row_batch_load<U>(row, nch, base, w);
        row_batch_acc<U>(w, ref, nch, base, dot, ss);
    }
    dot_out = warp_sum(dot);
    ss_out = warp_sum(ss);
}

template <int U>
__device__ __forceinline__ void warp_row_dot(const uint16_t *row, const uint16_t *ref, int d,
                                             float &dot_out, float &ss_out) {
    uint4 w[U];
    row_batch_load<U>(row, d >> 3, 0, w);
    warp_row_dot_from<U>(row, ref, d, w, dot_out, ss_out);
}

// A bf16 vector of d <= 16384 elements staged in shared memory (16-byte
// aligned, d bf16) by the 512-thread block: vec_issue starts its copies (at
// most kVecPer per thread), vec_finish waits for every cp.async of the
// thread and returns the squared norm to every thread (block-wide;
// synchronises the block).
__device__ __forceinline__ void vec_issue(const uint16_t *v, int d, uint16_t *dst) {
    const int nch = d >> 3;
#pragma unroll
    for (int u = 0; u < kVecPer; ++u) {
        const int ch = u * kThreads4 + threadIdx.x;
        if (ch < nch) cp_async16(dst + ch * 8, v + (size_t)ch * 8);
    }
}

__device__ float vec_finish(const uint16_t *dst, int d, float *scratch) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nch = d >> 3;
    cp_async_wait_all();
    __syncthreads();
    float part = 0.f;
#pragma unroll
    for (int u = 0; u < kVecPer; ++u) {
        const int ch = u * kThreads4 + threadIdx.x;
        if (ch < nch) {
            const uint4 w = *(const uint4 *)(dst + ch * 8);
            const float x[8] = {bf16lo(w.x), bf16hi(w.x), bf16lo(w.y), bf16hi(w.y),
                                bf16lo(w.z), bf16hi(w.z), bf16lo(w.w), bf16hi(w.w)};
#pragma unroll
            for (int e = 0; e < 8; ++e) part = fmaf(x[e], x[e], part);
        }
    }
    part = warp_sum(part);
    if (lane == 0) scratch[warp] = part;
    __syncthreads();
    float tot = 0.f;
    for (int w = 0; w < kThreads4 / 32; ++w) tot += scratch[w];
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

// Values written by earlier kernels that a tree-kernel CTA may need, loaded
// together with the sequence's outcome.  They are read in bounds but
// speculatively (possibly stale) and used only where the outcome says the
// successor scan wrote them.
struct TreePrefetch {
    int brs;       // thread t <= W: the branch count (t = 0), then the branch tokens
    int rr_c;      // thread t < k: the candidates as ranked by the successor scan
    float rr_s;
    int task_pos;  // the first row of this thread's warp: its successor candidate
    int task_n;    // and the candidate count of its branch
};

__device__ __forceinline__ TreePrefetch prefetch_tree(const TreeLaunch &a, const Workspace &ws,
                                                      int b, int r5) {
    TreePrefetch f;
    const int t = threadIdx.x, k = a.p.k, W = ws.W;
    f.brs = t <= W ? __ldcg(ws.brs + (int64_t)b * (W + 1) + t) : 0;
    f.rr_c = t < k ? __ldcg(ws.rr_cand + (int64_t)b * kMaxK + t) : 0;
    f.rr_s = t < k ? __ldcg(ws.rr_score + (int64_t)b * kMaxK + t) : 0.f;
    const int task = r5 * kRowsPerCta5 + (t >> 5);
    const int w = task / k, i = task - w * k;
    const bool in = w < W;
    f.task_pos = in ? __ldcg(ws.succ + ((int64_t)b * W + w) * kMaxK + i) : -1;
    f.task_n = in ? __ldcg(ws.succ_n + (int64_t)b * W + w) : 0;
    return f;
}

__device__ __forceinline__ int tok_at(const TokSrc &src, const int32_t *M, int p) {
    return src.s_tok ? src.s_tok[p] : __ldg(M + p);
}

// Branch set (Eq. 10-11) into s_br, count returned; s_cand holds the ranked
// candidates (s_cand[0] = j*).  Block-wide: every thread must call.
__device__ __forceinline__ int branch_set(const TreeLaunch &a, int b, const SeqView &v,
                                          const int *s_cand, int *s_next, int *s_br,
                                          int *s_misc, const TokSrc &src) {
    const int t = threadIdx.x, W = a.p.branch_width;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    // M[s_cand[q] + 1], the continuation of ranked candidate q
    auto next_of = [&](int q) {
        if (src.s_tok) return src.s_tok[s_cand[q] + 1];
        if (src.wsm) return src.wsm->win[src.wsm->slot[q]][0];
        return __ldg(M + s_cand[q] + 1);
    };
    if (a.next_topk) {
        const int32_t *row = a.next_topk + ((int64_t)b * a.ld + s_cand[0]) * a.Kn;
        if (t < a.Kn) s_next[t] = row[t];
    } else if (t < v.nc) {
        s_next[t] = next_of(t);
    }
    if (t == kThreads4 - 1) s_misc[0] = v.lex ? next_of(0) : -1;
    __syncthreads();
    if (t < 32) {  // warp 0: the first W distinct continuations (or the first W ids of
                   // the table row), then Eq. 11's removal of main[0], order kept
        const int lane = t;
        const int n = a.next_topk ? a.Kn : v.nc;
        const int main0 = s_misc[0];
        int nb = 0, taken = 0;
        for (int base = 0; base < n && taken < W; base += 32) {  // (nc <= 32: one pass)
            const int r = base + lane;
            const bool in = r < n;
            const int tkn = in ? s_next[r] : 0;
            bool keep;
            if (a.next_topk) {
                keep = in && tkn >= 0;
            } else {  // the first occurrence of each token in rank order
                const unsigned peers = __match_any_sync(0xffffffffu, tkn) &
                                       __ballot_sync(0xffffffffu, in);
                keep = in && __ffs(peers) - 1 == lane;
            }
            const unsigned below = (1u << lane) - 1u;
            const unsigned km = __ballot_sync(0xffffffffu, keep);
            const bool sel = keep && taken + __popc(km & below) < W;
            const bool fin = sel && !(v.lex && tkn == main0);
            const unsigned fm = __ballot_sync(0xffffffffu, fin);
            if (fin) s_br[nb + __popc(fm & below)] = tkn;
            nb += __popc(fm);
            taken += __popc(km);
        }
        if (lane == 0) s_misc[1] = nb;
    }
    __syncthreads();
    return s_misc[1];
}

// Warp 0 sorts n <= 32 (score, position) pairs in place by (score desc,
// position desc); s_slot, when given, is permuted alongside.
__device__ __forceinline__ void warp_sort_desc(int *s_cand, float *s_score, int n,
                                               int *s_slot) {
    const int lane = threadIdx.x & 31;
    const float sc = lane < n ? s_score[lane] : -INFINITY;
    const int cj = lane < n ? s_cand[lane] : -1;
    const int sl = (s_slot && lane < n) ? s_slot[lane] : 0;
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
        if (s_slot) s_slot[rank] = sl;
    }
    __syncwarp();
}

// The k most recent positions p in [lo, hi) with M[p] == br[w], for every
// branch w < nb, most recent first: store(w, rank, p) for rank < k, then
// count(w, c) once per branch (by thread w) with c = their number (<= k);
// s_tok[p - p0] holds M[p] and hi - lo <= 16 * kThreads4.  Block-wide (every
// thread).  Thread t owns the consecutive positions lo + pt t .. + pt - 1
// (pt <= 16) and keeps their tokens in registers; per branch it forms the bit
// mask of its matches, a warp with any match scans the counts from its top
// lane, and the warps' totals (wc: 16 * nb ints of scratch) give, after one
// CTA barrier per four branches, every match its rank: higher warps, then
// higher lanes, then higher positions first.
template <class Store, class Count>
__device__ __forceinline__ void scan_branches(const int *s_tok, int64_t p0, int64_t lo,
                                              int64_t hi, const int *br, int nb, int k, int *wc,
                                              Store store, Count count) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    constexpr int NW = kThreads4 / 32, PT = 16, NBC = 4;  // branches per pass
    const int n = hi > lo ? (int)(hi - lo) : 0;
    const int pt = (n + kThreads4 - 1) / kThreads4;  // <= PT
    const int q0 = (int)(lo - p0) + pt * t;          // s_tok index of the first position
    const int cnt = max(0, min(pt, n - pt * t));     // positions of this thread
    int tk[PT];
    if (cnt == PT && (q0 & 3) == 0) {
#pragma unroll
        for (int g = 0; g < PT / 4; ++g) {
            const int4 v = *reinterpret_cast<const int4 *>(s_tok + q0 + 4 * g);
            tk[4 * g] = v.x;
            tk[4 * g + 1] = v.y;
            tk[4 * g + 2] = v.z;
            tk[4 * g + 3] = v.w;
        }
    } else {
#pragma unroll
        for (int e = 0; e < PT; ++e) tk[e] = e < cnt ? s_tok[q0 + e] : 0;
    }
    const uint32_t valid = (1u << cnt) - 1u;  // cnt <= 16
    for (int w0 = 0; w0 < nb; w0 += NBC) {
        uint32_t m[NBC];
        int excl[NBC];  // matches of the higher lanes of this warp
#pragma unroll
        for (int j = 0; j < NBC; ++j) {
            m[j] = 0;
            excl[j] = 0;
            if (w0 + j >= nb) continue;
            const int bt = br[w0 + j];
#pragma unroll
            for (int e = 0; e < PT; ++e) m[j] |= (uint32_t)(tk[e] == bt) << e;
            m[j] &= valid;
            int tot = 0;
            if (__any_sync(0xffffffffu, m[j] != 0)) {
                const int c = __popc(m[j]);
                int incl = c;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int u = __shfl_down_sync(0xffffffffu, incl, o);
                    if (lane + o < 32) incl += u;
                }
                excl[j] = incl - c;
                tot = __shfl_sync(0xffffffffu, incl, 0);
            }
            if (lane == 0) wc[warp * nb + w0 + j] = tot;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < NBC; ++j) {
            if (m[j] == 0) continue;
            const int w = w0 + j;
            int off = excl[j];
            for (int u = warp + 1; u < NW; ++u) off += wc[u * nb + w];
            for (uint32_t h = m[j]; h && off < k; ++off) {
                const int e = 31 - __clz(h);
                h &= ~(1u << e);
                store(w, off, (int)(lo + pt * t + e));
            }
        }
    }
    if (t < nb) {
        int total = 0;
        for (int u = 0; u < NW; ++u) total += wc[u * nb + t];
        count(t, min(total, k));
    }
}

// ---------------------------------------------------------------------------
// Publishes the successor-candidate count of branch w of sequence b.  A
// branch token that never occurs earlier backs off (Sec. 3.5) to the
// embedding fallback with the branch token as the anchor: with a table, the
// (sequence, branch) pair is registered for the gathered pass.  On the step
// path a semantic hit's own anchor never occurred earlier either, and its
// backoff -- Eq. 4 with that anchor as the query over the same positions,
// threshold and k -- is exactly the fallback this step already ran: its
// candidate set (nc entries of s_cand, in any order; Eq. 14 takes a
// maximum) is copied instead of being scored again.  reuse: the sequence is
// such a hit, anchor its token.
__device__ __forceinline__ void register_successors(const TreeLaunch &a, const Workspace &ws,
                                                    int b, int w, int total, int token,
                                                    bool reuse, int anchor, int nc,
                                                    const int *s_cand) {
    if (total == 0 && reuse && token == anchor) {
        int32_t *dst = ws.succ + ((int64_t)b * ws.W + w) * kMaxK;
        for (int i = 0; i < nc; ++i) dst[i] = s_cand[i];
        ws.succ_n[(int64_t)b * ws.W + w] = nc;
        return;
    }
    ws.succ_n[(int64_t)b * ws.W + w] = total;
    if (total == 0 && a.emb.table) {
        const int idx = atomicAdd(ws.npairs, 1);
        ws.pair_b[idx] = b;
        ws.pair_tok[idx] = token;
        ws.pair_out[idx] = b * ws.W + w;
    }
}

// Lays out and writes the draft tree of sequence b (the root, the main chain
// of a lexical hit, then each branch with its successor chain) and the
// per-sequence outputs: tokens, parents, position ids, the ancestor mask,
// the ranked candidates (lexical / reranked), anchor, node count, statistics
// and status.  sm holds the ranked candidates (cand, score, slot), the
// branch set (br, nb branches), the successor picked per branch (succ, stok)
// when the sequence drafts successors, and the continuation windows (win)
// when use_win.  Block-wide (every thread).
__device__ __forceinline__ void emit_tree(const TreeLaunch &a, int b, const SeqView &v, TreeSmem &sm,
                          const TokSrc &src, bool use_win, int nb, int status0,
                          int32_t *dst = nullptr) {
    int *s_cand = sm.cand;
    float *s_score = sm.score;
    int *s_br = sm.br;
    int *s_succ = sm.succ;
    int *s_misc = sm.misc;
    int *node_par = sm.node_par;
    short *node_depth = sm.node_depth;
    short *node_path = sm.node_path;
    int *node_src = sm.node_src;
    const int t = threadIdx.x;
    const int k = a.p.k, W = a.p.branch_width, D = a.p.draft_len;
    const int succ_len = a.p.succ_len;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const int js = (v.lex || v.sem) ? s_cand[0] : -1;
    const int N = 1 + D + W * (1 + succ_len);
    // node layout, in parallel: the root, the main chain (l nodes), then per
    // branch w its node and its successor chain of added_w nodes, starting at
    // 1 + l + the sizes of the branches before it (a warp scan)
    const int l = (v.valid && v.lex) ? min(D, v.len - 1 - js) : 0;
    int *s_start = sm.next;  // (free once the branch set is built)
    const int nbv = v.valid ? nb : 0;
    if (t < 32) {
        const int lane = t;
        int carry = 1 + l, ext = 0;
        for (int base = 0; base < nbv; base += 32) {
            const int w = base + lane;
            int size = 0, added = 0;
            if (w < nbv) {
                if (v.need_succ && s_succ[w] >= 0) added = min(succ_len, v.len - 1 - s_succ[w]);
                size = 1 + added;
            }
            int incl = size;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += u;
            }
            if (w < nbv) s_start[w] = carry + incl - size;
            carry += __shfl_sync(0xffffffffu, incl, 31);
            ext += __popc(__ballot_sync(0xffffffffu, added > 0));
        }
        if (lane == 0) {
            s_misc[0] = v.valid ? carry : 0;
            s_misc[3] = ext;
        }
    }
    if (v.valid && t <= l) {  // the root and the main chain
        node_par[t] = t - 1;
        node_depth[t] = (short)t;
        node_path[t] = t == 0 ? 0 : 1;
        node_src[t] = t == 0 ? v.len - 1 : js + t;
    }
    __syncthreads();
    {
        const int lane = t & 31, warp = t >> 5;
        for (int w = warp; w < nbv; w += kThreads4 / 32) {  // branch w: its node, then
                                                             // its successors
            const int st = s_start[w];
            const int size = (w + 1 < nbv ? s_start[w + 1] : s_misc[0]) - st;
            if (lane < size && idx_ok(st + lane, 1, N, dst)) {
                const int nd = st + lane;
                node_par[nd] = lane == 0 ? 0 : nd - 1;
                node_depth[nd] = (short)(1 + lane);
                node_path[nd] = (short)(2 + w);
                node_src[nd] = lane == 0 ? -2 - w : s_succ[w] + lane;  // -2-w: the branch token
            }
        }
    }
    __syncthreads();
    const int n = s_misc[0];
    const int64_t ob = (int64_t)b * N;
    for (int i = t; i < N; i += kThreads4) {
        int tok = -1, par = -1, pos = -1;
        if (i < n) {
            const int s = node_src[i], path = node_path[i], depth = node_depth[i];
            if (s < 0)
                tok = s_br[-2 - s];
            else if (!idx_ok(s, 0, v.len, dst))
                tok = -1;
            else if (src.s_tok)
                tok = src.s_tok[s];
            else if (path == 1 && use_win && depth <= kWin)  // main chain: s = j* + depth
                tok = sm.win[sm.slot[0]][depth - 1];
            else if (path >= 2 && depth == 2)  // a branch's first successor token
                tok = sm.stok[path - 2];
            else
                tok = __ldg(M + s);
            par = node_par[i];
            pos = v.len - 1 + depth;
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

template <int U>
__device__ void tree_body(const TreeLaunch &a, const Workspace &ws, int b, const SeqView &v,
                          int r5, bool fused, TreeSmem &sm, uint16_t *s_ref, const TokSrc &src,
                          const TreePrefetch *pf, int nb_known, bool lists_smem);

// FUSED: the CTA that completes a sequence's scan (or CTA 0 of a sequence
// without successors) then builds that sequence's tree itself (tree_body,
// all scored rows in this CTA), so the tree stage is one kernel.  U: row
// loads in flight in tree_body.  Dynamic shared memory: d bf16 (the query or
// reference vector), then kSlice4 + 1 ints (this slice's tokens).
template <int U, bool FUSED>
__global__ void __launch_bounds__(kThreads4, U == 8 ? 2 : 1) succ_scan_kernel(TreeArgs args) {
    const TreeLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ TreeSmem sm;
    extern __shared__ __align__(16) uint16_t s_dyn[];
    uint16_t *s_q = s_dyn;
    int *s_tok = (int *)(s_dyn + a.d);
    int *s_cand = sm.cand;
    float *s_score = sm.score;
    int *s_next = sm.next;
    int *s_br = sm.br;
    int *s_misc = sm.misc;
    float *s_red = sm.red;

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nwarps = kThreads4 / 32;
    const int b = blockIdx.y, sl = blockIdx.x;
    const int k = a.p.k, d = a.d;
    const bool single = gridDim.x == 1;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const uint16_t *R = a.reps + (int64_t)b * a.ld * d;
    pdl_wait_then_release();
    // this slice's tokens, positions [p0, p0 + kSlice4] clipped at ld, copied
    // while the sequence's outcome is read (they do not depend on it)
    const int p0 = sl * kSlice4;
    const int nld = (int)min((int64_t)kSlice4 + 1, a.ld - p0);
    for (int i = t; i < nld; i += kThreads4) cp_async4(s_tok + i, M + p0 + i);
    const SeqView v = view_of(a, b);
    // a semantic hit of this step reuses its fallback for its anchor's backoff
    const bool reuse = a.lists_ready && v.sem && v.valid;
    const int anchor = reuse ? __ldg(M + v.len - 1) : 0;
    cp_async_wait_all();  // (also before an exit: the copies target this CTA's memory)
    if (!v.need_succ && !(FUSED && sl == 0)) return;
    __syncthreads();
    // with one slice the staged tokens are the whole history
    const TokSrc src{single ? s_tok : nullptr, nullptr};
    if constexpr (FUSED) {
        if (!v.need_succ) {
            tree_body<U>(a, ws, b, v, 0, true, sm, s_q, src, nullptr, -1, false);
            return;
        }
    }

    if (t < v.nc) {
        s_cand[t] = v.cand_t;
        s_score[t] = v.score_t;
    }
    __syncthreads();
    if (v.rr) {  // the ranking the branches depend on (each slice alike; the
                 // arithmetic of the tree kernel's rerank, so the scores agree)
        uint4 w0[8];  // each warp's first candidate row, loaded with the query
        if (warp < v.nc) row_batch_load<8>(R + (int64_t)s_cand[warp] * d, d >> 3, 0, w0);
        vec_issue(a.query + (int64_t)b * d, d, s_q);
        const float qss = vec_finish(s_q, d, s_red);
        if (warp < v.nc) {
            float dot, ss;
            warp_row_dot_from<8>(R + (int64_t)s_cand[warp] * d, s_q, d, w0, dot, ss);
            if (lane == 0) s_score[warp] = cosine_from(dot, ss, qss);
        }
        for (int ci = warp + nwarps; ci < v.nc; ci += nwarps) {
            float dot, ss;
            warp_row_dot<8>(R + (int64_t)s_cand[ci] * d, s_q, d, dot, ss);
            if (lane == 0) s_score[ci] = cosine_from(dot, ss, qss);
        }
        __syncthreads();
        if (warp == 0) warp_sort_desc(s_cand, s_score, v.nc, nullptr);
        __syncthreads();
    } else if (v.lex) {
        if (t < v.nc) s_score[t] = __int_as_float(0x7fc00000);  // NaN: not computed
        __syncthreads();
    }
    const int nb = branch_set(a, b, v, s_cand, s_next, s_br, s_misc, src);
    if (!FUSED && sl == 0) {  // the branch set, for the tree kernel
        int32_t *bo = ws.brs + (int64_t)b * (ws.W + 1);
        if (t == 0) bo[0] = nb;
        if (t < nb) bo[1 + t] = s_br[t];
    }

    const int p1 = min(p0 + kSlice4, v.len - 1);  // positions t <= len-2
    constexpr int G = 8;  // 32-position groups tested per pass (independent loads)
    // one slice: its lists are the merged result, written in place (no merge);
    // the fused kernel keeps them in shared memory (W*k <= 16)
    const bool lists_smem = FUSED && single;
    for (int w = warp; w < nb; w += nwarps) {
        const int bt = s_br[w];
        int32_t *part =
            single ? nullptr : ws.part4 + (((int64_t)b * ws.S4 + sl) * ws.W + w) * kPart4Ints;
        int32_t *lst = lists_smem ? sm.lpos + w * k
                                  : (single ? ws.succ + ((int64_t)b * ws.W + w) * kMaxK : part + 1);
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
                if (((m[u] >> lane) & 1u) && rank < k && idx_ok(p, p0, p1, ws.dev_status))
                    lst[rank] = p;
                cnt += __popc(m[u]);
            }
        }
        if (lists_smem) {  // entries past the count read as "no row"
            __syncwarp();
            for (int i = min(cnt, k) + lane; i < k; i += 32) lst[i] = -1;
        }
        if (lane == 0) {
            if (single)
                register_successors(a, ws, b, w, min(cnt, k), s_br[w], reuse, anchor, v.nc,
                                    s_cand);
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
            if (lane == 0)
                register_successors(a, ws, b, w, total, s_br[w], reuse, anchor, v.nc, s_cand);
        }
    }
    if (!FUSED && (v.lex || v.rr) && t < v.nc) {
        ws.rr_cand[(int64_t)b * kMaxK + t] = s_cand[t];
        ws.rr_score[(int64_t)b * kMaxK + t] = s_score[t];
    }
    if constexpr (FUSED) {
        __syncthreads();  // the lists and the ranking above are visible to the block
        tree_body<U>(a, ws, b, v, 0, true, sm, s_q, src, nullptr, nb, lists_smem);
    }
}

// The plan of the successor backoff pass: row prefix sums over the
// (sequence, branch) pairs registered by succ_scan_kernel (one CTA).
__global__ void __launch_bounds__(256) backoff_plan_kernel(TreeArgs args) {
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
// d bf16 of shared memory (16-byte aligned).  src: where history tokens are read.  pf: the
// tree kernel's prefetched values (NULL in the fused kernel).  nb_known >= 0:
// the fused scan left the ranked candidates and the branch set (nb_known
// branches) in sm.  lists_smem: the successor lists are in sm.lpos.
template <int U>
__device__ void tree_body(const TreeLaunch &a, const Workspace &ws, int b, const SeqView &v,
                          int r5, bool fused, TreeSmem &sm, uint16_t *s_ref, const TokSrc &src,
                          const TreePrefetch *pf, int nb_known, bool lists_smem) {
    int *s_cand = sm.cand;
    float *s_score = sm.score;
    int *s_next = sm.next;
    int *s_br = sm.br;
    int *s_succ = sm.succ;
    int *s_misc = sm.misc;
    float *s_red = sm.red;

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nwarps = kThreads4 / 32;
    const int k = a.p.k, d = a.d;
    const uint32_t flags = a.p.flags;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const uint16_t *R = a.reps + (int64_t)b * a.ld * d;
    // the status word is rewritten at the end; its token bit comes from
    // earlier kernels, so it is read now, off the tail's critical path
    const int status0 = (a.status && t == 0) ? a.status[b] : 0;
    if (t < kMaxK) sm.slot[t] = t;

    // ---- ranked candidates; with successors, the branch set
    int nb = 0;
    if (nb_known >= 0) {
        nb = nb_known;
    } else {
        if (t < v.nc) {  // the successor scan ranked these already
            const bool from_scan = pf && v.need_succ && (v.lex || v.rr);
            s_cand[t] = from_scan ? pf->rr_c : v.cand_t;
            s_score[t] = from_scan ? pf->rr_s : v.score_t;
        }
        if (pf && v.need_succ) {  // published by the successor scan
            if (t >= 1 && t <= ws.W) s_br[t - 1] = pf->brs;
            if (t == 0) s_misc[1] = pf->brs;
        }
        __syncthreads();
        if (v.need_succ) nb = s_misc[1];
    }

    // the rows this sequence scores, and the CTAs that share them: lexical
    // candidates against the query, or successor candidate (w, i) at w*k + i
    const bool rerank = v.rr && !v.need_succ;
    const int ntasks = v.need_succ ? nb * k : (rerank ? v.nc : 0);
    const int nctas = fused ? 1 : max(1, (ntasks + kRowsPerCta5 - 1) / kRowsPerCta5);
    if (r5 >= nctas) return;
    const bool local = nctas == 1;  // every row in this CTA: results stay in sm
    const int js0 = (v.lex || v.sem) ? s_cand[0] : -1;
    float *score5 = ws.score5 + (int64_t)b * ws.W * kMaxK;
    int32_t *tok5 = ws.tok5 + (int64_t)b * ws.W * kMaxK;
    // continuation windows of the candidates (branch tokens, main chain) when
    // the history is not staged
    const bool use_win = !src.s_tok && v.nc > 0 && (v.lex || (v.branch_on && !v.need_succ));

    // ---- this CTA's share of the scored rows, every independent load first
    const int task0 = fused ? 0 : r5 * kRowsPerCta5;
    const int task1 = fused ? ntasks : min(ntasks, task0 + kRowsPerCta5);
    auto row_of = [&](int task, bool first) -> int {
        if (!v.need_succ) return s_cand[task];
        if (lists_smem) return sm.lpos[task];
        const int w = task / k, i = task - w * k;
        int n, pos;
        if (first && pf) {
            n = pf->task_n;
            pos = pf->task_pos;
        } else {
            n = __ldcg(ws.succ_n + (int64_t)b * ws.W + w);
            pos = __ldcg(ws.succ + ((int64_t)b * ws.W + w) * kMaxK + i);
        }
        return i < n ? pos : -1;
    };
    const int first_task = task0 + warp;
    int row0 = first_task < task1 ? row_of(first_task, true) : -1;
    if (!idx_ok(row0, -1, v.len - 1, ws.dev_status)) row0 = -1;
    uint4 w0[U];
    if (row0 >= 0) row_batch_load<U>(R + (int64_t)row0 * d, d >> 3, 0, w0);
    if (ntasks > 0)
        vec_issue(v.need_succ ? R + (int64_t)(js0 + 1) * d : a.query + (int64_t)b * d, d, s_ref);
    const int tk0 = (v.need_succ && row0 >= 0 && lane == 0) ? tok_at(src, M, row0 + 1) : -1;
    if (use_win && t < v.nc * kWin) {
        const int r = t / kWin, o = t - r * kWin;
        const int p = s_cand[r] + 1 + o;
        sm.win[r][o] = p <= v.len - 1 ? __ldg(M + p) : -1;
    }
    if (ntasks > 0) {
        const float rss = vec_finish(s_ref, d, s_red);  // syncs the block
        auto record = [&](int task, int row, float sc, int tk) {  // lane 0
            if (local) {
                sm.lpos[task] = row;
                sm.lsc[task] = sc;
                sm.ltok[task] = tk;
            } else {
                if (row >= 0) score5[task] = sc;
                if (v.need_succ) tok5[task] = tk;
            }
        };
        if (first_task < task1) {  // the first row's loads are in flight already
            float sc = 0.f;
            if (row0 >= 0) {
                float dot, ss;
                warp_row_dot_from<U>(R + (int64_t)row0 * d, s_ref, d, w0, dot, ss);
                sc = cosine_from(dot, ss, rss);
            }
            if (lane == 0) record(first_task, row0, sc, tk0);
        }
        for (int task = first_task + nwarps; task < task1; task += nwarps) {
            int row = row_of(task, false);
            if (!idx_ok(row, -1, v.len - 1, ws.dev_status)) row = -1;
            float sc = 0.f;
            if (row >= 0) {
                float dot, ss;
                warp_row_dot<U>(R + (int64_t)row * d, s_ref, d, dot, ss);
                sc = cosine_from(dot, ss, rss);
            }
            if (lane == 0)
                record(task, row, sc, (v.need_succ && row >= 0) ? tok_at(src, M, row + 1) : -1);
        }
        if (!local) {
            __threadfence();
            __syncthreads();
            if (t == 0) s_misc[2] = atomicAdd(ws.ticket5 + b, 1) == nctas - 1;
            __syncthreads();
            if (!s_misc[2]) return;
            __threadfence();
        } else {
            __syncthreads();
        }
    } else {
        __syncthreads();  // the windows are visible to the block
    }

    // ---- the last CTA of the sequence: rank, branch, pick successors, emit
    if (rerank) {
        if (warp == 0) {
            if (lane < v.nc) s_score[lane] = local ? sm.lsc[lane] : __ldcg(score5 + lane);
            __syncwarp();
            warp_sort_desc(s_cand, s_score, v.nc, sm.slot);
        }
        __syncthreads();
    } else if (v.lex && (flags & ADAPLD_NO_LEX_RERANK)) {
        if (t < v.nc) s_score[t] = __int_as_float(0x7fc00000);  // NaN: not computed
        __syncthreads();
    }
    if (v.branch_on && !v.need_succ)
        nb = branch_set(a, b, v, s_cand, s_next, s_br, s_misc,
                        TokSrc{src.s_tok, use_win ? &sm : nullptr});
    if (v.need_succ) {
        for (int w = warp; w < nb; w += nwarps) {  // Eq. 14: argmax per branch
            float bs;
            int bj, btk;
            if (local) {
                const int pl = lane < k ? sm.lpos[w * k + lane] : -1;
                bs = pl >= 0 ? sm.lsc[w * k + lane] : -INFINITY;
                bj = pl;
                btk = pl >= 0 ? sm.ltok[w * k + lane] : -1;
            } else {
                // all four loads at once (lanes past the count are masked after)
                const int n = __ldcg(ws.succ_n + (int64_t)b * ws.W + w);
                const float sl = __ldcg(score5 + w * k + lane);
                const int pl = __ldcg(ws.succ + ((int64_t)b * ws.W + w) * kMaxK + lane);
                const int tl = __ldcg(tok5 + w * k + lane);
                bs = lane < n ? sl : -INFINITY;
                bj = lane < n ? pl : -1;
                btk = tl;
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) {
                const float os = __shfl_xor_sync(0xffffffffu, bs, o);
                const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
                const int ot = __shfl_xor_sync(0xffffffffu, btk, o);
                if (better(os, oj, bs, bj)) {
                    bs = os;
                    bj = oj;
                    btk = ot;
                }
            }
            if (lane == 0) {
                s_succ[w] = bj >= 0 ? bj : -1;
                sm.stok[w] = btk;
            }
        }
        __syncthreads();
    }

    emit_tree(a, b, v, sm, src, use_win, nb, status0, ws.dev_status);
}

// U: row loads in flight per lane.  U = 16 (one CTA per SM by registers)
// when the grid fits one wave, U = 8 (two CTAs per SM) otherwise; the
// scores are the same either way (see row_batch_acc).
template <int U>
__global__ void __launch_bounds__(kThreads4, U == 8 ? 2 : 1) tree_kernel(TreeArgs args) {
    __shared__ TreeSmem sm;
    extern __shared__ __align__(16) uint16_t s_ref[];  // [d] reference vector (bf16)
    pdl_wait_then_release();
    const TreePrefetch pf = prefetch_tree(args.p, args.ws, blockIdx.y, blockIdx.x);
    const SeqView v = view_of(args.p, blockIdx.y);
    tree_body<U>(args.p, args.ws, blockIdx.y, v, blockIdx.x, false, sm, s_ref,
                 TokSrc{nullptr, nullptr}, &pf, -1, false);
}

// ---------------------------------------------------------------------------
// The whole tree stage as one kernel of thread-block clusters (single-cache
// mode; histories of at most 16 slices of 8192 positions).  Grid (X, B),
// 512 threads; the X CTAs of a sequence are one cluster and share its work
// through distributed shared memory instead of global tickets:
//   P0  every CTA stages its slice of the history (span positions and the one
//       after), reads the outcome, and starts the copy of the reference
//       vector (the query for a rerank, R[j*+1] for successor rows) and the
//       candidates' continuation windows;
//   P1  (lexical hits that draft successors) the candidates are reranked
//       (Eq. 6-7) over the cluster's warps; rank 0 collects the scores and
//       every CTA sorts them alike;
//   P2  every CTA derives the branch set (Eq. 10-11);
//   P3  each CTA scans its slice for the branch tokens (every thread 16
//       consecutive positions held in registers, a bit mask per branch),
//       keeping the k most recent occurrences, and writes its lists into
//       every CTA's shared memory (or, when X * W * (k + 1) ints exceed
//       32 KB, leaves them in its own);
//   P4  after a cluster barrier every CTA merges the slices' lists (ranks
//       hold contiguous slices, higher ranks more recent) from its own
//       shared memory (or the other CTAs');
//   P5  the scored rows (successor candidates against R[j*+1], Eq. 13, or
//       the lexical candidates against the query, Eq. 6) are spread over the
//       cluster's warps, one row per warp; each score and the token after
//       its row go to rank 0's shared memory;
//   P6  after a second barrier rank 0 ranks (Eq. 7), picks each branch's
//       successor (Eq. 14) and writes the tree.
// Every CTA passes every cluster barrier (no early exit before them); the
// barriers' conditions depend only on the sequence, hence agree in a cluster.
// A first cluster barrier, arrived at on entry and waited for in P1, makes
// sure every CTA has started before any writes another's shared memory.
// A scored row is split into parts of 4096 elements (512 16-byte chunks,
// one batch of loads at U = 16), each part one warp's work item, so a warp
// waits for at most one batch of row loads per item.
constexpr int kPartCh = 512;
__host__ __device__ inline int row_parts(int d) { return ((d >> 3) + kPartCh - 1) / kPartCh; }

struct ClusterLayout {
    uint32_t tok, cnt, lst, mcnt, mlst, wc, sc, tk, pd, ps, gath, total;
};

// Bytes of the lists every CTA pushes into every other (X CTAs x W branches x
// (count + k positions)); above this they are read remotely instead.
constexpr size_t kPushBytes = 32 * 1024;
__host__ __device__ inline size_t push_bytes(int X, int W, int k) {
    return 4 * (size_t)X * W * (1 + k);
}

__host__ __device__ inline ClusterLayout cluster_layout(int d, int span, int W, int k, int T,
                                                       int X) {
    ClusterLayout L;
    size_t o = align_up((size_t)d * 2, 16);  // the reference vector (bf16)
    L.tok = (uint32_t)o;
    o = align_up(o + 4 * ((size_t)span + 1), 16);
    L.cnt = (uint32_t)o;  // this CTA's occurrences per branch
    o += 4 * (size_t)W;
    L.lst = (uint32_t)o;  // [W][k], most recent first
    o += 4 * (size_t)W * k;
    L.mcnt = (uint32_t)o;  // merged over the cluster
    o += 4 * (size_t)W;
    L.mlst = (uint32_t)o;
    o += 4 * (size_t)W * k;
    L.wc = (uint32_t)o;  // scan scratch: matches per (warp, branch)
    o += 4 * (size_t)(kThreads4 / 32) * W;
    L.sc = (uint32_t)o;  // rank 0: every task's score
    o += 4 * (size_t)T;
    L.tk = (uint32_t)o;  // rank 0: the token after every task's row
    o += 4 * (size_t)T;
    const int P = row_parts(d);
    L.pd = (uint32_t)o;  // rank 0: partial <row, ref> per (task, part)
    o += 4 * (size_t)T * P;
    L.ps = (uint32_t)o;  // rank 0: partial |row|^2 per (task, part)
    o += 4 * (size_t)T * P;
    L.gath = (uint32_t)o;  // every CTA's lists, [X][W][1 + k] (when pushed)
    if (push_bytes(X, W, k) <= kPushBytes) o += push_bytes(X, W, k);
    L.total = (uint32_t)o;
    return L;
}

struct ClusterArgs {
    TreeLaunch p;
    int span;  // history positions per CTA (<= kSlice4)
    int T;     // scored rows per sequence at most
    int32_t *dev_status;  // the workspace's status word (checked build)
};

template <int U>
__global__ void __launch_bounds__(kThreads4, U == 8 ? 2 : 1) tree_cluster_kernel(ClusterArgs args) {
    const TreeLaunch &a = args.p;
    __shared__ TreeSmem sm;
    extern __shared__ __align__(16) uint8_t dyn[];
    const int k = a.p.k, d = a.d, W = a.p.branch_width;
    const ClusterLayout L = cluster_layout(d, args.span, W, k, args.T, gridDim.x);
    uint16_t *s_ref = (uint16_t *)dyn;
    int *s_tok = (int *)(dyn + L.tok);
    int *s_cnt = (int *)(dyn + L.cnt);
    int *s_lst = (int *)(dyn + L.lst);
    int *s_mcnt = (int *)(dyn + L.mcnt);
    int *s_mlst = (int *)(dyn + L.mlst);
    int *s_wc = (int *)(dyn + L.wc);
    int *s_gath = (int *)(dyn + L.gath);
    float *s_sc = (float *)(dyn + L.sc);
    int *s_tk = (int *)(dyn + L.tk);
    float *s_pd = (float *)(dyn + L.pd);
    float *s_ps = (float *)(dyn + L.ps);
    int *s_cand = sm.cand;
    float *s_score = sm.score;

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nwarps = kThreads4 / 32;
    const int b = blockIdx.y, x = blockIdx.x, X = gridDim.x;
    const int gwarp = x * nwarps + warp, gwarps = X * nwarps;  // the cluster's warps
    const uint32_t flags = a.p.flags;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const uint16_t *R = a.reps + (int64_t)b * a.ld * d;
    pdl_wait_then_release();
    // every CTA of the cluster has started before another writes its shared
    // memory (the wait is in P1)
    cluster_arrive_relaxed();

    // ---- P0: the slice [p0, p0 + span] (clipped at ld) while the outcome is read
    const int64_t p0 = (int64_t)x * args.span;
    const int nld = p0 < a.ld ? (int)min((int64_t)args.span + 1, a.ld - p0) : 0;
    for (int i = t; i < nld; i += kThreads4) cp_async4(s_tok + i, M + p0 + i);
    const SeqView v = view_of(a, b);
    const int status0 = (a.status && t == 0 && x == 0) ? a.status[b] : 0;
    if (t < kMaxK) sm.slot[t] = t;
    if (t < v.nc) {
        s_cand[t] = v.cand_t;
        s_score[t] = v.score_t;
    }
    __syncthreads();
    const bool whole = X == 1;                      // the slice is the whole history
    const bool rank_first = v.rr && v.need_succ;    // reranked before the branch set
    const bool rerank_only = v.rr && !v.need_succ;  // reranked in P5
    const bool use_win = !whole && v.nc > 0 && (v.lex || v.branch_on);
    if (rank_first || rerank_only)
        vec_issue(a.query + (int64_t)b * d, d, s_ref);
    else if (v.need_succ)
        vec_issue(R + (int64_t)(s_cand[0] + 1) * d, d, s_ref);
    if (use_win && t < v.nc * kWin) {  // M[c+1 .. c+kWin] of each candidate c
        const int r = t / kWin, o = t - r * kWin;
        const int p = s_cand[r] + 1 + o;
        sm.win[r][o] = p <= v.len - 1 ? __ldg(M + p) : -1;
    }
    int32_t *dst = args.dev_status;
    auto tok_of = [&](int p) {  // M[p], from the slice where it is staged
        if (!idx_ok(p, 0, v.len, dst)) return -1;
        const int64_t q = p - p0;
        return (q >= 0 && q < nld) ? s_tok[q] : __ldg(M + p);
    };

    // ---- P1: the rerank the branch set depends on
    if (rank_first) {
        cluster_wait();
        const float qss = vec_finish(s_ref, d, s_red_of(sm));
        for (int q = gwarp; q < v.nc; q += gwarps) {
            float dot = 0.f, ss = 0.f;
            if (idx_ok(s_cand[q], 0, v.len - 1, dst))
                warp_row_dot<U>(R + (int64_t)s_cand[q] * d, s_ref, d, dot, ss);
            if (lane == 0) st_cluster_f32(&s_sc[q], 0, cosine_from(dot, ss, qss));
        }
        cluster_sync_all();
        if (t < v.nc) s_score[t] = ld_cluster_f32(&s_sc[t], 0);
        __syncthreads();
        if (warp == 0) warp_sort_desc(s_cand, s_score, v.nc, sm.slot);
        __syncthreads();
        vec_issue(R + (int64_t)(s_cand[0] + 1) * d, d, s_ref);  // the successor reference
    } else {
        cluster_wait();
        cp_async_wait_all();
        __syncthreads();  // the slice and the windows are visible
    }

    // ---- P2: the branch set; P3: this slice's occurrences of each branch token
    int nb = 0;
    if (v.need_succ) {
        nb = branch_set(a, b, v, s_cand, sm.next, sm.br, sm.misc,
                        TokSrc{whole ? s_tok : nullptr, use_win ? &sm : nullptr});
        const int64_t p1 = min(p0 + args.span, (int64_t)v.len - 1);  // positions <= len-2
        scan_branches(
            s_tok, p0, p0, p1, sm.br, nb, k, s_wc,
            [&](int w, int rank, int p) {
                if (idx_ok(rank, 0, k, dst) && idx_ok(w, 0, nb, dst) && idx_ok(p, p0, p1, dst))
                    s_lst[w * k + rank] = p;
            },
            [&](int w, int c) { s_cnt[w] = c; });
    }
    // with room for them, this slice's lists go into every CTA's shared
    // memory (slot x of [X][W][1 + k]) before the barrier, so the merge reads
    // local memory only
    const bool push = push_bytes(X, W, k) <= kPushBytes;
    if (push && v.need_succ) {
        __syncthreads();  // this CTA's lists are complete
        const int per = nb * (1 + k);
        for (int i = t; i < X * per; i += kThreads4) {
            const int r = i / per, j = i - r * per, w = j / (1 + k), e = j - w * (1 + k);
            const int val = e == 0 ? s_cnt[w] : s_lst[w * k + e - 1];
            st_cluster_i32(&s_gath[(x * W + w) * (1 + k) + e], r, val);
        }
    }
    cluster_sync_all();  // every slice's lists are complete (and pushed)

    // ---- P4: the successor candidates of each branch, most recent first
    if (v.need_succ) {
        for (int w = warp; w < nb; w += nwarps) {
            int total;
            if (push)
                total = warp_merge_desc(
                    X, k, [&](int r) { return s_gath[(r * W + w) * (1 + k)]; },
                    [&](int r, int i) { return s_gath[(r * W + w) * (1 + k) + 1 + i]; },
                    s_mlst + w * k);
            else
                total = warp_merge_desc(
                    X, k, [&](int r) { return ld_cluster_i32(&s_cnt[w], r); },
                    [&](int r, int i) { return ld_cluster_i32(&s_lst[w * k + i], r); },
                    s_mlst + w * k);
            if (lane == 0) s_mcnt[w] = total;
        }
        __syncthreads();
    }

    // ---- P5: the scored rows over the cluster's warps, in parts; the partial
    // sums (and the token after each row) go to rank 0
    const int ntasks = v.need_succ ? nb * k : (rerank_only ? v.nc : 0);
    const int nch = d >> 3, P = row_parts(d);
    float rss = 0.f;
    if (ntasks > 0) {
        auto row_of = [&](int task) {
            const int w = task / k, i = task - w * k;
            const int row = !v.need_succ ? s_cand[task] : (i < s_mcnt[w] ? s_mlst[task] : -1);
            return idx_ok(row, -1, v.len - 1, dst) ? row : -1;
        };
        // item = (task, part); a warp's items are gwarp, gwarp + gwarps, ...
        auto part_dot = [&](int row, int part, uint4 (&w)[U], bool loaded, float &dot,
                            float &ss) {
            const uint16_t *rp = R + (int64_t)row * d;
            const int base = part * kPartCh, end = min(base + kPartCh, nch);
            dot = 0.f;
            ss = 0.f;
            for (int c0 = base; c0 < end; c0 += 32 * U) {
                if (!(loaded && c0 == base)) row_batch_load<U>(rp, end, c0, w);
                row_batch_acc<U>(w, s_ref, end, c0, dot, ss);
            }
            dot = warp_sum(dot);
            ss = warp_sum(ss);
        };
        const int items = ntasks * P;
        const int task0 = gwarp / P, part0 = gwarp - task0 * P;
        const int row0 = gwarp < items ? row_of(task0) : -1;
        uint4 w0[U];
        if (row0 >= 0)
            row_batch_load<U>(R + (int64_t)row0 * d, min(part0 * kPartCh + kPartCh, nch),
                              part0 * kPartCh, w0);
        const int tk0 = (v.need_succ && row0 >= 0 && part0 == 0 && lane == 0)
                            ? tok_of(row0 + 1) : -1;
        rss = vec_finish(s_ref, d, s_red_of(sm));
        for (int it = gwarp; it < items; it += gwarps) {
            const int task = it / P, part = it - task * P;
            const int row = it == gwarp ? row0 : row_of(task);
            float dot = 0.f, ss = 0.f;
            if (row >= 0) part_dot(row, part, w0, it == gwarp, dot, ss);
            if (lane == 0 && idx_ok(it, 0, (int64_t)args.T * P, dst)) {
                st_cluster_f32(&s_pd[it], 0, dot);
                st_cluster_f32(&s_ps[it], 0, ss);
                if (v.need_succ && part == 0)
                    st_cluster_i32(&s_tk[task], 0,
                                   it == gwarp ? tk0 : (row >= 0 ? tok_of(row + 1) : -1));
            }
        }
    }
    cp_async_wait_all();  // (a reference row staged for no row: done before any exit)
    cluster_sync_all();  // rank 0 holds every score; no CTA reads another's memory after this
    if (x != 0) return;

    // ---- P6 (rank 0): the cosines from the partial sums (parts in order), rank,
    // branch, pick successors, emit
    for (int task = t; task < ntasks; task += kThreads4) {
        float dot = 0.f, ss = 0.f;
        for (int part = 0; part < P; ++part) {
            dot += s_pd[task * P + part];
            ss += s_ps[task * P + part];
        }
        const bool real = v.need_succ ? (task - (task / k) * k) < s_mcnt[task / k] : true;
        s_sc[task] = real ? cosine_from(dot, ss, rss) : -INFINITY;
    }
    __syncthreads();
    if (rerank_only) {
        if (t < v.nc) s_score[t] = s_sc[t];
        __syncthreads();
        if (warp == 0) warp_sort_desc(s_cand, s_score, v.nc, sm.slot);
        __syncthreads();
    } else if (v.lex && (flags & ADAPLD_NO_LEX_RERANK)) {
        if (t < v.nc) s_score[t] = __int_as_float(0x7fc00000);  // NaN: not computed
        __syncthreads();
    }
    if (v.branch_on && !v.need_succ)
        nb = branch_set(a, b, v, s_cand, sm.next, sm.br, sm.misc,
                        TokSrc{whole ? s_tok : nullptr, use_win ? &sm : nullptr});
    if (v.need_succ) {
        for (int w = warp; w < nb; w += nwarps) {  // Eq. 14: argmax per branch
            const bool in = lane < s_mcnt[w];
            float bs = in ? s_sc[w * k + lane] : -INFINITY;
            int bj = in ? s_mlst[w * k + lane] : -1;
            int btk = in ? s_tk[w * k + lane] : -1;
#pragma unroll
            for (int o = 16; o; o >>= 1) {
                const float os = __shfl_xor_sync(0xffffffffu, bs, o);
                const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
                const int ot = __shfl_xor_sync(0xffffffffu, btk, o);
                if (better(os, oj, bs, bj)) {
                    bs = os;
                    bj = oj;
                    btk = ot;
                }
            }
            if (lane == 0) {
                sm.succ[w] = bj >= 0 ? bj : -1;
                sm.stok[w] = btk;
            }
        }
        __syncthreads();
    }
    emit_tree(a, b, v, sm, TokSrc{whole ? s_tok : nullptr, nullptr}, use_win, nb, status0, dst);
}

}  // namespace

// Successor rows per sequence up to which the fused kernel scores them in the
// CTA that completes the scan (one row per warp, as a tree-kernel CTA would)
// instead of a tree kernel spreading them over CTAs.  Measured on GB300: with
// 16 rows (configs 1 and 4) fusing saves 2.4-2.7 us per step; with 24 or 64
// rows (configs 2 and 3) the second kernel's parallel rows win by 4-14 us.
constexpr int kMaxFusedTasks = kRowsPerCta5;
static_assert(kMaxFusedTasks <= kMaxK, "fused lists live in TreeSmem::lpos");

// The cluster kernel's shape for this launch: CTAs per sequence (enough for
// every slice of 8192 positions and, up to 8 -- or 16 when the grid then
// still fits one CTA per SM -- one warp per scored row) and positions per CTA.
// Returns false where it does not apply (token-embedding mode, whose
// successor backoff runs between the scan and the scoring; histories of more
// than 16 slices; shared memory beyond one SM).
bool cluster_shape(const TreeLaunch &a, int sms, int tasks, int *X, int *span, size_t *smem) {
    if (a.emb.table) return false;
    if (const char *e = std::getenv("ADAPLD_TREE_CLUSTER"))  // A/B switch for measurements
        if (e[0] == '0') return false;
    const int S = chunks_of(a.ld - 1, kSlice4);
    if (S > kWideClusterL) return false;
    const int R = (tasks + kRowsPerCta5 - 1) / kRowsPerCta5;
    const int cap = (int64_t)a.B * kWideClusterL <= sms ? kWideClusterL : kMaxClusterL;
    int x = R < cap ? R : cap;
    if (x < S) x = S;
    // one CTA per sequence: the older single kernel (succ_scan_kernel<U, true>)
    // measured faster (config 4: 21.2 against 25.2 us; config 1: 12.9 against
    // 15.0)
    if (x < 2) return false;
    const int64_t n = a.ld - 1;
    int sp = (int)((n + x - 1) / x);
    if (sp < 1) sp = 1;
    const size_t dyn =
        cluster_layout(a.d, sp, a.p.branch_width, a.p.k, tasks, x).total;
    if (dyn + sizeof(TreeSmem) > 227 * 1024) return false;
    *X = x;
    *span = sp;
    *smem = dyn;
    return true;
}

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
    int X = 0, span = 0;
    size_t csmem = 0;
    if (cluster_shape(a, sms, tasks, &X, &span, &csmem)) {  // the stage as one kernel
        ClusterArgs ca{a, span, tasks, ws.dev_status};
        // 16 row loads in flight per lane (one CTA per SM) while the grid fits
        // one wave; not with clusters of 16, of which only 7 are resident at
        // one CTA per SM on GB300 (config 5's 8 sequences took two waves)
        auto kern = ((int64_t)X * a.B <= sms && X <= kMaxClusterL) ? tree_cluster_kernel<16>
                                                                   : tree_cluster_kernel<8>;
        cudaError_t e =
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)csmem);
        if (e != cudaSuccess) return e;
        if (X > kMaxClusterL) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e != cudaSuccess) return e;
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(X, a.B);
        cfg.blockDim = dim3(kThreads4);
        cfg.dynamicSmemBytes = csmem;
        cfg.stream = s;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = X;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = X > 1 ? 2 : 1;  // a plain launch is a cluster of one CTA
        return counted(cudaLaunchKernelEx(&cfg, kern, ca));
    }
    const size_t vsmem = (size_t)a.d * sizeof(uint16_t);  // the staged query / reference row
    const size_t ssmem = vsmem + (size_t)(kSlice4 + 1) * sizeof(int);  // + a slice's tokens
    if (succ_possible) {
        cudaError_t e;
        if (!a.emb.table && W * k <= kMaxFusedTasks) {  // scan and tree in one kernel
            auto kern = (int64_t)ws.S4 * a.B <= sms ? succ_scan_kernel<16, true>
                                                    : succ_scan_kernel<8, true>;
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)ssmem);
            if (e != cudaSuccess) return e;
            return launch_dependent(kern, dim3(ws.S4, a.B), dim3(kThreads4), ssmem, s, args);
        }
        if (a.emb.table && !a.lists_ready) {  // distinct-token lists for the backoff
            DedupeLaunch da{a.tokens, a.ld,  a.lengths, a.B,     a.emb.vocab, nullptr, nullptr,
                            a.status, true, false,     nullptr, false,       k,       nullptr,
                            nullptr,  nullptr};
            e = launch_dedupe(da, ws, s);
            if (e != cudaSuccess) return e;
        }
        e = cudaFuncSetAttribute(succ_scan_kernel<8, false>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ssmem);
        if (e != cudaSuccess) return e;
        e = launch_dependent(succ_scan_kernel<8, false>, dim3(ws.S4, a.B), dim3(kThreads4), ssmem,
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
