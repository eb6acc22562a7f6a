// Rerank and draft-tree construction (Sec. 3.4-3.6, Eq. 6-15, Algorithm 1).
//
// Grid (S4 slices, B sequences), 512 threads.
//  1. Every participating CTA of a sequence rebuilds the anchor and branch set:
//     lexical hits are reranked by Eq. 6 (one warp per candidate row, the
//     query in shared memory as fp32), semantic hits keep their Eq. 4 order;
//     j* = the first candidate; branch tokens come from the caller's cached
//     next-token table row at j* or, without one, are the first W distinct
//     continuation tokens of the ranked candidates; Eq. 11 removes the main
//     path's first token on a lexical hit.
//  2. When successor drafting applies (Algorithm 1: semantic hits; or every
//     hit under ADAPLD_SUCC_ON_STRICT) the token history is cut into slices
//     of 8192 positions, one CTA each; a warp per branch token scans its slice
//     backwards with ballots and keeps the k most recent occurrences.  The
//     last slice CTA (atomic ticket) merges them, scores every occurrence t by
//     cos(R[t], R[j*+1]) (Eq. 13) and keeps the argmax (Eq. 14).
//  3. The finishing CTA lays out the tree (root, main chain, branch paths with
//     their successors) and writes tokens, parents, position ids and the
//     ancestor mask.  Without successor drafting only slice 0 does any work.
#include "common.cuh"

namespace adapld {

namespace {

struct TreeArgs {
    TreeLaunch p;
    Workspace ws;
};

// <row, ref> and |row|^2 of one bf16 row against an fp32 vector in shared
// memory; one warp, 8 independent 16-byte loads per lane in flight.
__device__ __forceinline__ void warp_row_dot(const uint16_t *row, const float *ref, int d,
                                             float &dot_out, float &ss_out) {
    const int lane = threadIdx.x & 31;
    const int nch = d >> 3;
    float dot = 0.f, ss = 0.f;
    for (int base = 0; base < nch; base += 32 * 8) {
        uint4 w[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int ch = base + u * 32 + lane;
            w[u] = ch < nch ? ldg_nc_v4(row + (size_t)ch * 8) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
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
        float x[8] = {bf16lo(w.x), bf16hi(w.x), bf16lo(w.y), bf16hi(w.y),
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

__global__ void __launch_bounds__(kThreads4) tree_kernel(TreeArgs args) {
    const TreeLaunch &a = args.p;
    const Workspace &ws = args.ws;
    extern __shared__ __align__(16) float dsm[];
    const int d = a.d, k = a.p.k, W = a.p.branch_width, D = a.p.draft_len;
    const int succ_len = a.p.succ_len;
    const uint32_t flags = a.p.flags;
    float *vec = dsm;                                  // [d]   query, then R[j*+1]
    int *s_tok = (int *)(vec + d);                     // [kSlice4]
    int *s_sc = s_tok + kSlice4;                       // [kMaxW * kMaxK]
    float *s_ss = (float *)(s_sc + kMaxW * kMaxK);     // [kMaxW * kMaxK]
    int *node_par = (int *)(s_ss + kMaxW * kMaxK);     // [kMaxNodes]
    int *node_depth = node_par + kMaxNodes;            // [kMaxNodes]
    int *node_path = node_depth + kMaxNodes;           // [kMaxNodes]
    int *node_src = node_path + kMaxNodes;             // [kMaxNodes]
    __shared__ int s_cand[kMaxK];
    __shared__ float s_score[kMaxK];
    __shared__ int s_next[kMaxW];
    __shared__ int s_br[kMaxW];
    __shared__ int s_scn[kMaxW];
    __shared__ int s_succ[kMaxW];
    __shared__ float scratch[32];
    __shared__ int s_nb, s_main0, s_flag, s_n, s_ext;

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nwarps = kThreads4 / 32;
    const int b = blockIdx.y, sl = blockIdx.x;
    const int len = a.lengths[b];
    const bool valid = len >= 1 && (int64_t)len <= a.ld;
    // candidates come from the caller on the standalone path: check the range
    bool cand_ok = true;
    const int nc0 = valid ? min(a.n_cand[b], k) : 0;
    for (int i = 0; i < nc0; ++i) {
        const int c = a.cand[(int64_t)b * k + i];
        cand_ok &= c >= 0 && c <= len - 2;
    }
    const int hk = (valid && cand_ok) ? a.hit_kind[b] : ADAPLD_HIT_NONE;
    const int nc = cand_ok ? nc0 : 0;
    const bool lex = hk == ADAPLD_HIT_LEX && nc > 0;
    const bool sem = hk == ADAPLD_HIT_SEM && nc > 0;
    const bool branch_on = !(flags & ADAPLD_NO_BRANCH) && W > 0 && (lex || sem);
    const bool need_succ = branch_on && !(flags & ADAPLD_NO_SUCC) &&
                           (sem || (lex && (flags & ADAPLD_SUCC_ON_STRICT)));
    if (!need_succ && sl != 0) return;

    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const uint16_t *R = a.reps + (int64_t)b * a.ld * d;

    // ---- 1. anchor and branch set ------------------------------------------------
    if (t < nc) {
        s_cand[t] = a.cand[(int64_t)b * k + t];
        s_score[t] = a.score[(int64_t)b * k + t];
    }
    __syncthreads();
    if (lex) {
        if (!(flags & ADAPLD_NO_LEX_RERANK)) {
            const float qss = block_load_vec(a.query + (int64_t)b * d, vec, d, scratch);
            for (int ci = warp; ci < nc; ci += nwarps) {
                float dot, ss;
                warp_row_dot(R + (int64_t)s_cand[ci] * d, vec, d, dot, ss);
                if (lane == 0) s_score[ci] = cosine_from(dot, ss, qss);
            }
            __syncthreads();
            if (warp == 0) {  // sort by (score desc, position desc)
                const float sc = lane < nc ? s_score[lane] : -INFINITY;
                const int cj = lane < nc ? s_cand[lane] : -1;
                int rank = 0;
                for (int m = 0; m < nc; ++m) {
                    const float os = __shfl_sync(0xffffffffu, sc, m);
                    const int oj = __shfl_sync(0xffffffffu, cj, m);
                    rank += better(os, oj, sc, cj) ? 1 : 0;
                }
                __syncwarp();
                if (lane < nc) {
                    s_cand[rank] = cj;
                    s_score[rank] = sc;
                }
            }
        } else if (t < nc) {
            s_score[t] = __int_as_float(0x7fc00000);  // NaN: not computed
        }
        __syncthreads();
    }
    const int js = (lex || sem) ? s_cand[0] : -1;
    if (branch_on) {
        if (a.next_topk) {
            const int32_t *row = a.next_topk + ((int64_t)b * a.ld + js) * a.Kn;
            if (t < a.Kn) s_next[t] = row[t];
        } else if (t < nc) {
            s_next[t] = M[s_cand[t] + 1];
        }
        if (t == kThreads4 - 1) s_main0 = lex ? M[js + 1] : -1;
        __syncthreads();
        if (t == 0) {
            int nb = 0;
            if (a.next_topk) {
                for (int r = 0; r < a.Kn && nb < W; ++r)
                    if (s_next[r] >= 0) s_br[nb++] = s_next[r];
            } else {
                for (int r = 0; r < nc && nb < W; ++r) {
                    const int tkn = s_next[r];
                    bool dup = false;
                    for (int e = 0; e < nb; ++e) dup |= s_br[e] == tkn;
                    if (!dup) s_br[nb++] = tkn;
                }
            }
            if (lex) {  // Eq. 11
                int m = 0;
                for (int e = 0; e < nb; ++e)
                    if (s_br[e] != s_main0) s_br[m++] = s_br[e];
                nb = m;
            }
            s_nb = nb;
        }
    } else if (t == 0) {
        s_nb = 0;
    }
    __syncthreads();
    const int nb = s_nb;

    // ---- 2. successor candidates over this slice ----------------------------------
    if (need_succ) {
        const int p0 = sl * kSlice4;
        const int p1 = min(p0 + kSlice4, len - 1);  // positions t <= len-2
        for (int i = t; i < p1 - p0; i += kThreads4) s_tok[i] = M[p0 + i];
        __syncthreads();
        for (int w = warp; w < nb; w += nwarps) {
            const int bt = s_br[w];
            int32_t *pp = ws.part4 + (((int64_t)b * ws.S4 + sl) * ws.W + w) * kPart4Ints;
            int cnt = 0;
            for (int top = p1 - 1; top >= p0 && cnt < k; top -= 32) {
                const int p = top - lane;
                const bool hit = p >= p0 && s_tok[p - p0] == bt;
                const unsigned m = __ballot_sync(0xffffffffu, hit);
                const int rank = cnt + __popc(m & ((1u << lane) - 1u));
                if (hit && rank < k) pp[1 + rank] = p;
                cnt += __popc(m);
            }
            if (lane == 0) pp[0] = min(cnt, k);
        }
        __threadfence();
        __syncthreads();
        if (t == 0) s_flag = atomicAdd(ws.ticket4 + b, 1) == (int)gridDim.x - 1;
        __syncthreads();
        if (!s_flag) return;
        __threadfence();
        // merge the slices, most recent first
        for (int w = warp; w < nb; w += nwarps) {
            int total = 0;
            for (int s2 = (int)gridDim.x - 1; s2 >= 0 && total < k; --s2) {
                const int32_t *pp = ws.part4 + (((int64_t)b * ws.S4 + s2) * ws.W + w) * kPart4Ints;
                const int n = __ldcg(pp);
                const int take = min(n, k - total);
                if (lane < take) s_sc[w * kMaxK + total + lane] = __ldcg(pp + 1 + lane);
                total += take;
            }
            if (lane == 0) s_scn[w] = total;
        }
        __syncthreads();
        // Eq. 13-14: rerank the occurrences against R[j*+1]
        const float rss = block_load_vec(R + (int64_t)(js + 1) * d, vec, d, scratch);
        for (int task = warp; task < nb * kMaxK; task += nwarps) {
            const int w = task / kMaxK, i = task % kMaxK;
            if (i >= s_scn[w]) continue;
            float dot, ss;
            warp_row_dot(R + (int64_t)s_sc[w * kMaxK + i] * d, vec, d, dot, ss);
            if (lane == 0) s_ss[w * kMaxK + i] = cosine_from(dot, ss, rss);
        }
        __syncthreads();
        for (int w = warp; w < nb; w += nwarps) {
            const int n = s_scn[w];
            float bs = lane < n ? s_ss[w * kMaxK + lane] : -INFINITY;
            int bj = lane < n ? s_sc[w * kMaxK + lane] : -1;
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

    // ---- 3. the tree ----------------------------------------------------------------
    const int N = 1 + D + W * (1 + succ_len);
    if (t == 0) {
        int n = 0, ext = 0;
        if (valid) {
            node_par[0] = -1;
            node_depth[0] = 0;
            node_path[0] = 0;
            node_src[0] = len - 1;
            n = 1;
            if (lex) {
                const int l = min(D, len - 1 - js);
                for (int i = 0; i < l; ++i, ++n) {
                    node_par[n] = i == 0 ? 0 : n - 1;
                    node_depth[n] = i + 1;
                    node_path[n] = 1;
                    node_src[n] = js + 1 + i;
                }
            }
            for (int w = 0; w < nb; ++w) {
                const int bnode = n;
                node_par[n] = 0;
                node_depth[n] = 1;
                node_path[n] = 2 + w;
                node_src[n] = -2 - w;  // the branch token itself
                ++n;
                if (need_succ && s_succ[w] >= 0) {
                    const int tb = s_succ[w];
                    int added = 0;
                    for (int i = 1; i <= succ_len && tb + i <= len - 1; ++i, ++n, ++added) {
                        node_par[n] = n - 1;
                        node_depth[n] = 1 + i;
                        node_path[n] = 2 + w;
                        node_src[n] = tb + i;
                    }
                    (void)bnode;
                    if (added > 0) ++ext;
                }
            }
        }
        s_n = n;
        s_ext = ext;
    }
    __syncthreads();
    const int n = s_n;
    const int64_t ob = (int64_t)b * N;
    for (int i = t; i < N; i += kThreads4) {
        int tok = -1, par = -1, pos = -1;
        if (i < n) {
            const int src = node_src[i];
            tok = src >= 0 ? M[src] : s_br[-2 - src];
            par = node_par[i];
            pos = len - 1 + node_depth[i];
        }
        a.out.draft_tokens[ob + i] = tok;
        a.out.parents[ob + i] = par;
        a.out.positions[ob + i] = pos;
    }
    uint8_t *mk = a.out.mask + (int64_t)b * N * N;
    for (int idx = t; idx < N * N; idx += kThreads4) {
        const int i = idx / N, j = idx % N;
        const bool anc = i < n && j < n &&
                         (j == 0 || (node_path[i] == node_path[j] && j <= i && node_path[i] != 0) ||
                          j == i);
        mk[idx] = anc ? 1 : 0;
    }
    if (lex && t < k) {
        a.cand[(int64_t)b * k + t] = t < nc ? s_cand[t] : -1;
        a.score[(int64_t)b * k + t] = t < nc ? s_score[t] : 0.f;
    }
    if (t == 0) {
        a.out.anchor[b] = js;
        a.out.n_nodes[b] = n;
        if (a.out.stats) {
            atomicAdd(a.out.stats + (lex ? 0 : (sem ? 1 : 2)), 1);
            if (s_ext) atomicAdd(a.out.stats + 3, s_ext);
        }
        if (a.status)
            a.status[b] = (valid ? 0 : ADAPLD_SEQ_BAD_LENGTH) | (cand_ok ? 0 : ADAPLD_SEQ_BAD_CANDIDATE);
    }
}

}  // namespace

size_t tree_smem_bytes(int d) {
    return (size_t)d * 4 + (size_t)kSlice4 * 4 + 2 * (size_t)kMaxW * kMaxK * 4 +
           4 * (size_t)kMaxNodes * 4;
}

cudaError_t launch_tree(const TreeLaunch &a, const Workspace &ws, cudaStream_t s) {
    TreeArgs args{a, ws};
    const size_t smem = tree_smem_bytes(a.d);
    cudaError_t e = cudaFuncSetAttribute(tree_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid(ws.S4, a.B);
    tree_kernel<<<grid, kThreads4, smem, s>>>(args);
    return cudaGetLastError();
}

}  // namespace adapld
