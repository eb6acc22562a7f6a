// Greedy verification of the draft trees and the append to the memory
// (Sec. 3.6; Appendix C, Eq. 16: at temperature 0 a draft token is accepted
// iff it equals the target model's greedy choice; Algorithm 1 appends the
// accepted tokens and the bonus token).
//
// The work is the argmax of every tree node's logit row (N rows of V bf16
// per sequence, HBM-bound), then a walk over at most N nodes.
//
// verify_kernel, grid (S splits, N nodes, B), 256 threads.  CTA (s, i, b)
// reads split s of node i's row in 32 KB groups (8 independent 16-byte
// loads per thread, all issued before any is used; groups s, s + S, ...)
// and stores the first index of the maximum as a 64-bit key that orders by
// value, then by the smaller index (S <= 1024 / N keeps the partial keys
// within the workspace).  CTAs of nodes >= n_nodes[b] exit at once.  No
// counters and no fences: walk_kernel, one CTA per sequence and launched as
// a programmatic dependent (so every key is visible), takes the largest key
// per node, loads the tree into shared memory, walks from the root with warp
// ballots (the child whose token equals the choice at the current node),
// writes the new tokens (accepted draft tokens, then the choice after the
// last accepted node) and appends them, with the hidden states of the root
// and the accepted nodes, to the memory.
#include <climits>

#include "common.cuh"

namespace adapld {

namespace {

constexpr int kThreadsV = 256;
constexpr int kLoadsV = 8;                          // 16-byte loads per thread
constexpr int kChunksV = kThreadsV * kLoadsV;       // 16-byte chunks per CTA (32 KB)

struct VerifyArgs {
    VerifyLaunch p;
    Workspace ws;
    int S;  // splits per row
};

// (value, index) order of the choice: higher value, then the smaller index.
__device__ __forceinline__ bool beats(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

// A key whose unsigned order is the choice order: the value's bits made
// monotone (negative values inverted, positive ones offset by the sign bit;
// -0 folded onto +0 so that the two tie), then the complemented index.
// Never 0 for a non-NaN value, so 0 means "no value yet".
__device__ __forceinline__ unsigned long long choice_key(float v, int i) {
    uint32_t u = __float_as_uint(v == 0.0f ? 0.0f : v);
    u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    return ((unsigned long long)u << 32) | (0xffffffffu - (uint32_t)i);
}

// Index of a key; a row without a non-NaN value chooses index 0.
__device__ __forceinline__ int key_index(unsigned long long key) {
    return key == 0ull ? 0 : (int)(0xffffffffu - (uint32_t)(key & 0xffffffffull));
}

__device__ __forceinline__ void take8(uint4 w, int i0, float &bv, int &bi) {
    const uint32_t w4[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float lo = bf16lo(w4[e]), hi = bf16hi(w4[e]);
        if (beats(lo, i0 + 2 * e, bv, bi)) {
            bv = lo;
            bi = i0 + 2 * e;
        }
        if (beats(hi, i0 + 2 * e + 1, bv, bi)) {
            bv = hi;
            bi = i0 + 2 * e + 1;
        }
    }
}

__global__ void __launch_bounds__(kThreadsV) verify_kernel(VerifyArgs args) {
    const VerifyLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ float s_v[kThreadsV / 32];
    __shared__ int s_i[kThreadsV / 32];

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int split = blockIdx.x, node = blockIdx.y, b = blockIdx.z;
    const int N = a.N, V = a.V, S = args.S;
    // the walk kernel may be scheduled now; it waits for this grid to finish
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int n = min(a.n_nodes[b], N);
    if (node >= n) return;  // (also every CTA of an empty tree)

    // ---- this split of the target's row after the node: first index of the maximum
    const uint16_t *row = a.logits + ((int64_t)b * N + node) * V;
    const int nch = V >> 3;
    float bv = -INFINITY;
    int bi = INT_MAX;
    for (int c0 = split * kChunksV; c0 < nch; c0 += S * kChunksV) {
        uint4 w[kLoadsV];
#pragma unroll
        for (int u = 0; u < kLoadsV; ++u) {
            const int ch = c0 + u * kThreadsV + t;
            if (ch < nch) w[u] = ldg_nc_v4(row + (size_t)ch * 8);
        }
#pragma unroll
        for (int u = 0; u < kLoadsV; ++u) {
            const int ch = c0 + u * kThreadsV + t;
            if (ch < nch) take8(w[u], ch * 8, bv, bi);
        }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (beats(ov, oi, bv, bi)) {
            bv = ov;
            bi = oi;
        }
    }
    if (lane == 0) {
        s_v[warp] = bv;
        s_i[warp] = bi;
    }
    __syncthreads();
    if (t == 0) {
        for (int k = 1; k < kThreadsV / 32; ++k)
            if (beats(s_v[k], s_i[k], bv, bi)) {
                bv = s_v[k];
                bi = s_i[k];
            }
        ws.vpart[((int64_t)b * N + node) * S + split] = bi < V ? choice_key(bv, bi) : 0ull;
    }
}

// walk_kernel, one CTA per sequence, launched as a programmatic dependent of
// verify_kernel (so every partial key is visible): the largest key per node,
// the walk, the new tokens and the append.
__global__ void __launch_bounds__(kThreadsV) walk_kernel(VerifyArgs args) {
    const VerifyLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ int s_tok[kMaxNodes], s_par[kMaxNodes], s_tgt[kMaxNodes];
    __shared__ int s_path[kMaxNodes];
    __shared__ int s_nacc;
    pdl_wait_then_release();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int b = blockIdx.x;
    const int N = a.N, S = args.S;
    const int n = min(a.n_nodes[b], N);
    int32_t *new_b = a.new_tokens + (int64_t)b * N;
    if (n <= 0) {  // an empty tree: nothing to verify or append
        for (int i = t; i < N; i += kThreadsV) new_b[i] = -1;
        if (t == 0) {
            a.n_accept[b] = 0;
            a.n_new[b] = 0;
            if (a.status) a.status[b] = 0;
        }
        return;
    }

    // ---- the last CTA of sequence b: walk the tree
    for (int i = t; i < n; i += kThreadsV) {
        s_tok[i] = a.draft_tokens[(int64_t)b * N + i];
        s_par[i] = a.parents[(int64_t)b * N + i];
        const unsigned long long *kp = ws.vpart + ((int64_t)b * N + i) * S;
        unsigned long long key = 0ull;
        for (int j0 = 0; j0 < S; j0 += 8) {  // eight partial keys in flight at a time
            unsigned long long kk[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) kk[j] = j0 + j < S ? __ldcg(kp + j0 + j) : 0ull;
#pragma unroll
            for (int j = 0; j < 8; ++j) key = max(key, kk[j]);
        }
        s_tgt[i] = key_index(key);
    }
    __syncthreads();
    if (warp == 0) {
        int cur = 0, acc = 0;
        for (;;) {
            const int want = s_tgt[cur];
            int next = -1;
            for (int base = 1; base < n && next < 0; base += 32) {
                const int i = base + lane;
                // a node has one parent and the search skips the root, so
                // the walk never revisits a node: it ends within n steps on
                // any parents[] (acc <= n - 1 keeps s_path in bounds)
                const unsigned m =
                    __ballot_sync(0xffffffffu, i < n && s_par[i] == cur && s_tok[i] == want);
                if (m) next = base + __ffs(m) - 1;
            }
            if (lane == 0) s_path[acc] = cur;
            if (next < 0) break;
            ++acc;
            cur = next;
        }
        if (lane == 0) s_nacc = acc;
    }
    __syncthreads();
    const int acc = s_nacc, n_new = acc + 1;
    // new tokens: the accepted nodes' tokens, then the choice after the last
    for (int i = t; i < N; i += kThreadsV) {
        int v = -1;
        if (i < acc)
            v = s_tok[s_path[i + 1]];
        else if (i == acc)
            v = s_tgt[s_path[acc]];
        new_b[i] = v;
    }
    int full = 0, bad = 0;
    if (a.tokens) {
        const int len = a.lengths[b];
        bad = len < 0 || (int64_t)len > a.ld;
        full = !bad && (int64_t)len + n_new > a.ld;
        if (!bad && !full) {
            int32_t *Mb = a.tokens + (int64_t)b * a.ld;
            for (int i = t; i < n_new; i += kThreadsV)
                Mb[len + i] = i < acc ? s_tok[s_path[i + 1]] : s_tgt[s_path[acc]];
            if (a.node_reps) {  // row len+i <- hidden state after the new position's predecessor
                const int nch = a.d >> 3;
                for (int idx = t; idx < n_new * nch; idx += kThreadsV) {
                    const int i = idx / nch, ch = idx % nch;
                    const uint4 r = ldg_nc_v4(a.node_reps + ((int64_t)b * N + s_path[i]) * a.d +
                                              (size_t)ch * 8);
                    *(uint4 *)(a.reps + ((int64_t)b * a.ld + len + i) * a.d + (size_t)ch * 8) = r;
                    if (i == n_new - 1)
                        *(uint4 *)(a.query + (int64_t)b * a.d + (size_t)ch * 8) = r;
                }
            }
        }
    }
    __syncthreads();  // every thread has read lengths[b] before it changes
    if (t == 0) {
        a.n_accept[b] = acc;
        a.n_new[b] = n_new;
        if (a.tokens && !full && !bad) a.lengths[b] += n_new;
        if (a.status) a.status[b] = (full ? ADAPLD_SEQ_FULL : 0) | (bad ? ADAPLD_SEQ_BAD_LENGTH : 0);
    }
}

}  // namespace

cudaError_t launch_verify(const VerifyLaunch &a, const Workspace &ws, cudaStream_t s) {
    const int groups = (int)(((int64_t)(a.V >> 3) + kChunksV - 1) / kChunksV);
    const int S = max(1, min(groups, kMaxNodes / a.N));
    VerifyArgs args{a, ws, S};
    verify_kernel<<<dim3(S, a.N, a.B), kThreadsV, 0, s>>>(args);
    cudaError_t e = counted(cudaGetLastError());
    if (e != cudaSuccess) return e;
    return launch_dependent(walk_kernel, dim3(a.B), dim3(kThreadsV), 0, s, args);
}

}  // namespace adapld
