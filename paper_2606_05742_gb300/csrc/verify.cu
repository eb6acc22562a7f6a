// Greedy verification of the draft trees and the append to the memory
// (Sec. 3.6; Appendix C, Eq. 16: at temperature 0 a draft token is accepted
// iff it equals the target model's greedy choice; Algorithm 1 appends the
// accepted tokens and the bonus token).
//
// verify_kernel, grid (N nodes, B), 512 threads.  CTA (i, b) streams the
// target's next-token logits after node i (V bf16, 16-byte loads) and keeps
// the first index of the maximum; CTAs of nodes >= n_nodes[b] exit.  The last
// CTA of a sequence (atomic ticket) loads the tree and the choices into
// shared memory, walks from the root with warp ballots (the child whose token
// equals the choice at the current node), writes the new tokens (accepted
// draft tokens, then the choice after the last accepted node) and appends
// them, with the hidden states of the root and the accepted nodes, to the
// memory.
#include <climits>

#include "common.cuh"

namespace adapld {

namespace {

constexpr int kThreadsV = 512;

struct VerifyArgs {
    VerifyLaunch p;
    Workspace ws;
};

// (value, index) order of the choice: higher value, then the smaller index.
__device__ __forceinline__ bool beats(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

__global__ void __launch_bounds__(kThreadsV) verify_kernel(VerifyArgs args) {
    const VerifyLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ float s_v[kThreadsV / 32];
    __shared__ int s_i[kThreadsV / 32];
    __shared__ int s_tok[kMaxNodes], s_par[kMaxNodes], s_tgt[kMaxNodes];
    __shared__ int s_path[kMaxNodes];
    __shared__ int s_flag, s_nacc;

    pdl_wait_then_release();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int node = blockIdx.x, b = blockIdx.y;
    const int N = a.N, V = a.V;
    const int n = min(a.n_nodes[b], N);
    int32_t *new_b = a.new_tokens + (int64_t)b * N;
    if (n <= 0) {  // an empty tree: nothing to verify or append
        if (node == 0) {
            for (int i = t; i < N; i += kThreadsV) new_b[i] = -1;
            if (t == 0) {
                a.n_accept[b] = 0;
                a.n_new[b] = 0;
                if (a.status) a.status[b] = 0;
            }
        }
        return;
    }
    if (node >= n) return;

    // ---- the target's choice after this node: first index of the maximum
    const uint16_t *row = a.logits + ((int64_t)b * N + node) * V;
    float bv = -INFINITY;
    int bi = INT_MAX;
    for (int ch = t; ch < (V >> 3); ch += kThreadsV) {
        const uint4 w = ldg_nc_v4(row + (size_t)ch * 8);
        const uint32_t w4[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float lo = bf16lo(w4[e]), hi = bf16hi(w4[e]);
            const int i0 = ch * 8 + 2 * e;
            if (beats(lo, i0, bv, bi)) {
                bv = lo;
                bi = i0;
            }
            if (beats(hi, i0 + 1, bv, bi)) {
                bv = hi;
                bi = i0 + 1;
            }
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
        for (int w = 1; w < kThreadsV / 32; ++w)
            if (beats(s_v[w], s_i[w], bv, bi)) {
                bv = s_v[w];
                bi = s_i[w];
            }
        ws.vtarget[(int64_t)b * kMaxNodes + node] = bi < V ? bi : 0;
        __threadfence();
        s_flag = atomicAdd(ws.vticket + b, 1) == n - 1;
    }
    __syncthreads();
    if (!s_flag) return;
    __threadfence();

    // ---- the last CTA of sequence b: walk the tree
    for (int i = t; i < n; i += kThreadsV) {
        s_tok[i] = a.draft_tokens[(int64_t)b * N + i];
        s_par[i] = a.parents[(int64_t)b * N + i];
        s_tgt[i] = __ldcg(ws.vtarget + (int64_t)b * kMaxNodes + i);
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
                    const uint4 w = ldg_nc_v4(a.node_reps + ((int64_t)b * N + s_path[i]) * a.d +
                                              (size_t)ch * 8);
                    *(uint4 *)(a.reps + ((int64_t)b * a.ld + len + i) * a.d + (size_t)ch * 8) = w;
                    if (i == n_new - 1)
                        *(uint4 *)(a.query + (int64_t)b * a.d + (size_t)ch * 8) = w;
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
    VerifyArgs args{a, ws};
    verify_kernel<<<dim3(a.N, a.B), kThreadsV, 0, s>>>(args);
    return cudaGetLastError();
}

}  // namespace adapld
