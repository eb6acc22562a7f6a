// Shared device helpers and the workspace layout of the AdaPLD sm_103a library.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "adapld.h"

namespace adapld {

// ---- limits and tiling ------------------------------------------------------
constexpr int kMaxK = 32;          // candidates per list (one per warp lane)
constexpr int kMaxW = 64;          // branch width
constexpr int kMaxNodes = 1024;    // draft-tree node slots
constexpr int kChunk1 = 4096;      // distinct-token lists: positions per CTA
constexpr int kThreads1 = 256;
constexpr int kChunkL = 8192;      // lexical scan: positions per chunk
constexpr int kThreadsL = 512;
constexpr int kMaxClusterL = 8;    // lexical scan: CTAs per sequence (one portable cluster)
constexpr int kWideClusterL = 16;  // ... when the whole grid fits one CTA per SM
constexpr int kPlanInKernelB = 288;  // below this B the semantic kernel derives its plan
constexpr int kSlice4 = 8192;      // successor scan: positions per CTA
constexpr int kThreads4 = 512;
constexpr int kMaxGrid2 = 1024;    // semantic kernel: CTAs at most
constexpr int kConsumers2 = 256;   // semantic kernel: consumer threads (8 warps)
constexpr int kMaxStages2 = 8;
constexpr int kSlotInts = 68;      // partial top-k slot: count, 32 ids, 32 scores (+pad)
constexpr int kPart4Ints = 1 + kMaxK;
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // bounded waits: 2 s

// ---- workspace --------------------------------------------------------------
// Counters (zeroed by every call) come first, then scratch that every call
// fully rewrites before reading.
struct Workspace {
    int32_t *dev_status;     // [1]  ADAPLD_DEV_* bits
    int32_t *done2;          // [B]  semantic kernel: CTAs done per sequence
    int32_t *ticket4;        // [B]  successor scan: slices done per sequence
    int32_t *ticket5;        // [B]  tree kernel: CTAs done per sequence
    int32_t *npairs;         // [1]  successor backoff: (sequence, branch) pairs
    int32_t *gticket_rep;    // [1]  distinct-token lists: sequences done (plan)
    int32_t *done3;          // [B*W] successor backoff: CTAs done per pair
    int32_t *rticket;        // [B]  distinct-token lists: chunks counted per sequence
    int32_t *xticket;        // [B]  expansion of the fallback lists: slices done
    int32_t *xticket2;       // [B*W] expansion of the backoff lists: slices done
    int64_t *plan;           // [B+1] prefix sums of semantic rows per sequence
    int32_t *slots2;         // [B + kMaxGrid2][kSlotInts] partial top-k lists
    int32_t *part4;          // [B][S4][W][kPart4Ints] per-slice successor lists
    int32_t *succ;           // [B][W][kMaxK] merged successor candidates
    int32_t *succ_n;         // [B][W] their counts
    int32_t *rr_cand;        // [B][kMaxK] reranked lexical candidates (successor scan)
    float *rr_score;         // [B][kMaxK] their scores
    float *score5;           // [B][W*kMaxK] scores computed by the tree kernel
    int32_t *tok5;           // [B][W*kMaxK] first successor token of each scored candidate
    int32_t *brs;            // [B][1 + W] branch count and branch tokens (successor scan)
    int64_t *plan3;          // [B*W+1] successor backoff plan
    int32_t *slots3;         // [B*W + kMaxGrid2][kSlotInts] its partial lists
    int32_t *pair_b;         // [B*W] real sequence of each backoff pair
    int32_t *pair_tok;       // [B*W] its branch token (the query anchor)
    int32_t *pair_out;       // [B*W] its row b*W + w in succ / succ_n
    float *succ_es;          // [B*W][kMaxK] backoff candidates' embedding scores
    unsigned long long *vpart;  // [B][N][S], N*S <= kMaxNodes: verification, packed
                                //   (logit, index) maximum per node and row split
    // distinct-token lists (two-representation mode): a row of the token-
    // embedding fallback depends only on the token, so each token of a
    // history is scored once
    unsigned long long *htab;   // [B][H] hash of (token + 1) << 32 | latest position
    int32_t *rep_tok;        // [B][ld] distinct tokens by latest position, then the anchor
    int32_t *rep_len;        // [B] distinct tokens + 1 (a length: rows = rep_len - 1)
    int32_t *rep_cnt;        // [B][C1] distinct tokens per chunk, then chunk offsets
    uint32_t *rep_bits;      // [B][C1][128] one bit per position: latest occurrence
    int32_t *xpart;          // [B*W][S4][kMaxK][kPart4Ints] expansion: per-slice lists
    // the union of the fallback sequences' distinct tokens (two-representation
    // mode, small batches: every table row is read once per step, not once per
    // sequence holding it); NULL where union_enabled() is false
    uint32_t *uhash;         // [UH] union bitmap (bit u: token u), after htab (one memset clears both)
    int32_t *ucount;         // [1]  union tokens (a counter)
    int32_t *ulist;          // [B * ld] the union's tokens, in no particular order
    int32_t *rep_pos;        // [B][ld] latest position of each listed token
    float *score_pos;        // [B][ld] Eq. 4 score of the token whose latest position it is
    int64_t UH;              // union bitmap words (a power of two >= 2 B (ld-1))
    int64_t H;               // hash slots per sequence (a power of two >= 2 (ld-1))
    size_t htab_bytes;       // htab and uhash
    size_t counters_bytes;
    size_t total_bytes;
    int C1, S4, W;
};

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

__host__ __device__ inline int chunks_of(int64_t n, int64_t per) {
    return (int)((n < 1 ? 1 : n + per - 1) / per);
}

// Hash slots per sequence for the distinct-token lists: a power of two of at
// least twice the candidate positions, so the load factor stays <= 1/2.
__host__ __device__ inline int64_t hash_slots(int64_t ld) {
    int64_t h = 64;
    while (h < 2 * (ld - 1)) h <<= 1;
    return h;
}

// The union pass of the two-representation fallback applies to batches of at
// most 16 sequences (its query slices then fit the stages of 4 KB row slices
// next to the rows; with more queries the per-sequence lists measured faster)
// whose positions its hash can hold.
constexpr int kUnionMaxB = 16;
__host__ __device__ inline bool union_enabled(int32_t B, int64_t ld) {
    return B <= kUnionMaxB && (int64_t)B * (ld - 1) <= ((int64_t)1 << 24);
}

// Lays the workspace out at `base` (NULL: sizing only).
inline Workspace layout_workspace(void *base, int32_t B, int64_t ld, int32_t W) {
    Workspace w{};
    w.C1 = chunks_of(ld - 1, kChunk1);
    w.S4 = chunks_of(ld - 1, kSlice4);
    w.W = W < 1 ? 1 : W;
    char *p = (char *)base;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *r = p ? p + off : nullptr;
        off = align_up(off + bytes, 256);
        return r;
    };
    const size_t BW = (size_t)B * w.W;
    w.counters_bytes = sizeof(int32_t) * (4 + 5 * (size_t)B + 2 * BW);
    w.dev_status = (int32_t *)take(w.counters_bytes);
    if (p) {
        w.npairs = w.dev_status + 1;
        w.gticket_rep = w.dev_status + 2;
        w.ucount = w.dev_status + 3;
        w.done2 = w.dev_status + 4;
        w.ticket4 = w.done2 + B;
        w.ticket5 = w.ticket4 + B;
        w.done3 = w.ticket5 + B;
        w.rticket = w.done3 + BW;
        w.xticket = w.rticket + B;
        w.xticket2 = w.xticket + B;
    }
    w.plan = (int64_t *)take(sizeof(int64_t) * ((size_t)B + 1));
    w.slots2 = (int32_t *)take(sizeof(int32_t) * ((size_t)B + kMaxGrid2) * kSlotInts);
    w.part4 = (int32_t *)take(sizeof(int32_t) * (size_t)B * w.S4 * w.W * kPart4Ints);
    w.succ = (int32_t *)take(sizeof(int32_t) * (size_t)B * w.W * kMaxK);
    w.succ_n = (int32_t *)take(sizeof(int32_t) * (size_t)B * w.W);
    w.rr_cand = (int32_t *)take(sizeof(int32_t) * (size_t)B * kMaxK);
    w.rr_score = (float *)take(sizeof(float) * (size_t)B * kMaxK);
    w.score5 = (float *)take(sizeof(float) * (size_t)B * w.W * kMaxK);
    w.tok5 = (int32_t *)take(sizeof(int32_t) * (size_t)B * w.W * kMaxK);
    w.brs = (int32_t *)take(sizeof(int32_t) * (size_t)B * (w.W + 1));
    w.plan3 = (int64_t *)take(sizeof(int64_t) * (BW + 1));
    w.slots3 = (int32_t *)take(sizeof(int32_t) * (BW + kMaxGrid2) * kSlotInts);
    w.pair_b = (int32_t *)take(sizeof(int32_t) * BW);
    w.pair_tok = (int32_t *)take(sizeof(int32_t) * BW);
    w.pair_out = (int32_t *)take(sizeof(int32_t) * BW);
    w.succ_es = (float *)take(sizeof(float) * BW * kMaxK);
    w.vpart = (unsigned long long *)take(sizeof(unsigned long long) * (size_t)B * kMaxNodes);
    w.H = hash_slots(ld);
    const bool uni = union_enabled(B, ld);
    w.UH = uni ? hash_slots((int64_t)B * (ld - 1) + 1) : 0;
    const size_t hbytes = sizeof(unsigned long long) * (size_t)B * w.H;
    w.htab_bytes = hbytes + sizeof(uint32_t) * (size_t)w.UH;
    w.htab = (unsigned long long *)take(w.htab_bytes);
    w.uhash = (p && uni) ? (uint32_t *)((char *)w.htab + hbytes) : nullptr;
    w.ulist = uni ? (int32_t *)take(sizeof(int32_t) * (size_t)B * ld) : nullptr;
    w.rep_pos = uni ? (int32_t *)take(sizeof(int32_t) * (size_t)B * ld) : nullptr;
    w.score_pos = uni ? (float *)take(sizeof(float) * (size_t)B * ld) : nullptr;
    w.rep_tok = (int32_t *)take(sizeof(int32_t) * (size_t)B * ld);
    w.rep_len = (int32_t *)take(sizeof(int32_t) * (size_t)B);
    w.rep_cnt = (int32_t *)take(sizeof(int32_t) * (size_t)B * w.C1);
    w.rep_bits = (uint32_t *)take(sizeof(uint32_t) * (size_t)B * w.C1 * (kChunk1 / 32));
    w.xpart = (int32_t *)take(sizeof(int32_t) * BW * w.S4 * kMaxK * kPart4Ints);
    w.total_bytes = off;
    return w;
}

// ---- device helpers ------------------------------------------------------------
#ifdef __CUDACC__

// The checked build (-DADAPLD_CHECKED: a debug library, build.build(checked=
// True)) tests every computed index below before the access it guards: a
// failed test raises ADAPLD_DEV_INTERNAL in the status word (nullable) and
// the access is skipped -- never a trap.  In the normal build the tests
// compile to nothing.
#ifdef ADAPLD_CHECKED
constexpr bool kChecked = true;
#else
constexpr bool kChecked = false;
#endif

// The table row a token id reads: ids outside [0, vocab) read row 0.
__device__ __forceinline__ int canon(int tok, int vocab) {
    return tok >= 0 && tok < vocab ? tok : 0;
}

// lowbias32, an integer hash published by C. Wellons (hash-prospector).
__device__ __forceinline__ uint32_t hash32(uint32_t x) {
    x ^= x >> 16;
    x *= 0x7feb352du;
    x ^= x >> 15;
    x *= 0x846ca68bu;
    x ^= x >> 16;
    return x;
}

// lo <= i < hi (always true in the normal build).
__device__ __forceinline__ bool idx_ok(int64_t i, int64_t lo, int64_t hi, int32_t *status) {
    if constexpr (!kChecked) {
        return true;
    } else {
        const bool ok = i >= lo && i < hi;
        if (!ok && status) atomicOr(status, ADAPLD_DEV_INTERNAL);
        return ok;
    }
}

// Programmatic dependent launch: wait until the previous kernel in the stream
// has completed and its writes are visible (a no-op when this kernel was not
// launched as a dependent), then allow the next kernel to begin launching.
// Calling the two in this order keeps completion transitive along the chain.
__device__ __forceinline__ void pdl_wait_then_release() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// The ranking order used everywhere: higher score first, ties to the larger
// (more recent) position.
__device__ __forceinline__ bool better(float sa, int ja, float sb, int jb) {
    return sa > sb || (sa == sb && ja > jb);
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Waits for the phase of `bar` with the given parity to complete; gives up
// after limit_ns and returns false.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity,
                                                  uint64_t limit_ns = kWaitLimitNs) {
    if (mbar_try_wait(bar, parity)) return true;
    uint64_t t0 = global_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (global_ns() - t0 > limit_ns) return false;
    }
    return true;
}

// One bulk (non-tensor) TMA copy global -> shared, completing on `bar`.
// Both addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}

__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ uint64_t l2_evict_normal_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ void named_bar_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

__device__ __forceinline__ void named_bar_arrive(int id, int count) {
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Asynchronous global -> shared copies (no registers held while in flight).
__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem)), "l"(gmem));
}
__device__ __forceinline__ void cp_async4(void *smem, const void *gmem) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(smem)), "l"(gmem));
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.wait_all;" ::: "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Thread-block clusters: a barrier over every thread of the cluster (release
// of this thread's earlier writes, acquire of the others'), and a 32-bit load
// from the shared memory of CTA `rank` of the cluster at the offset of
// `local` in this CTA's shared memory.
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// The two halves of a cluster barrier, for work placed between them.
__device__ __forceinline__ void cluster_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// The same barrier for a thread with no shared-memory writes to publish.
__device__ __forceinline__ void cluster_sync_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t cluster_addr(const void *local, uint32_t rank) {
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
    return remote;
}
__device__ __forceinline__ int ld_cluster_i32(const int *local, uint32_t rank) {
    int v;
    asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(cluster_addr(local, rank)) : "memory");
    return v;
}
__device__ __forceinline__ float ld_cluster_f32(const float *local, uint32_t rank) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(cluster_addr(local, rank)) : "memory");
    return v;
}
__device__ __forceinline__ void st_cluster_i32(int *local, uint32_t rank, int v) {
    asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(cluster_addr(local, rank)), "r"(v) : "memory");
}
__device__ __forceinline__ void st_cluster_f32(float *local, uint32_t rank, float v) {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(cluster_addr(local, rank)), "f"(v) : "memory");
}

__device__ __forceinline__ uint4 ldg_nc_v4(const void *p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Cosine from fp32 accumulators, zero when either norm is zero.
__device__ __forceinline__ float cosine_from(float dot, float ss, float qss) {
    return (ss > 0.f && qss > 0.f) ? dot / (sqrtf(ss) * sqrtf(qss)) : 0.f;
}

// Warp-resident top-k list: lane i < n holds the i-th best (s, j).
struct WarpTopK {
    float s;
    int j;
    int n;  // warp-uniform count

    __device__ __forceinline__ void reset() {
        s = -INFINITY;
        j = -1;
        n = 0;
    }

    // Inserts the candidates held by the lanes with `want` set.  All 32 lanes
    // must call.  k <= 32.
    __device__ __forceinline__ void insert(bool want, float cs, int cj, int k) {
        const int lane = threadIdx.x & 31;
        float ks = __shfl_sync(0xffffffffu, s, k - 1);
        int kj = __shfl_sync(0xffffffffu, j, k - 1);
        unsigned m = __ballot_sync(0xffffffffu, want && (n < k || better(cs, cj, ks, kj)));
        while (m) {
            int src = __ffs(m) - 1;
            m &= m - 1;
            float xs = __shfl_sync(0xffffffffu, cs, src);
            int xj = __shfl_sync(0xffffffffu, cj, src);
            if (n == k && !better(xs, xj, ks, kj)) continue;
            int pos = __popc(__ballot_sync(0xffffffffu, lane < n && better(s, j, xs, xj)));
            float us = __shfl_up_sync(0xffffffffu, s, 1);
            int uj = __shfl_up_sync(0xffffffffu, j, 1);
            if (lane > pos) {
                s = us;
                j = uj;
            } else if (lane == pos) {
                s = xs;
                j = xj;
            }
            n = n < k ? n + 1 : k;
            ks = __shfl_sync(0xffffffffu, s, k - 1);
            kj = __shfl_sync(0xffffffffu, j, k - 1);
        }
    }
};

// Concatenates per-part lists, highest part first, into out[0..k) with one
// warp: count_of(p) gives part p's list length, entry_of(p, i) its i-th
// entry.  Every lane loads one part's count and fills one output slot per
// group of 32 parts, so the merge costs a few memory round trips, not one per
// part.  All 32 lanes must call; returns the number written (<= k).
template <class CountF, class EntryF>
__device__ __forceinline__ int warp_merge_desc(int nparts, int k, CountF count_of, EntryF entry_of,
                                               int32_t *out) {
    const int lane = threadIdx.x & 31;
    int total = 0;
    for (int base = 0; base < nparts && total < k; base += 32) {
        const int part = nparts - 1 - (base + lane);
        const int n = base + lane < nparts ? count_of(part) : 0;
        int incl = n;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += u;
        }
        const int excl = incl - n;
        const int group = __shfl_sync(0xffffffffu, incl, 31);
        // output slot `lane` of this group comes from the last part whose
        // range starts at or before it
        int src = 0;
#pragma unroll
        for (int m = 0; m < 32; ++m) {
            const int e = __shfl_sync(0xffffffffu, excl, m);
            const int nn = __shfl_sync(0xffffffffu, n, m);
            if (nn > 0 && e <= lane) src = m;
        }
        const int e_src = __shfl_sync(0xffffffffu, excl, src);
        if (lane < group && total + lane < k)
            out[total + lane] = entry_of(nparts - 1 - (base + src), lane - e_src);
        total = min(k, total + group);
    }
    return total;
}

// Block-wide exclusive scan of one int64 per thread (blockDim.x <= 1024).
__device__ inline int64_t block_exclusive_scan(int64_t v, int64_t *total, int64_t *scratch) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int64_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int64_t u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += u;
    }
    if (lane == 31) scratch[warp] = incl;
    __syncthreads();
    int64_t before = 0, all = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
        if (w < warp) before += scratch[w];
        all += scratch[w];
    }
    __syncthreads();
    *total = all;
    return before + incl - v;
}

// One CTA builds the semantic plan plan[0..B]: prefix sums of the rows
// (len - 1) of the selected sequences with a valid length (selection:
// hit_kind != LEX when hit_kind is given, else active[b] != 0, NULL = all);
// with init_out, selected sequences get default outputs (no candidates).
// Lengths are read through L2 (they may come from the same kernel's CTAs).
__device__ inline void build_plan_cta(const int32_t *lengths, int64_t ld, int32_t B,
                                      const int32_t *hit_kind, const uint8_t *active,
                                      int64_t *plan, bool init_out, int32_t k, int32_t *cand,
                                      float *score, int32_t *n_cand) {
    __shared__ int64_t scratch[32];
    int64_t carry = 0;
    for (int base = 0; base < B; base += blockDim.x) {
        const int b = base + threadIdx.x;
        int64_t rows = 0;
        if (b < B) {
            const int len = __ldcg(lengths + b);
            const bool valid = len >= 1 && (int64_t)len <= ld;
            bool sel;
            if (hit_kind)
                sel = __ldcg(hit_kind + b) != ADAPLD_HIT_LEX;
            else
                sel = active ? active[b] != 0 : true;
            if (sel && valid) rows = len - 1;
            if (sel && init_out) {
                n_cand[b] = 0;
                for (int i = 0; i < k; ++i) {
                    cand[(int64_t)b * k + i] = -1;
                    score[(int64_t)b * k + i] = 0.f;
                }
            }
        }
        int64_t total;
        const int64_t ex = block_exclusive_scan(rows, &total, scratch);
        if (b < B) plan[b] = carry + ex;
        carry += total;
    }
    if (threadIdx.x == 0) plan[B] = carry;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ int warp_max_i(int v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

#endif  // __CUDACC__

// ---- host-side launchers (one per kernel) ---------------------------------------
// Counts a kernel launch that was enqueued (e == cudaSuccess) in the
// process-wide counter adapld_kernel_launches() reports; returns e.
cudaError_t counted(cudaError_t e);

// Launches `kern` as a programmatic dependent of the previous kernel in the
// stream (it must call pdl_wait_then_release before reading that kernel's
// outputs).
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t s, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return counted(cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...));
}

// Streaming multiprocessors of the current device (0 on error).
int device_sms();

struct LexLaunch {
    const int32_t *tokens;
    int64_t ld;
    const int32_t *lengths;
    int32_t B, n_max, k;
    int32_t *hit_kind, *match_n, *cand, *n_cand;
    float *score;            // optional: zeroed for every sequence
    int32_t *status;         // optional
    int32_t *stats;          // optional: zeroed
    // optional: words the kernel zeroes (the workspace counters of the later
    // kernels of a step, which then needs no memset); the lexical kernel
    // itself uses no counters
    int32_t *zero = nullptr;
    size_t zero_words = 0;
};
// Launched as a programmatic dependent of the previous kernel in the stream
// (it waits for it before touching memory).
cudaError_t launch_lexical(const LexLaunch &a, const Workspace &ws, cudaStream_t s);

// Semantic plan from the lexical outcomes, for batches too large for the
// semantic kernel to derive it (B >= kPlanInKernelB): one CTA, launched as a
// programmatic dependent of the lexical kernel.
cudaError_t launch_outcome_plan(const int32_t *lengths, int64_t ld, int32_t B,
                                const int32_t *hit_kind, const Workspace &ws, cudaStream_t s);

// Semantic work plan for the standalone semantic entry point (one CTA):
// ws.plan[b] = rows of earlier selected sequences (selection: active == NULL
// means all, else active[b] != 0; a sequence needs a valid length); selected
// sequences get default outputs (no candidates).
cudaError_t launch_plan(const int32_t *lengths, int64_t ld, int32_t B, const uint8_t *active,
                        int32_t k, int32_t *cand, float *score, int32_t *n_cand,
                        const Workspace &ws, cudaStream_t s);

struct SemLaunch {
    const uint16_t *reps;
    int64_t ld;
    int32_t d;
    const uint16_t *query;
    const int32_t *lengths;
    const uint8_t *active;   // standalone path (plan built by a separate kernel)
    int32_t B, k;
    float tau;
    int32_t *cand;
    float *score;
    int32_t *n_cand;
    int32_t *hit_kind;       // step path: set SEM / NONE at the final merge
    bool plan_ready;         // step path: the lexical kernel built the plan
    // token-embedding rows (Eq. 4 as printed): `reps` is then the embedding
    // table [vocab][d] and row j of sequence b is reps[tokens[b*ld + j]]
    const int32_t *tokens = nullptr;
    int32_t vocab = 0;
    // virtual sequences (successor backoff): sequence p scores the positions
    // of real sequence vseq_b[p] against reps[vseq_tok[p]] and writes row
    // vseq_out[p] of cand / score (row stride out_stride) and n_cand; their
    // count is *nvseq; plan, slots and counters come from the backoff part
    // of the workspace
    const int32_t *vseq_b = nullptr, *vseq_tok = nullptr, *vseq_out = nullptr;
    const int32_t *nvseq = nullptr;
    int32_t out_stride = 0;  // 0: k
    int32_t *status = nullptr;  // per real sequence ADAPLD_SEQ_* bits (nullable)
    // step path, B < kPlanInKernelB: the kernel derives the plan from
    // hit_kind and lengths (the lexical kernel wrote no plan)
    bool plan_from_outcome = false;
};
cudaError_t launch_semantic(const SemLaunch &a, const Workspace &ws, cudaStream_t s);

struct TreeLaunch {
    const int32_t *tokens;
    // (the token-embedding table, when given, is the last member)
    int64_t ld;
    const int32_t *lengths;
    const uint16_t *reps;
    int32_t d;
    const uint16_t *query;
    int32_t B;
    const int32_t *hit_kind;
    int32_t *cand;
    float *score;
    const int32_t *n_cand;
    const int32_t *next_topk;
    int32_t Kn;
    adapld_params p;
    adapld_tree_out out;
    int32_t *status;
    adapld_embeddings emb = {nullptr, 0, 0};  // token embeddings (two-representation mode)
    bool lists_ready = false;  // the distinct-token lists were built by this call already
};
cudaError_t launch_tree(const TreeLaunch &a, const Workspace &ws, cudaStream_t s);

// Distinct-token lists of the histories (two-representation mode; csrc/
// dedupe.cu).  For every selected sequence with a valid length:
// rep_tok[b][0..n) = the distinct tokens of positions [0, len-2] (ids outside
// [0, vocab) count as token 0, whose table row they read), ordered by their
// latest position; rep_tok[b][n] = the anchor token M[len-1] (as stored);
// rep_len[b] = n + 1, or 0 for an invalid length or an unselected sequence.
// Scoring rep rows r < n against a query scores every position of the token
// at once, and rank order r follows the latest position, so a top-k over the
// lists ranks tokens exactly as the per-position top-k would rank their
// latest occurrences.  Needs ws.htab zeroed beforehand.
struct DedupeLaunch {
    const int32_t *tokens;
    int64_t ld;
    const int32_t *lengths;
    int32_t B, vocab;
    const uint8_t *active;   // selection (NULL = every sequence)
    // when given, sequences with a lexical hit are left out (their lists are
    // needed only if lexical hits draft successors)
    const int32_t *skip_lex_of;
    int32_t *status;         // ADAPLD_SEQ_BAD_TOKEN bits (nullable)
    bool pdl;                // launched as a programmatic dependent of a kernel
    // semantic plan over the lists (built by the last sequence), selection as
    // in build_plan_cta
    bool build_plan;
    const int32_t *hit_kind;
    bool init_out;
    int32_t k;
    int32_t *cand;
    float *score;
    int32_t *n_cand;
    // also record each listed token's position (rep_pos) and insert the
    // tokens of the fallback sequences (hit_kind != LEX when hit_kind is
    // given, else every selected one) into the union hash
    bool union_insert = false;
};
cudaError_t launch_dedupe(const DedupeLaunch &a, const Workspace &ws, cudaStream_t s);

// Expansion of top-k lists over distinct tokens (rep indices, as written by
// the semantic kernel over the lists) into the top-k positions under (score
// desc, position desc): every position of a listed token has that token's
// score.  Virtual sequence p (real sequence vseq_b[p], output row
// vseq_out[p]; identity when NULL, count *nvseq when given) rewrites its row
// of cand / score / n_cand (row stride `stride`) in place.  Real sequences
// are expanded when hit_kind[b] == SEM (hit_kind given) or active[b] != 0.
struct ExpandLaunch {
    const int32_t *tokens;
    int64_t ld;
    const int32_t *lengths;
    int32_t vocab;
    int32_t P;               // virtual sequences the grid covers
    const int32_t *nvseq;    // device count (nullable: P)
    const int32_t *vseq_b, *vseq_out;
    int32_t *cand;
    float *score;
    int32_t *n_cand;
    int32_t stride, k;
    const int32_t *hit_kind;
    const uint8_t *active;
    int32_t *ticket;         // [P] slices done
};
cudaError_t launch_expand(const ExpandLaunch &a, const Workspace &ws, cudaStream_t s);

// The union pass of the two-representation fallback (csrc/union.cu), after
// the distinct-token lists were built with union_insert: every token of the
// union is read from the table once and scored against the queries (anchor
// embeddings) of every fallback sequence that holds it; then each sequence's
// top-k over its list.  Writes cand (list indices, for the expansion),
// score, n_cand and, with hit_kind, SEM / NONE for the fallback sequences
// (hit_kind != LEX; with active instead, the selected ones).
struct UnionLaunch {
    const uint16_t *table;   // [vocab][d] bf16
    int32_t vocab, d;
    int64_t ld;
    int32_t B;
    int32_t *hit_kind;       // step path (nullable)
    const uint8_t *active;   // standalone selection (NULL = every sequence)
    int32_t k;
    float tau;
    int32_t *cand;
    float *score;
    int32_t *n_cand;
    int32_t *status;         // ADAPLD_SEQ_BAD_TOKEN for an anchor outside the table
};
cudaError_t launch_union(const UnionLaunch &a, const Workspace &ws, cudaStream_t s);
// Whether the union pass serves a batch of this shape.
bool union_applies(int32_t B, int64_t ld, int32_t d, int32_t vocab);

struct VerifyLaunch {
    const uint16_t *logits;  // [B][N][V] bf16
    int32_t V;
    const int32_t *draft_tokens, *parents, *n_nodes;
    int32_t B, N;
    int32_t *n_accept, *new_tokens, *n_new;
    int32_t *tokens;         // append (nullable, with lengths)
    int64_t ld;
    int32_t *lengths;
    const uint16_t *node_reps;  // [B][N][d] (nullable)
    uint16_t *reps;
    int32_t d;
    uint16_t *query;
    int32_t *status;         // nullable
};
cudaError_t launch_verify(const VerifyLaunch &a, const Workspace &ws, cudaStream_t s);

}  // namespace adapld
