// Distinct-token lists for the token-embedding fallback (Eq. 4 as printed:
// cos(e_{M_j}, e_a)) and their expansion back to positions.
//
// Under Eq. 4 the score of position j depends only on the token M[j], so a
// history of len positions needs only as many table rows as it has distinct
// tokens (about a sixth to a quarter of the positions on Zipf-like text).
// Exactness is kept by ranking tokens by their latest position: the top-k
// positions under (score desc, position desc) all belong to tokens among the
// top-k of that token list, and expansion recovers their positions.
//
//  rep_insert_kernel  grid (C1 chunks of 4096 positions, B), 256 threads:
//      inserts (token, position) into the sequence's open-addressing hash
//      (key token + 1 in the high word, the latest position in the low word:
//      atomicCAS to claim a slot, atomicMax to keep the latest position);
//      lanes holding the same token in a warp insert once (__match_any_sync).
//  rep_count_kernel   same grid: marks the positions that are the latest
//      occurrence of their token (a bit each) and counts them per chunk; the
//      last chunk of a sequence turns the counts into offsets and writes
//      rep_len and the anchor; the last sequence builds the semantic plan
//      over the lists.
//  rep_scatter_kernel same grid: writes each chunk's marked positions'
//      tokens in position order at the chunk's offset.
//  The list kernels issue a thread's 16 token loads, then its 16 first hash
//  probes, before using any (the load factor keeps nearly every lookup at
//  its first slot), so a chunk costs a few memory round trips.
//  expand_kernel      grid (S4 slices of 8192 positions, P), 512 threads: per
//      listed token (a warp each) the k most recent positions in the slice;
//      the last slice merges per token, then over tokens by (score desc,
//      position desc) and rewrites the list as positions.
//
// Every probe loop is bounded by the table size (the load factor is at most
// 1/2, so it never comes close); running past it would raise
// ADAPLD_DEV_INTERNAL.
#include "common.cuh"

namespace adapld {

namespace {

struct DedupeArgs {
    DedupeLaunch p;
    Workspace ws;
};

struct ExpandArgs {
    ExpandLaunch p;
    Workspace ws;
};

__device__ __forceinline__ bool seq_selected(const DedupeLaunch &a, int b, int &len) {
    len = a.lengths[b];
    if (len < 1 || (int64_t)len > a.ld) return false;
    if (a.skip_lex_of && __ldcg(a.skip_lex_of + b) == ADAPLD_HIT_LEX) return false;
    return a.active ? a.active[b] != 0 : true;
}

// Whether sequence b's distinct tokens join the union pass (the fallback
// sequences: no lexical hit on the step path; the selected ones otherwise).
__device__ __forceinline__ bool joins_union(const DedupeLaunch &a, const Workspace &ws, int b) {
    if (!a.union_insert || !ws.uhash) return false;
    return a.hit_kind ? __ldcg(a.hit_kind + b) != ADAPLD_HIT_LEX : true;
}

// Latest position stored for token u (-1 if absent or past the probe bound).
__device__ __forceinline__ int hash_lookup(const unsigned long long *T, int64_t H, int u) {
    const unsigned long long key = (unsigned long long)(uint32_t)(u + 1);
    uint64_t h = hash32((uint32_t)u) & (uint64_t)(H - 1);
    for (int64_t probe = 0; probe < H; ++probe) {
        const unsigned long long cur = __ldcg(T + h);
        if (cur == 0ull) return -1;
        if ((cur >> 32) == key) return (int)(uint32_t)(cur & 0xffffffffull);
        h = (h + 1) & (uint64_t)(H - 1);
    }
    return -1;
}

constexpr int kPerThread = kChunk1 / kThreads1;  // positions per thread and chunk (16)
constexpr int kWordsPerChunk = kChunk1 / 32;        // latest-occurrence bit words (128)

// Inserts positions [j0, j1) of sequence b into its hash (all threads of the
// CTA).  A token id outside the table sets *s_bad.
__device__ void insert_chunk(const DedupeLaunch &a, const Workspace &ws, int b, int j0, int j1,
                             int *s_bad) {
    const int t = threadIdx.x, lane = t & 31;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    unsigned long long *T = ws.htab + (int64_t)b * ws.H;
    const uint64_t mask = (uint64_t)(ws.H - 1);
    bool bad = false, lost = false;
    // all token loads, then all first-probe loads, in flight together
    int u[kPerThread];
#pragma unroll
    for (int e = 0; e < kPerThread; ++e) {
        const int j = j0 + e * kThreads1 + t;
        const int raw = j < j1 ? M[j] : 0;
        u[e] = canon(raw, a.vocab);
        bad |= j < j1 && raw != u[e];
    }
    bool lead[kPerThread];
    unsigned long long seen[kPerThread];
#pragma unroll
    for (int e = 0; e < kPerThread; ++e) {
        const int j = j0 + e * kThreads1 + t;
        const unsigned act = __ballot_sync(0xffffffffu, j < j1);
        lead[e] = false;
        if (j < j1) {
            // lanes hold consecutive positions: the highest lane of a group
            // of equal tokens has the latest one and inserts for the group
            const unsigned same = __match_any_sync(act, u[e]);
            lead[e] = lane == 31 - __clz(same);
        }
        seen[e] = lead[e] ? __ldcg(T + (hash32((uint32_t)u[e]) & mask)) : 0ull;
    }
#pragma unroll
    for (int e = 0; e < kPerThread; ++e) {
        if (!lead[e]) continue;
        const int j = j0 + e * kThreads1 + t;
        const unsigned long long mine =
            ((unsigned long long)(uint32_t)(u[e] + 1) << 32) | (unsigned long long)(uint32_t)j;
        uint64_t h = hash32((uint32_t)u[e]) & mask;
        if ((seen[e] >> 32) == (mine >> 32)) {  // the token's slot: keep the latest position
            if ((uint32_t)seen[e] < (uint32_t)j) atomicMax(T + h, mine);
            continue;
        }
        int64_t probe = 0;
        for (; probe < ws.H; ++probe) {
            const unsigned long long old = atomicCAS(T + h, 0ull, mine);
            if (old == 0ull) break;
            if ((old >> 32) == (mine >> 32)) {
                if ((uint32_t)old < (uint32_t)j) atomicMax(T + h, mine);
                break;
            }
            h = (h + 1) & mask;
        }
        lost |= probe == ws.H;
    }
    if (bad) *s_bad = 1;
    if (lost) atomicOr(ws.dev_status, ADAPLD_DEV_INTERNAL);
}

// Marks the positions of [j0, j1) that are the latest occurrence of their
// token: bit lane of words[e * 8 + warp] for position j0 + e*256 + warp*32 +
// lane (every word of the chunk is written).  Returns this thread's count.
__device__ int mark_chunk(const DedupeLaunch &a, const Workspace &ws, int b, int j0, int j1,
                          uint32_t *words) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    const unsigned long long *T = ws.htab + (int64_t)b * ws.H;
    const uint64_t mask = (uint64_t)(ws.H - 1);
    int u[kPerThread];
#pragma unroll
    for (int e = 0; e < kPerThread; ++e) {
        const int j = j0 + e * kThreads1 + t;
        u[e] = j < j1 ? canon(M[j], a.vocab) : 0;
    }
    unsigned long long seen[kPerThread];
#pragma unroll
    for (int e = 0; e < kPerThread; ++e) {
        const int j = j0 + e * kThreads1 + t;
        seen[e] = j < j1 ? __ldcg(T + (hash32((uint32_t)u[e]) & mask)) : 0ull;
    }
    int mine = 0;
#pragma unroll
    for (int e = 0; e < kPerThread; ++e) {
        const int j = j0 + e * kThreads1 + t;
        bool latest = false;
        if (j < j1) {
            const unsigned long long key = (unsigned long long)(uint32_t)(u[e] + 1);
            const int pos = (seen[e] >> 32) == key ? (int)(uint32_t)seen[e]
                                                   : hash_lookup(T, ws.H, u[e]);
            latest = pos == j;
        }
        const unsigned word = __ballot_sync(0xffffffffu, latest);
        if (lane == 0) words[e * (kThreads1 / 32) + warp] = word;
        mine += latest;
    }
    return mine;
}

// Adds token u to the union: bit u of the union bitmap (a reduction, no
// reply awaited).
__device__ __forceinline__ void union_insert(uint32_t *U, int u) {
    atomicOr(U + (u >> 5), 1u << (u & 31));
}

// Writes the marked positions' tokens of the chunk starting at j0 in
// position order to out (s_word: the chunk's 128 words in shared memory),
// and with pos_out their positions, adding each token to the union bitmap
// when uh is given.  One scan over the word counts gives every offset.
__device__ void scatter_chunk(const DedupeLaunch &a, int b, int j0, const uint32_t *s_word,
                              int *s_off, int64_t *s_scan, int32_t *out, int64_t room,
                              int32_t *dst, int32_t *pos_out, uint32_t *uh) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t w = t < kWordsPerChunk ? s_word[t] : 0u;
    int64_t all;
    const int64_t ex = block_exclusive_scan(__popc(w), &all, s_scan);
    if (t < kWordsPerChunk) s_off[t] = (int)ex;
    __syncthreads();
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    // word i = e * 8 + warp holds positions j0 + e * 256 + warp * 32 + lane
#pragma unroll 4
    for (int e = 0; e < kPerThread; ++e) {
        const int i = e * (kThreads1 / 32) + warp;
        const uint32_t wi = s_word[i];
        const int o = s_off[i] + __popc(wi & ((1u << lane) - 1u));
        if (((wi >> lane) & 1u) && idx_ok(o, 0, room, dst)) {
            const int j = j0 + e * kThreads1 + t;
            const int u = canon(M[j], a.vocab);
            out[o] = u;
            if (pos_out) pos_out[o] = j;
            if (uh) union_insert(uh, u);
        }
    }
}

__global__ void __launch_bounds__(kThreads1) rep_insert_kernel(DedupeArgs args) {
    const DedupeLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ int s_bad;
    pdl_wait_then_release();
    const int t = threadIdx.x;
    const int b = blockIdx.y, c = blockIdx.x;
    int len;
    if (!seq_selected(a, b, len)) return;
    const int j0 = c * kChunk1, j1 = min(j0 + kChunk1, len - 1);  // positions <= len-2
    if (j0 >= j1) return;
    if (t == 0) s_bad = 0;
    __syncthreads();
    insert_chunk(a, ws, b, j0, j1, &s_bad);
    __syncthreads();
    if (t == 0 && s_bad && a.status) atomicOr(a.status + b, ADAPLD_SEQ_BAD_TOKEN);
}

// rep_count_kernel: marks the latest occurrences (ws.rep_bits) and counts
// them per chunk; the last chunk of a sequence turns the counts into
// offsets, writes rep_len and the anchor; the last sequence builds the plan.
// SINGLE (every history fits one chunk, C1 == 1): the kernel also inserts
// the chunk first and scatters it after, so the lists take one kernel.
template <bool SINGLE>
__global__ void __launch_bounds__(kThreads1) rep_count_kernel(DedupeArgs args) {
    const DedupeLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ int s_flag, s_bad;
    __shared__ int64_t s_scan[32];
    __shared__ uint32_t s_word[SINGLE ? kWordsPerChunk : 1];
    __shared__ int s_off[SINGLE ? kWordsPerChunk : 1];
    pdl_wait_then_release();
    const int t = threadIdx.x;
    const int b = blockIdx.y, c = blockIdx.x;
    int len;
    const bool sel = seq_selected(a, b, len);
    bool seq_done = false;  // this CTA finishes sequence b (then takes the global ticket)
    if (!sel) {
        if (c != 0) return;
        if (t == 0) ws.rep_len[b] = 0;
        seq_done = true;
    } else {
        const int j0 = c * kChunk1, j1 = min(j0 + kChunk1, len - 1);
        const int32_t *M = a.tokens + (int64_t)b * a.ld;
        if (SINGLE) {
            if (t == 0) s_bad = 0;
            __syncthreads();
            insert_chunk(a, ws, b, j0, j1, &s_bad);
            __syncthreads();  // this CTA's inserts are the whole sequence's
            if (t == 0 && s_bad && a.status) atomicOr(a.status + b, ADAPLD_SEQ_BAD_TOKEN);
        }
        uint32_t *words =
            SINGLE ? s_word : ws.rep_bits + ((int64_t)b * ws.C1 + c) * kWordsPerChunk;
        const int mine = mark_chunk(a, ws, b, j0, j1, words);
        int64_t total;  // the block's sum
        (void)block_exclusive_scan(mine, &total, s_scan);
        if (SINGLE) {  // one chunk: offset 0, no ticket
            const bool uni = joins_union(a, ws, b);
            scatter_chunk(a, b, j0, s_word, s_off, s_scan, ws.rep_tok + (int64_t)b * a.ld, a.ld,
                          ws.dev_status, uni ? ws.rep_pos + (int64_t)b * a.ld : nullptr,
                          uni ? ws.uhash : nullptr);
            if (t == 0) {
                ws.rep_len[b] = (int)total + 1;
                ws.rep_tok[(int64_t)b * a.ld + total] = M[len - 1];  // the anchor (as stored)
            }
        } else {
            if (t == 0) ws.rep_cnt[(int64_t)b * ws.C1 + c] = (int)total;
            __threadfence();
            __syncthreads();
            if (t == 0) s_flag = atomicAdd(ws.rticket + b, 1) == (int)gridDim.x - 1;
            __syncthreads();
            if (!s_flag) return;
            __threadfence();
            // last chunk of b: chunk counts -> offsets, n = distinct tokens
            int64_t carry = 0;
            for (int base = 0; base < (int)gridDim.x; base += kThreads1) {
                const int cc = base + t;
                const int64_t v =
                    cc < (int)gridDim.x ? __ldcg(ws.rep_cnt + (int64_t)b * ws.C1 + cc) : 0;
                int64_t all;
                const int64_t ex = block_exclusive_scan(v, &all, s_scan);
                if (cc < (int)gridDim.x) ws.rep_cnt[(int64_t)b * ws.C1 + cc] = (int)(carry + ex);
                carry += all;
            }
            if (t == 0) {
                ws.rep_len[b] = (int)carry + 1;
                ws.rep_tok[(int64_t)b * a.ld + carry] = M[len - 1];  // the anchor (as stored)
            }
        }
        seq_done = true;
    }
    if (!seq_done || !a.build_plan) return;
    // ---- the last sequence overall: the semantic plan over the lists
    __threadfence();
    __syncthreads();
    if (t == 0) s_flag = atomicAdd(ws.gticket_rep, 1) == a.B - 1;
    __syncthreads();
    if (!s_flag) return;
    __threadfence();
    build_plan_cta(ws.rep_len, a.ld, a.B, a.hit_kind, a.hit_kind ? nullptr : a.active, ws.plan,
                   a.init_out, a.k, a.cand, a.score, a.n_cand);
}

// rep_scatter_kernel: the chunk's latest occurrences, in position order, at
// the chunk's offset.
__global__ void __launch_bounds__(kThreads1) rep_scatter_kernel(DedupeArgs args) {
    const DedupeLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ int64_t s_scan[32];
    __shared__ int s_off[kWordsPerChunk];
    __shared__ uint32_t s_word[kWordsPerChunk];
    pdl_wait_then_release();
    const int t = threadIdx.x;
    const int b = blockIdx.y, c = blockIdx.x;
    int len;
    if (!seq_selected(a, b, len)) return;
    const int j0 = c * kChunk1, j1 = min(j0 + kChunk1, len - 1);
    if (j0 >= j1) return;
    const uint32_t *bits = ws.rep_bits + ((int64_t)b * ws.C1 + c) * kWordsPerChunk;
    if (t < kWordsPerChunk) s_word[t] = __ldcg(bits + t);
    __syncthreads();
    const int off = __ldcg(ws.rep_cnt + (int64_t)b * ws.C1 + c);
    if (!idx_ok(off, 0, a.ld, ws.dev_status)) return;
    const bool uni = joins_union(a, ws, b);
    scatter_chunk(a, b, j0, s_word, s_off, s_scan, ws.rep_tok + (int64_t)b * a.ld + off,
                  a.ld - off, ws.dev_status,
                  uni ? ws.rep_pos + (int64_t)b * a.ld + off : nullptr, uni ? ws.uhash : nullptr);
}

// ---------------------------------------------------------------- expansion
constexpr int kExpandThreads = kThreads4;  // 16 warps
constexpr int kExpandWarps = kExpandThreads / 32;

struct ExpandShared {
    int tok[kSlice4];         // canonical tokens of the slice
    int key[kMaxK];           // listed tokens
    float sc[kMaxK];          // their scores
    int lst[kMaxK][kMaxK];    // per token: the k most recent positions
    int cnt[kMaxK];
    int flag;
};

// Slice sl of virtual sequence p (the whole CTA; every branch is uniform).
__device__ void expand_one(const ExpandLaunch &a, const Workspace &ws, ExpandShared &sh, int p,
                           int sl) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int b = a.vseq_b ? a.vseq_b[p] : p;
    const int64_t row = a.vseq_out ? a.vseq_out[p] : p;
    const int k = a.k;
    int32_t *crow = a.cand + row * a.stride;
    float *srow = a.score + row * a.stride;
    const int32_t *M = a.tokens + (int64_t)b * a.ld;
    // every load that does not depend on another at once (one memory round
    // trip): this slice's tokens, positions [p0, p0 + kSlice4) clipped at ld,
    // copied to shared memory, and the sequence's outcome, length, list
    // length and candidates
    const int p0 = sl * kSlice4;
    const int nld = (int)min((int64_t)kSlice4, a.ld - p0);
    for (int i = t; i < nld; i += kExpandThreads) cp_async4(sh.tok + i, M + p0 + i);
    bool skip = false;
    if (!a.vseq_b) {
        if (a.hit_kind) skip = a.hit_kind[b] != ADAPLD_HIT_SEM;
        else if (a.active) skip = !a.active[b];
    }
    const int len = a.lengths[b];
    const int ncr = a.n_cand[row];
    const int rl = ws.rep_len[b];
    const int r = t < k ? crow[t] : -1;
    const float sct = t < k ? srow[t] : 0.f;
    cp_async_wait_all();  // (also before an exit: the copies target this CTA's memory)
    if (skip || len < 2 || (int64_t)len > a.ld) return;
    const int n = min(ncr, k);
    if (n <= 0) return;
    if (t < n) {
        sh.key[t] = r >= 0 && r < rl - 1 ? ws.rep_tok[(int64_t)b * a.ld + r] : -1;
        sh.sc[t] = sct;
    }
    const int p1 = min(p0 + kSlice4, len - 1);
    __syncthreads();  // the copies of every thread have landed
    for (int i = t; i < p1 - p0; i += kExpandThreads) sh.tok[i] = canon(sh.tok[i], a.vocab);
    __syncthreads();

    // the k most recent positions of each listed token in this slice
    const bool single = gridDim.x == 1;
    constexpr int U = 8;
    for (int i = warp; i < n; i += kExpandWarps) {
        const int key = sh.key[i];
        int32_t *part = single ? nullptr
                               : ws.xpart + (((int64_t)p * ws.S4 + sl) * kMaxK + i) * kPart4Ints;
        int cnt = 0;
        for (int top = p1 - 1; top >= p0 && cnt < k; top -= 32 * U) {
            unsigned m[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = top - 32 * u - lane;
                m[u] = __ballot_sync(0xffffffffu, q >= p0 && sh.tok[q - p0] == key);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = top - 32 * u - lane;
                const int rank = cnt + __popc(m[u] & ((1u << lane) - 1u));
                if (((m[u] >> lane) & 1u) && rank < k && idx_ok(q, p0, p1, ws.dev_status)) {
                    if (single)
                        sh.lst[i][rank] = q;
                    else
                        part[1 + rank] = q;
                }
                cnt += __popc(m[u]);
            }
        }
        if (lane == 0) {
            if (single)
                sh.cnt[i] = min(cnt, k);
            else
                part[0] = min(cnt, k);
        }
    }
    if (!single) {
        __threadfence();
        __syncthreads();
        if (t == 0) sh.flag = atomicAdd(a.ticket + p, 1) == (int)gridDim.x - 1;
        __syncthreads();
        if (!sh.flag) return;
        __threadfence();
        // per token: merge the slices, most recent first
        for (int i = warp; i < n; i += kExpandWarps) {
            const int32_t *pw = ws.xpart + ((int64_t)p * ws.S4 * kMaxK + i) * kPart4Ints;
            const int64_t stride = (int64_t)kMaxK * kPart4Ints;  // next slice, same token
            const int total = warp_merge_desc(
                (int)gridDim.x, k, [&](int s2) { return __ldcg(pw + s2 * stride); },
                [&](int s2, int e) { return __ldcg(pw + s2 * stride + 1 + e); }, sh.lst[i]);
            if (lane == 0) sh.cnt[i] = total;
        }
    }
    __syncthreads();
    // over tokens: (score desc, position desc), the first k
    if (warp == 0) {
        WarpTopK tk;
        tk.reset();
        for (int i = 0; i < n; ++i) {
            const int c = idx_ok(sh.cnt[i], 0, k + 1, ws.dev_status) ? sh.cnt[i] : 0;
            tk.insert(lane < c, sh.sc[i], lane < c ? sh.lst[i][lane] : -1, k);
        }
        if (lane < k) {
            crow[lane] = lane < tk.n ? tk.j : -1;
            srow[lane] = lane < tk.n ? tk.s : 0.f;
        }
        if (lane == 0) a.n_cand[row] = tk.n;
    }
}

__global__ void __launch_bounds__(kExpandThreads) expand_kernel(ExpandArgs args) {
    __shared__ ExpandShared sh;
    pdl_wait_then_release();
    const ExpandLaunch &a = args.p;
    const int P = a.nvseq ? min(*a.nvseq, a.P) : a.P;
    // virtual sequences blockIdx.y, + gridDim.y, ... (the y extent is capped)
    for (int p = blockIdx.y; p < P; p += gridDim.y) {
        expand_one(a, args.ws, sh, p, blockIdx.x);
        __syncthreads();  // before the next p reuses the shared state
    }
}

}  // namespace

cudaError_t launch_dedupe(const DedupeLaunch &a, const Workspace &ws, cudaStream_t s) {
    DedupeArgs args{a, ws};
    const dim3 grid(ws.C1, a.B);
    if (ws.C1 == 1)  // every history is one chunk: one kernel builds the lists
        return a.pdl ? launch_dependent(rep_count_kernel<true>, grid, dim3(kThreads1), 0, s, args)
                     : (rep_count_kernel<true><<<grid, kThreads1, 0, s>>>(args),
                        counted(cudaGetLastError()));
    cudaError_t e = a.pdl ? launch_dependent(rep_insert_kernel, grid, dim3(kThreads1), 0, s, args)
                          : (rep_insert_kernel<<<grid, kThreads1, 0, s>>>(args),
                             counted(cudaGetLastError()));
    if (e != cudaSuccess) return e;
    e = launch_dependent(rep_count_kernel<false>, grid, dim3(kThreads1), 0, s, args);
    if (e != cudaSuccess) return e;
    return launch_dependent(rep_scatter_kernel, grid, dim3(kThreads1), 0, s, args);
}

cudaError_t launch_expand(const ExpandLaunch &a, const Workspace &ws, cudaStream_t s) {
    ExpandArgs args{a, ws};
    const int gy = a.P < 65535 ? (a.P < 1 ? 1 : a.P) : 65535;
    return launch_dependent(expand_kernel, dim3(ws.S4, gy), dim3(kExpandThreads), 0, s, args);
}

}  // namespace adapld
