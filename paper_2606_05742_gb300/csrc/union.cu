// Two-representation fallback over the union of the batch's distinct tokens
// (Sec. 3.3, Eq. 4 as printed: cos(e_{M_j}, e_a) over token embeddings).
//
// The per-sequence path (semantic_kernel over each fallback sequence's
// distinct-token list) reads a table row once per sequence that holds its
// token; frequent tokens occur in most histories, so a batch reads two to
// six times the rows its union needs.  Here each row of the union is read
// from HBM once per step, and its dot products with the queries of all the
// fallback sequences (the anchors' table rows) form one dense contraction,
// union rows x queries over d, which runs on the tensor cores:
//
//  union_compact_kernel  the union bitmap over the vocabulary (a bit per
//      token, set by the list scatter with one atomic OR) into a list of
//      tokens in a scrambled order (every score is computed the same way
//      wherever its row lands; a token-ordered list read slower).
//  union_mma_kernel<NT>  persistent, one CTA per SM: 2 producer warps and
//      8 MMA warps.  A tile is 16 union rows; its K dimension (d) streams
//      through a ring of stages of 2048-element slices (4 KB; 2 KB when more
//      than 8 queries leave room for one such stage only), each stage the
//      tile's row slices and the live queries' slices (8 per query tile
//      holding one), as many stages as fit 227 KB (2 or 3): the producers'
//      lanes issue one bulk copy (cp.async.bulk) per slice, completing on the
//      stage's mbarrier.  Long slices read fastest (a copy-only probe over
//      random table rows: 1 KB slices 2.0 TB/s, 2 KB 3.7, 4 KB 5.9-6.5,
//      whole 16 KB rows 6.7-6.9).  Each MMA warp takes a K group of an
//      eighth of the stage, in two halves: it loads a half's fragments by
//      ldmatrix (slices padded by 16 bytes, so the 8 rows of a fragment hit
//      different banks), multiplies the 16 rows by the queries (mma.sync
//      m16n8k16, bf16 in, fp32 accumulate; query tiles past the last query
//      skipped) and sums the squares of its A fragments on the CUDA cores for
//      |row|^2; the stage's slot is released once the second half's
//      fragments are in registers, before their arithmetic, so the ring
//      refills during it (release after all the arithmetic: 225 us at config
//      5; norms by two more MMAs of the fragment with itself, which made the
//      tensor pipe the pace: 245 us).  At the end of a tile every warp leaves
//      its K group's partial sums in shared memory and, after one barrier,
//      the thread of each of the tile's (row, query) pairs adds them in a
//      fixed order and takes the pair: the row token's latest position in the
//      query's sequence (the list kernels' hash; -1: the sequence does not
//      hold it; the first probes of a thread's pairs were loaded while the
//      tile streamed) and the cosine written to score_pos[b][latest
//      position].
//  seq_topk_kernel  a cluster of 8 CTAs per fallback sequence: over its list
//      (entry r: the token whose latest position is rep_pos[r]) the top-k by
//      (score desc, r desc) at or above tau, a slice of the list per CTA,
//      merged in CTA rank 0; r order is latest-position order, so this is the
//      ranking the expansion expects.
//
// Every mbarrier wait is bounded: on expiry the CTA raises ADAPLD_DEV_TIMEOUT,
// stops issuing copies, drains those in flight and finishes without scores.
#include <cstdlib>

#include "common.cuh"

namespace adapld {

namespace {

struct UnionArgs {
    UnionLaunch p;
    Workspace ws;
};

struct CompactArgs {
    Workspace ws;
    int64_t cap;      // ulist entries (B * ld)
    uint32_t nwords;  // bitmap words covering the vocabulary
    uint32_t nsteps;  // the power of two >= nwords the visiting order runs over
};

// Whether sequence b is scored by the union pass and listed (the same test
// in every kernel here): a fallback sequence with a list.
__device__ __forceinline__ bool union_seq(const UnionLaunch &a, const Workspace &ws, int b,
                                          int *rows) {
    const int rl = ws.rep_len[b];
    *rows = rl - 1;
    if (rl < 1) return false;
    if (a.hit_kind) return a.hit_kind[b] != ADAPLD_HIT_LEX;
    return a.active ? a.active[b] != 0 : true;
}

// The union bitmap's set bits into the union list.  Word w is visited at
// step i with w = i * 0x9E3779B1 mod 2^n (odd multiplier: a bijection of the
// 2^n >= nwords steps), so the list is in scrambled token order: tiles of
// consecutive entries, which the MMA kernel's CTAs take in turn, read rows
// from all over the table (a token-ordered list read slower).  Each CTA
// takes a range of steps and appends its tokens with one atomic add per
// 2048 steps.
__global__ void __launch_bounds__(256) union_compact_kernel(CompactArgs args) {
    const Workspace &ws = args.ws;
    __shared__ int64_t s_scan[32];
    __shared__ int s_base;
    pdl_wait_then_release();
    constexpr int kPer = 8;  // steps per thread and round
    const uint32_t nsteps = args.nsteps;  // a power of two >= nwords
    const uint32_t per_cta = (nsteps + gridDim.x - 1) / gridDim.x;
    const uint32_t lo = blockIdx.x * per_cta;
    const uint32_t hi = min(lo + per_cta, nsteps);
    for (uint32_t base = lo; base < hi; base += 256 * kPer) {
        uint32_t word[kPer], widx[kPer];
        int mine = 0;
#pragma unroll
        for (int e = 0; e < kPer; ++e) {
            const uint32_t i = base + (uint32_t)e * 256 + threadIdx.x;
            widx[e] = (i * 0x9E3779B1u) & (nsteps - 1u);
            word[e] = (i < hi && widx[e] < args.nwords) ? __ldcg(ws.uhash + widx[e]) : 0u;
            mine += __popc(word[e]);
        }
        int64_t total;
        const int64_t ex = block_exclusive_scan(mine, &total, s_scan);
        if (threadIdx.x == 0) s_base = total ? atomicAdd(ws.ucount, (int)total) : 0;
        __syncthreads();
        int o = s_base + (int)ex;
#pragma unroll
        for (int e = 0; e < kPer; ++e)
            for (uint32_t m = word[e]; m; m &= m - 1)
                if (idx_ok(o, 0, args.cap, ws.dev_status))
                    ws.ulist[o++] = (int)(widx[e] * 32u + (uint32_t)(__ffs(m) - 1));
        __syncthreads();  // before s_base is rewritten
    }
}

// Latest position of token u in a sequence's hash T (-1: absent), from the
// value v already loaded from its first slot h.
__device__ __forceinline__ int hash_latest(const unsigned long long *T, int64_t H, int u,
                                           uint64_t h, unsigned long long v) {
    const unsigned long long key = (unsigned long long)(uint32_t)(u + 1);
    for (int64_t probe = 0; probe < H; ++probe) {
        if (v == 0ull) return -1;
        if ((v >> 32) == key) return (int)(uint32_t)(v & 0xffffffffull);
        h = (h + 1) & (uint64_t)(H - 1);
        v = __ldcg(T + h);
    }
    return -1;
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

// d += a * b: one m16n8k16 tile, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                          uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Tile shape per query-tile count NT (NQ = 8 NT queries at most): TR union
// rows per tile, K chunks of KC elements per stage.  The 8 MMA warps split a
// stage into RG = TR / 16 row groups x KG = 8 / RG K groups.
template <int NT> struct UCfg;
template <> struct UCfg<2> { static constexpr int TR = 16, KC = 2048; };

constexpr int kUConsumers = 8;  // MMA warps
constexpr int kUProducers = 2;  // copy-issuing warps (a bulk copy costs its thread
                                // about 100 cycles to issue)
constexpr int kUThreads = (kUConsumers + kUProducers) * 32;

template <int NT>
struct UGeom {
    static constexpr int TR = UCfg<NT>::TR, KC = UCfg<NT>::KC, NSMAX = 6;
    static constexpr int NQ = NT * 8, RG = TR / 16, KG = kUConsumers / RG;
    static constexpr int REDW = NQ + 1;             // partial dots + |row|^2 per row
    static constexpr size_t RED = sizeof(float) * (size_t)2 * KG * TR * REDW;  // two tiles
    // the ring takes what the reduction buffer, the mbarriers and the shared
    // variables leave of 227 KB; its stage count follows the live queries
    static constexpr size_t RING = 227 * 1024 - RED - 2 * NSMAX * sizeof(uint64_t) - 2048;
    static constexpr size_t SMEM = RING + RED + 2 * NSMAX * sizeof(uint64_t);
    // with every query tile live, two stages of KC / 2-element slices fit
    static_assert(RING >= 2 * (size_t)(TR + NQ) * (KC + 16), "two stages at the most queries");
    static_assert((KC / 2 / KG) % 16 == 0 && TR <= 64, "whole k16 steps per warp; rows by two lanes");
};

__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t (&r)[2]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];"
                 : "=r"(r[0]), "=r"(r[1])
                 : "r"(addr));
}

// One stage of an MMA warp, in two halves of its ks <= KMAX k16 steps: the
// first half's fragments are loaded and multiplied, then the second half's
// are loaded, the stage's slot is released (`empty`) and they are multiplied
// -- the ring refills while the second half computes.  A fragments: 16 rows;
// B fragments: NTL live query tiles of 8 (an x2 load for one tile, an x4 for
// two).  The rows' squares go to ss0 (row g) and ss1 (row g + 8).
template <int KH, int NTL, int NT>
__device__ __forceinline__ void half_mma(uint32_t sb, uint32_t a_off, uint32_t b_off,
                                         uint32_t b_off_last, int k0, int ks,
                                         uint32_t (&af)[KH][4], uint32_t (&bf)[KH][2 * NTL]) {
#pragma unroll
    for (int i = 0; i < KH; ++i) {
        const int k16 = k0 + i;
        if (k16 < ks) {
            ldsm_x4(sb + a_off + k16 * 32, af[i]);
            if constexpr (NTL == 1) {
                uint32_t b2[2];
                ldsm_x2(sb + b_off_last + k16 * 32, b2);
                bf[i][0] = b2[0];
                bf[i][1] = b2[1];
            } else {
                uint32_t b4[4];
                ldsm_x4(sb + b_off + k16 * 32, b4);
#pragma unroll
                for (int e = 0; e < 4; ++e) bf[i][e] = b4[e];
            }
        }
    }
}

template <int KH, int NTL, int NT>
__device__ __forceinline__ void half_math(int k0, int ks, const uint32_t (&af)[KH][4],
                                          const uint32_t (&bf)[KH][2 * NTL],
                                          float (&acc)[NT][4], float &ss0, float &ss1) {
#pragma unroll
    for (int i = 0; i < KH; ++i) {
        if (k0 + i < ks) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float lo = bf16lo(af[i][e]), hi = bf16hi(af[i][e]);
                if (e & 1) {
                    ss1 = fmaf(lo, lo, ss1);
                    ss1 = fmaf(hi, hi, ss1);
                } else {
                    ss0 = fmaf(lo, lo, ss0);
                    ss0 = fmaf(hi, hi, ss0);
                }
            }
            mma_16816(acc[0], af[i], bf[i][0], bf[i][1]);
            if constexpr (NTL == 2) mma_16816(acc[1], af[i], bf[i][2], bf[i][3]);
        }
    }
}

template <int KMAX, int NTL, int NT>
__device__ __forceinline__ void stage_mma(uint32_t sb, uint32_t a_off, uint32_t b_off,
                                          uint32_t b_off_last, int ks, uint64_t *empty,
                                          int lane, float (&acc)[NT][4], float &ss0,
                                          float &ss1) {
    static_assert(NTL <= NT && NTL <= 2 && KMAX % 2 == 0, "one or two live query tiles");
    constexpr int KH = KMAX / 2;
    uint32_t af[KH][4];
    uint32_t bf[KH][2 * NTL];
    half_mma<KH, NTL, NT>(sb, a_off, b_off, b_off_last, 0, ks, af, bf);
    half_math<KH, NTL, NT>(0, ks, af, bf, acc, ss0, ss1);
    half_mma<KH, NTL, NT>(sb, a_off, b_off, b_off_last, KH, ks, af, bf);
    // (the warp's shared-memory reads are ordered before lane 0's arrive by
    // the warp barrier and the arrive's release semantics)
    __syncwarp();
    if (lane == 0) mbar_arrive(empty);
    half_math<KH, NTL, NT>(KH, ks, af, bf, acc, ss0, ss1);
}

struct UnionShared {
    int sel[kUnionMaxB];    // the fallback sequences
    int qtok[kUnionMaxB];   // their anchors' table rows
    float qss[kUnionMaxB];  // |query|^2
    int64_t scan[32];
    int nsel;
    int abort;
};

// NT: query tiles of 8 (the queries, rounded up, are NT * 8 <= 64).
template <int NT>
__global__ void __launch_bounds__(kUThreads, 1) union_mma_kernel(UnionArgs args) {
    using G = UGeom<NT>;
    const UnionLaunch &a = args.p;
    const Workspace &ws = args.ws;
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t *ring = smem;
    float *red = (float *)(smem + G::RING);  // [2][KG][TR][REDW]
    uint64_t *full = (uint64_t *)(smem + G::RING + G::RED);
    uint64_t *empty = full + G::NSMAX;
    UnionShared &sh = *(UnionShared *)(empty + G::NSMAX);

    pdl_wait_then_release();
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int d = a.d;
    // ---- the fallback sequences and their query rows (every CTA alike)
    {
        int rows = 0;
        const bool in = t < a.B && union_seq(a, ws, t, &rows) && rows > 0;
        int64_t total;
        const int64_t ex = block_exclusive_scan(in ? 1 : 0, &total, sh.scan);
        if (in) {
            const int raw = ws.rep_tok[(int64_t)t * a.ld + rows];  // the anchor, as stored
            const int row = canon(raw, a.vocab);
            if (row != raw && blockIdx.x == 0 && a.status)
                atomicOr(a.status + t, ADAPLD_SEQ_BAD_TOKEN);
            sh.sel[ex] = t;
            sh.qtok[ex] = row;
        }
        if (t == 0) {
            sh.nsel = (int)total;
            sh.abort = 0;
            for (int i = 0; i < G::NSMAX; ++i) {
                mbar_init(&full[i], kUProducers);
                mbar_init(&empty[i], kUConsumers);
            }
            fence_barrier_init();
        }
    }
    __syncthreads();
    const int nsel = sh.nsel;
    const int U = *ws.ucount;
    const int ntiles = (U + G::TR - 1) / G::TR;
    if (nsel == 0 || (int)blockIdx.x >= ntiles) return;
    // a stage: TR row slices and the live query tiles' slices, of KC
    // elements, or KC / 2 where KC would leave room for one stage only
    const int ntl = (nsel + 7) >> 3;
    const int KC = (size_t)2 * (G::TR + 8 * ntl) * (G::KC * 2 + 16) <= G::RING ? G::KC
                                                                              : G::KC / 2;
    const int PITCH = KC * 2 + 16;  // bytes per staged slice (padded)
    const int KW = KC / G::KG;      // K elements per MMA warp and stage
    const int nk = (d + KC - 1) / KC;  // K chunks per tile
    const int stage_bytes = (G::TR + 8 * ntl) * PITCH;
    const int NS = min(G::NSMAX, (int)(G::RING / stage_bytes));
    const int my_tiles = (ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
    const int total_it = my_tiles * nk;

    // ------------------------------------------------------------ producers
    // A stage's copies (its rows, then its queries) are numbered c = 0 ..
    // nrows + nsel - 1; producer warp pw issues c = pw + kUProducers (lane +
    // 32 h), each warp announcing its own bytes on the stage's mbarrier.
    if (warp >= kUConsumers) {
        const int pw = warp - kUConsumers;
        int it = 0;
        bool failed = false;
        for (int ti = 0; ti < my_tiles && !failed; ++ti) {
            const int tile = (int)blockIdx.x + ti * (int)gridDim.x;
            const int nrows = min(G::TR, U - tile * G::TR);
            const int ncopies = nrows + nsel;
            const int mine = ncopies > pw ? (ncopies - pw + kUProducers - 1) / kUProducers : 0;
            int tk[2];  // the table row of each of this lane's copies
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int c = pw + kUProducers * (lane + 32 * h);
                tk[h] = c < nrows ? ws.ulist[tile * G::TR + c] : (c < ncopies ? sh.qtok[c - nrows] : 0);
                // (checked build: a table row outside the table reads row 0)
                if (c < ncopies && !idx_ok(tk[h], 0, a.vocab, ws.dev_status)) tk[h] = 0;
            }
            for (int kc = 0; kc < nk; ++kc, ++it) {
                const int s = it % NS, r = it / NS;
                int ok = 1;
                if (lane == 0) {
                    if (r > 0 && !mbar_wait_bounded(&empty[s], (r - 1) & 1)) ok = 0;
                    if (*(volatile int *)&sh.abort) ok = 0;
                }
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) {
                    failed = true;
                    break;
                }
                const int k0 = kc * KC, kl = min(KC, d - k0);
                const uint32_t bytes = (uint32_t)kl * 2;
                uint8_t *st = ring + (size_t)s * stage_bytes;
                if (lane == 0) mbar_arrive_expect_tx(&full[s], bytes * (uint32_t)mine);
                __syncwarp();
                const uint64_t pol = l2_evict_normal_policy();
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int c = pw + kUProducers * (lane + 32 * h);
                    if (c < ncopies)
                        bulk_g2s(st + (size_t)(c < nrows ? c : G::TR + c - nrows) * PITCH,
                                 a.table + (int64_t)tk[h] * d + k0, bytes, &full[s], pol);
                }
            }
        }
        if (failed && lane == 0) {
            sh.abort = 1;
            atomicOr(ws.dev_status, ADAPLD_DEV_TIMEOUT);
            for (int i = max(0, it - NS); i < it; ++i)  // copies still in flight
                (void)mbar_wait_bounded(&full[i % NS], (uint32_t)(i / NS) & 1);
        }
        return;
    }

    // ------------------------------------------------------------ consumers
    for (int q = warp; q < nsel; q += kUConsumers) {  // |query|^2, a warp per query
        const uint16_t *qr = a.table + (int64_t)sh.qtok[q] * d;
        float part = 0.f;
        for (int ch = lane; ch < (d >> 3); ch += 32) {
            const uint4 w = ldg_nc_v4(qr + (size_t)ch * 8);
            const uint32_t w4[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                part = fmaf(bf16lo(w4[e]), bf16lo(w4[e]), part);
                part = fmaf(bf16hi(w4[e]), bf16hi(w4[e]), part);
            }
        }
        part = warp_sum(part);
        if (lane == 0) sh.qss[q] = part;
    }
    named_bar_sync(1, kUConsumers * 32);  // qss visible

    const int rg = warp % G::RG, kg = warp / G::RG;  // row group, K group
    const int g = lane >> 2, cq = (lane & 3) * 2;    // accumulator row / query of this lane
    // fragment addresses: A = rows 16 rg + lane % 16, k half lane / 16; B =
    // queries (lane % 8) + 8 (lane / 16), k half (lane / 8) % 2
    const uint32_t ring_s = smem_u32(ring);
    const uint32_t a_off = (uint32_t)((rg * 16 + (lane & 15)) * PITCH + (lane >> 4) * 16 +
                                      kg * KW * 2);
    const uint32_t b_off = (uint32_t)((G::TR + (lane & 7) + ((lane >> 4) << 3)) * PITCH +
                                      ((lane >> 3) & 1) * 16 + kg * KW * 2);
    // the last, odd query tile: lanes 16..31 repeat its rows (the stage has
    // no slices past the live tiles)
    const uint32_t b_off_last = (uint32_t)((G::TR + (lane & 7)) * PITCH +
                                           ((lane >> 3) & 1) * 16 + kg * KW * 2);
    float acc[NT][4];
    float ss0 = 0.f, ss1 = 0.f;  // |row g|^2, |row g + 8|^2: this lane's share of its K group
    // the tile's (row, query) pairs of this thread: pair pi = r * nsel + q
    // for pi = t + 256 m; the first kBatch have their row token (loaded at
    // the tile's first chunk) and first hash probe (at its second) in flight
    // while the tile streams, so the epilogue waits for no load of theirs
    constexpr int kPer = (G::TR * G::NQ + kUConsumers * 32 - 1) / (kUConsumers * 32);
    constexpr int kBatch = kPer < 8 ? kPer : 8;
    const int npairs = G::TR * nsel;
    int pu[kBatch];
    uint32_t ph[kBatch];
    unsigned long long pv[kBatch];
    bool aborted = false;
    for (int it = 0; it < total_it; ++it) {
        const int ti = it / nk, kc = it - ti * nk;
        const int s = it % NS;
        const int tile = (int)blockIdx.x + ti * (int)gridDim.x;
        if (kc == 0) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
#pragma unroll
                for (int j = 0; j < NT; ++j) acc[j][e] = 0.f;
                ss0 = ss1 = 0.f;
            }
#pragma unroll
            for (int m = 0; m < kBatch; ++m) {
                const int pi = t + m * kUConsumers * 32;
                const int row = tile * G::TR + pi / nsel;
                pu[m] = (pi < npairs && row < U) ? __ldcg(ws.ulist + row) : -1;
            }
        }
        if (kc == min(1, nk - 1)) {
#pragma unroll
            for (int m = 0; m < kBatch; ++m) {
                const int pi = t + m * kUConsumers * 32;
                const int q = pi - (pi / nsel) * nsel;
                ph[m] = pu[m] >= 0 ? (uint32_t)(hash32((uint32_t)pu[m]) & (uint64_t)(ws.H - 1)) : 0u;
                pv[m] = pu[m] >= 0 ? __ldcg(ws.htab + (int64_t)sh.sel[q] * ws.H + ph[m]) : 0ull;
            }
        }
        if (!aborted && *(volatile int *)&sh.abort) aborted = true;  // the producer gave up
        if (!aborted && !mbar_wait_bounded(&full[s], (uint32_t)(it / NS) & 1)) {
            aborted = true;
            if (lane == 0) {
                sh.abort = 1;
                atomicOr(ws.dev_status, ADAPLD_DEV_TIMEOUT);
            }
        }
        if (!aborted) {
            const int kl = min(KC, d - kc * KC);
            const int ks = max(0, min(KW, kl - kg * KW)) / 16;  // k16 steps of this warp
            const uint32_t sb = ring_s + (uint32_t)(s * stage_bytes);
            // the warp's fragments of the whole stage go to registers first,
            // so the slot is released before the arithmetic
            if (ntl == 1)
                stage_mma<16, 1>(sb, a_off, b_off, b_off_last, ks, &empty[s], lane, acc, ss0, ss1);
            else
                stage_mma<8, 2>(sb, a_off, b_off, b_off_last, ks, &empty[s], lane, acc, ss0, ss1);
        } else {
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
        }
        if (kc != nk - 1) continue;

        // ---- the tile's epilogue: the rows' |row|^2 over the quad of lanes
        // holding them
        float n0 = ss0, n1 = ss1;
        n0 += __shfl_xor_sync(0xffffffffu, n0, 1);
        n0 += __shfl_xor_sync(0xffffffffu, n0, 2);
        n1 += __shfl_xor_sync(0xffffffffu, n1, 1);
        n1 += __shfl_xor_sync(0xffffffffu, n1, 2);
        // every MMA warp leaves its K group's partial sums in red[ti % 2][kg]
        // (two buffers by tile parity: a warp that starts the next tile's
        // epilogue early never meets this tile's reads, which end before the
        // next barrier)
        const int r0 = rg * 16 + g;
        float *const rbuf = red + (size_t)(ti & 1) * G::KG * G::TR * G::REDW;
        {
            float *rp = rbuf + (size_t)kg * G::TR * G::REDW;
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                if (j >= ntl) break;
                rp[r0 * G::REDW + j * 8 + cq] = acc[j][0];
                rp[r0 * G::REDW + j * 8 + cq + 1] = acc[j][1];
                rp[(r0 + 8) * G::REDW + j * 8 + cq] = acc[j][2];
                rp[(r0 + 8) * G::REDW + j * 8 + cq + 1] = acc[j][3];
            }
            if ((lane & 3) == 0) {
                rp[r0 * G::REDW + G::NQ] = n0;
                rp[(r0 + 8) * G::REDW + G::NQ] = n1;
            }
        }
        named_bar_sync(1, kUConsumers * 32);
        // every (row, query) pair of the tile: the row token's latest
        // position in the query's sequence (-1: not held), then the cosine
        // at that position; all first probes of a thread in flight together
        if (!aborted) {
#pragma unroll 1
            for (int m0 = 0; m0 < kPer; m0 += kBatch) {
                int uu[kBatch];
                uint32_t hh[kBatch];
                unsigned long long vv[kBatch];
#pragma unroll
                for (int m = 0; m < kBatch; ++m) {
                    if (m0 == 0) {
                        uu[m] = pu[m];
                        hh[m] = ph[m];
                        vv[m] = pv[m];
                        continue;
                    }
                    const int pi = t + (m0 + m) * kUConsumers * 32;
                    const int r = pi / nsel, q = pi - r * nsel;
                    const int row = tile * G::TR + r;
                    uu[m] = (pi < npairs && row < U) ? __ldcg(ws.ulist + row) : -1;
                    hh[m] = uu[m] >= 0 ? (uint32_t)(hash32((uint32_t)uu[m]) & (uint64_t)(ws.H - 1))
                                       : 0u;
                    vv[m] = uu[m] >= 0 ? __ldcg(ws.htab + (int64_t)sh.sel[q] * ws.H + hh[m]) : 0ull;
                }
#pragma unroll
                for (int m = 0; m < kBatch; ++m) {
                    if (uu[m] < 0) continue;
                    const int pi = t + (m0 + m) * kUConsumers * 32;
                    const int r = pi / nsel, q = pi - r * nsel;
                    const int b = sh.sel[q];
                    const int pos =
                        hash_latest(ws.htab + (int64_t)b * ws.H, ws.H, uu[m], hh[m], vv[m]);
                    if (pos >= 0 && idx_ok(pos, 0, a.ld, ws.dev_status)) {
                        // the pair's dot and the row's |row|^2, K groups in order
                        float dot = 0.f, ss = 0.f;
#pragma unroll
                        for (int p = 0; p < G::KG; ++p) {
                            dot += rbuf[((size_t)p * G::TR + r) * G::REDW + q];
                            ss += rbuf[((size_t)p * G::TR + r) * G::REDW + G::NQ];
                        }
                        ws.score_pos[(int64_t)b * a.ld + pos] = cosine_from(dot, ss, sh.qss[q]);
                    }
                }
            }
        }
    }
}


// The per-sequence top k over the union scores: a cluster of kTopkSlices
// CTAs per fallback sequence, CTA x ranking slice x of the sequence's list
// (entry r: the token whose latest position is rep_pos[r]; 8 entries per
// lane in flight), by (score desc, r desc) at or above tau; r order is
// latest-position order, so this is the ranking the expansion expects.
// Each CTA pushes its best k into CTA rank 0's shared memory, which merges
// them after one cluster barrier.
constexpr int kTopkSlices = 8;

__global__ void __launch_bounds__(kThreads4) seq_topk_kernel(UnionArgs args) {
    const UnionLaunch &a = args.p;
    const Workspace &ws = args.ws;
    __shared__ float wl_s[kThreads4 / 32][32];
    __shared__ int wl_j[kThreads4 / 32][32];
    __shared__ int wl_n[kThreads4 / 32];
    __shared__ float m_s[kTopkSlices][32];  // rank 0: every slice's list
    __shared__ int m_j[kTopkSlices][32];
    __shared__ int m_n[kTopkSlices];
    pdl_wait_then_release();
    const int b = blockIdx.y, x = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5;
    int n = 0;
    if (!union_seq(a, ws, b, &n)) return;  // the whole cluster (b is its sequence)
    cluster_arrive_relaxed();  // every CTA has started before the pushes (waited below)
    const int k = a.k;
    const float tau = a.tau;
    const int32_t *pos = ws.rep_pos + (int64_t)b * a.ld;
    const float *sc = ws.score_pos + (int64_t)b * a.ld;
    const int per = (n + kTopkSlices - 1) / kTopkSlices;
    const int lo = x * per, hi = min(n, lo + per);
    WarpTopK tk;
    tk.reset();
    constexpr int U8 = 8;  // list entries per lane per step, loads in flight together
    for (int base = lo + warp * 32 * U8; base < hi; base += kThreads4 * U8) {
        int p[U8];
#pragma unroll
        for (int u = 0; u < U8; ++u) {
            const int r = base + u * 32 + lane;
            p[u] = r < hi ? pos[r] : -1;
        }
        float s[U8];
#pragma unroll
        for (int u = 0; u < U8; ++u)
            s[u] = (p[u] >= 0 && idx_ok(p[u], 0, a.ld, ws.dev_status)) ? sc[p[u]] : -INFINITY;
#pragma unroll
        for (int u = 0; u < U8; ++u) {
            const int r = base + u * 32 + lane;
            tk.insert(r < hi && s[u] >= tau, s[u], r, k);
        }
    }
    wl_s[warp][lane] = tk.s;
    wl_j[warp][lane] = tk.j;
    if (lane == 0) wl_n[warp] = tk.n;
    __syncthreads();
    cluster_wait();
    if (warp == 0) {
        WarpTopK f;
        f.reset();
        for (int w = 0; w < kThreads4 / 32; ++w)
            f.insert(lane < wl_n[w], wl_s[w][lane], wl_j[w][lane], k);
        st_cluster_f32(&m_s[x][lane], 0, f.s);
        st_cluster_i32(&m_j[x][lane], 0, f.j);
        if (lane == 0) st_cluster_i32(&m_n[x], 0, f.n);
    }
    cluster_sync_all();  // the slices' lists are in rank 0
    if (x != 0 || warp != 0) return;
    WarpTopK f;
    f.reset();
    for (int r = 0; r < kTopkSlices; ++r) f.insert(lane < m_n[r], m_s[r][lane], m_j[r][lane], k);
    if (lane < k) {
        a.cand[(int64_t)b * k + lane] = lane < f.n ? f.j : -1;
        a.score[(int64_t)b * k + lane] = lane < f.n ? f.s : 0.f;
    }
    if (lane == 0) {
        a.n_cand[b] = f.n;
        if (a.hit_kind) a.hit_kind[b] = f.n > 0 ? ADAPLD_HIT_SEM : ADAPLD_HIT_NONE;
    }
}

template <int NT>
cudaError_t launch_mma(const UnionArgs &args, int sms, cudaStream_t s) {
    auto kern = union_mma_kernel<NT>;
    const size_t smem = UGeom<NT>::SMEM + sizeof(UnionShared);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_dependent(kern, dim3(sms), dim3(kUThreads), smem, s, args);
}

}  // namespace

bool union_applies(int32_t B, int64_t ld, int32_t d, int32_t vocab) {
    if (const char *e = std::getenv("ADAPLD_EMB_UNION"))  // A/B switch for measurements
        if (e[0] == '0') return false;
    // the bitmap (the workspace's UH words) must cover the vocabulary
    return union_enabled(B, ld) && d % 16 == 0 &&
           ((int64_t)vocab + 31) / 32 <= hash_slots((int64_t)B * (ld - 1) + 1);
}

cudaError_t launch_union(const UnionLaunch &a, const Workspace &ws, cudaStream_t s) {
    const int sms = device_sms();
    if (sms <= 0) return cudaErrorInvalidDevice;
    const uint32_t nwords = (uint32_t)(((int64_t)a.vocab + 31) / 32);
    uint32_t nsteps = 1;
    while (nsteps < nwords) nsteps <<= 1;
    CompactArgs ca{ws, (int64_t)a.B * a.ld, nwords, nsteps};
    cudaError_t e = launch_dependent(union_compact_kernel, dim3(2 * sms), dim3(256), 0, s, ca);
    if (e != cudaSuccess) return e;
    UnionArgs ua{a, ws};
    static_assert(kUnionMaxB <= 16, "two query tiles of 8");
    e = launch_mma<2>(ua, sms, s);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kTopkSlices, a.B);
    cfg.blockDim = dim3(kThreads4);
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = kTopkSlices;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return counted(cudaLaunchKernelEx(&cfg, seq_topk_kernel, ua));
}

}  // namespace adapld
