/*
 * adapld.h - C ABI of the GB300 (sm_103a) AdaPLD draft-construction library.
 *
 * One call of adapld_step() performs, for B independent sequences, the
 * per-decoding-step draft construction of AdaPLD (arXiv 2606.05742):
 *
 *   1. lexical anchoring (Sec. 3.3, Eq. 3), generalised from the last token to
 *      the longest suffix n-gram of length <= n_max;
 *   2. semantic fallback retrieval for sequences without a lexical hit
 *      (Sec. 3.3, Eq. 4-5): cosine of the query against every cached
 *      per-position representation, threshold tau, top-k;
 *   3. hidden-state rerank (Sec. 3.4, Eq. 6-7) and branched reuse construction
 *      (Sec. 3.5, Eq. 8-15; Algorithm 1): main span copy, branch tokens,
 *      successor tokens, emitted as a flat draft tree for tree attention
 *      (Sec. 3.6).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - All array arguments are DEVICE pointers owned by the caller.  The library
 *    never allocates or frees memory and keeps no state between calls; all
 *    temporary storage is the caller's workspace (see
 *    adapld_workspace_bytes()).
 *  - Work is enqueued asynchronously on `stream`; outputs are valid once the
 *    stream has been synchronised.  No entry point synchronises the host
 *    except adapld_read_device_status().  Calls on different streams are
 *    independent provided they use different workspaces and outputs.
 *  - adapld_step(), adapld_step_ex() (without events) and
 *    adapld_accept_greedy() enqueue device work only: a decode loop may
 *    capture them into a CUDA graph once and replay it, since every size
 *    the kernels act on (lengths, tree sizes) is read on the device.
 *  - Sequence b (0 <= b < B) of the token history is tokens[b*ld .. b*ld+len_b)
 *    with len_b = lengths[b]; the query anchor is tokens[b*ld + len_b - 1].
 *  - Representations are bf16, passed as uint16_t bit patterns.  Row j of
 *    sequence b is reps[(b*ld + j)*d .. +d): the representation that belongs
 *    to candidate position j, i.e. the prefix state h_{j-1} of Eq. 6 in the
 *    paper's 1-indexed notation (or the token embedding of Eq. 4 if the
 *    caller stores those).  query[b*d .. +d) is the current state
 *    h_{|M|-1}.  Row j*+1 is the successor reference h_{j*} of Eq. 13.
 *  - Positions are 0-indexed; candidates are positions j in [0, len_b-2].
 *  - Rankings use one total order: higher cosine first, equal cosines broken
 *    towards the more recent (larger) position.
 *  - Return value: ADAPLD_OK (0) or a negative ADAPLD_ERR_* code.  Argument
 *    errors are detected on the host before anything is enqueued.  Problems
 *    that depend on device data (a length outside [1, ld]) are reported per
 *    sequence in the status output instead, never by a device trap.
 */
#ifndef ADAPLD_H
#define ADAPLD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t / CUstream; 0 is the legacy default stream. */
typedef struct CUstream_st *adapld_stream_t;

/* ---- status codes --------------------------------------------------------- */
#define ADAPLD_OK 0
#define ADAPLD_ERR_NULL (-1)          /* a required pointer is NULL            */
#define ADAPLD_ERR_BATCH (-2)         /* B outside [1, 65535]                  */
#define ADAPLD_ERR_NMAX (-3)          /* n_max outside [1, 8]                  */
#define ADAPLD_ERR_K (-4)             /* k outside [1, 32]                     */
#define ADAPLD_ERR_WIDTH (-5)         /* branch_width outside [0, 64]          */
#define ADAPLD_ERR_DRAFT_LEN (-6)     /* draft_len outside [1, 256]            */
#define ADAPLD_ERR_DIM (-7)           /* d outside [8, 16384] or d % 8 != 0    */
#define ADAPLD_ERR_ALIGN (-8)         /* reps or query not 16-byte aligned     */
#define ADAPLD_ERR_WORKSPACE (-9)     /* workspace NULL or too small           */
#define ADAPLD_ERR_LD (-10)           /* ld < 1                                */
#define ADAPLD_ERR_TOO_LARGE (-11)    /* B*ld >= 2^31 or tree > 1024 nodes     */
#define ADAPLD_ERR_SUCC_LEN (-12)     /* succ_len outside [1, 16]              */
#define ADAPLD_ERR_TOPK_TABLE (-13)   /* next_topk given with Kn < 1           */
#define ADAPLD_ERR_TAU (-14)          /* tau is NaN                            */
#define ADAPLD_ERR_STATIC_LIMIT (-15) /* B > ADAPLD_STATIC_MAX_B for the
                                         workspace-free entry point           */
#define ADAPLD_ERR_EMBEDDINGS (-16)   /* embedding table NULL or misaligned,
                                         vocab < 1, or dim not a multiple of 8
                                         in [8, 16384]                        */
#define ADAPLD_ERR_VOCAB (-17)        /* V < 8 or V % 8 != 0, or logits not
                                         16-byte aligned                      */
#define ADAPLD_ERR_CUDA (-20)         /* a CUDA runtime call failed            */

/* ---- retrieval outcome per sequence (Eq. 5, Algorithm 1) ------------------- */
#define ADAPLD_HIT_NONE 0 /* nothing retrieved: the caller takes an AR step   */
#define ADAPLD_HIT_LEX 1  /* lexical (strict) hit                             */
#define ADAPLD_HIT_SEM 2  /* semantic fallback hit                            */

/* ---- per-sequence status bits (adapld_step_out.status) --------------------- */
#define ADAPLD_SEQ_BAD_LENGTH 1 /* len_b outside [1, ld]: hit NONE, 0 nodes    */
#define ADAPLD_SEQ_BAD_CANDIDATE 2 /* adapld_build_draft_tree() was given a
                                      candidate outside [0, len_b-2]: the
                                      sequence is treated as retrieving nothing */
#define ADAPLD_SEQ_BAD_TOKEN 4 /* a token id outside [0, vocab) met the
                                  embedding table: row 0 was used instead */
#define ADAPLD_SEQ_FULL 8      /* adapld_accept_greedy(): the append would
                                  pass ld, nothing was appended          */

/* ---- device status bits (adapld_read_device_status) ------------------------ */
#define ADAPLD_DEV_TIMEOUT 1  /* a bounded wait in a kernel expired; that
                                 call's outputs are not valid                  */
#define ADAPLD_DEV_INTERNAL 2 /* an internal index check failed (a bug)       */

/* ---- flags (adapld_params.flags) ------------------------------------------ */
#define ADAPLD_NO_LEX_RERANK 1u  /* lexical anchor = most recent match; no
                                    Eq. 6 gathers; lexical scores are NaN    */
#define ADAPLD_SUCC_ON_STRICT 2u /* successor drafting on lexical hits too
                                    (the prose of Sec. 3.5; Algorithm 1 runs it
                                    on semantic hits only, the default)       */
#define ADAPLD_NO_SEMANTIC 4u    /* lexical-only retrieval (Table 4 ablation) */
#define ADAPLD_NO_BRANCH 8u      /* no branch or successor paths (Table 4)    */
#define ADAPLD_NO_SUCC 16u       /* no successor drafting (Table 4)           */

/*
 * Draft-construction hyper-parameters (Algorithm 1 inputs).
 *   n_max        longest suffix n-gram tried by lexical anchoring, [1, 8]
 *   k            candidates kept by retrieval (and successor candidates per
 *                branch), [1, 32]
 *   branch_width W: branch tokens before Eq. 11's removal, [0, 64]
 *                (the paper's K; 8 in its experiments)
 *   draft_len    D: maximum main-copy length l_m of Eq. 8, [1, 256]
 *   succ_len     tokens appended per branch by successor drafting, [1, 16]
 *                (the paper appends one, Eq. 15)
 *   tau          semantic threshold of Eq. 4 (0.1 in the paper); -INFINITY
 *                keeps every row (pure top-k)
 *   flags        ADAPLD_* switches above
 */
typedef struct adapld_params {
    int32_t n_max;
    int32_t k;
    int32_t branch_width;
    int32_t draft_len;
    int32_t succ_len;
    float tau;
    uint32_t flags;
} adapld_params;

/*
 * Draft-tree outputs (Sec. 3.6; the flat layout is this library's reading, the
 * paper prints none).  N = adapld_tree_nodes(params) slots per sequence:
 * node 0 is the anchor token (parent -1, position len-1), then the main chain
 * (lexical hits), then per branch its token (parent 0) followed by its
 * successor tokens, each the child of the previous.  Parents precede
 * children; position id = len-1+depth; mask[i][j] = 1 iff node j is node i
 * or one of its ancestors.  Unused slots hold token/parent/position -1 and
 * mask 0.  A NONE outcome yields the root alone (n_nodes 1); an invalid
 * length yields n_nodes 0.
 *   anchor       [B]        j* (Eq. 7), -1 when nothing was retrieved
 *   draft_tokens [B][N]     int32
 *   parents      [B][N]     int32
 *   positions    [B][N]     int32
 *   mask         [B][N][N]  uint8
 *   n_nodes      [B]        int32
 *   stats        [4] int32 or NULL: lexical hits, semantic hits, empty
 *                retrievals (Eq. 17-18 counts) and branches extended by a
 *                successor.  Overwritten by adapld_step(); accumulated (not
 *                cleared) by adapld_build_draft_tree().
 */
typedef struct adapld_tree_out {
    int32_t *anchor;
    int32_t *draft_tokens;
    int32_t *parents;
    int32_t *positions;
    uint8_t *mask;
    int32_t *n_nodes;
    int32_t *stats;
} adapld_tree_out;

/*
 * All outputs of adapld_step().  Every pointer except status and stats is
 * required.
 *   hit_kind [B]     ADAPLD_HIT_*
 *   match_n  [B]     length of the matched suffix n-gram (0 unless lexical)
 *   cand     [B][k]  ranked candidates: for a lexical hit reranked by Eq. 6
 *                    (recency order with ADAPLD_NO_LEX_RERANK), for a semantic
 *                    hit by Eq. 4; cand[b][0] = j*.  Padding -1.
 *   score    [B][k]  float cosines of cand (padding 0; NaN for lexical
 *                    candidates under ADAPLD_NO_LEX_RERANK)
 *   n_cand   [B]     number of valid entries in cand
 *   status   [B]     ADAPLD_SEQ_* bits, or NULL
 *   tree             draft-tree outputs (see adapld_tree_out)
 */
typedef struct adapld_step_out {
    int32_t *hit_kind;
    int32_t *match_n;
    int32_t *cand;
    float *score;
    int32_t *n_cand;
    int32_t *status;
    adapld_tree_out tree;
} adapld_step_out;

/*
 * Token-embedding table of the target model, for the two-representation mode
 * (Sec. 3.3, Eq. 4 as printed: the fallback compares token embeddings
 * e_{M_j} with e_a; the hidden-state cache then reranks the candidates,
 * Eq. 6).  table: [vocab][dim] bf16 bits, 16-byte aligned, dim a multiple of 8
 * in [8, 16384].  Token ids outside [0, vocab) read row 0 and raise
 * ADAPLD_SEQ_BAD_TOKEN for their sequence.
 */
typedef struct adapld_embeddings {
    const uint16_t *table;
    int32_t vocab;
    int32_t dim;
} adapld_embeddings;

/* Optional CUDA events recorded around each kernel of adapld_step_ex(), for
 * timing a single stage inside a step.  Any member may be NULL.  The events
 * are cudaEvent_t handles, passed as void*. */
typedef struct adapld_step_events {
    void *lexical_begin, *lexical_end;
    void *semantic_begin, *semantic_end;
    void *tree_begin, *tree_end;
} adapld_step_events;

/* Node slots of one draft tree: 1 + draft_len + branch_width*(1+succ_len). */
int32_t adapld_tree_nodes(const adapld_params *p);

/* Workspace bytes needed by any entry point for B sequences of capacity ld and
 * dimension d under parameters p (0 if the arguments are invalid).  The
 * workspace is device memory, 256-byte aligned, with no initialisation
 * required; one workspace may be reused by consecutive calls on one stream.
 * About 21 of the ~23 bytes per history position (B*ld) hold the distinct-token
 * lists of the token-embedding mode (a hash of 2*ld slots of 8 bytes, the
 * lists and a bit per position); the rest is a few KB per sequence. */
size_t adapld_workspace_bytes(int32_t B, int64_t ld, int32_t d, const adapld_params *p);

/* Human-readable text for a status code (static storage). */
const char *adapld_status_string(int code);

/*
 * Lexical anchoring (Sec. 3.3, Eq. 3; generalised to the longest suffix).
 * For each sequence: n* = the largest n <= min(n_max, len-1) such that the
 * last n tokens also occur ending at some j <= len-2; the k most recent such
 * j are written to cand[b][0..n_cand) in descending order, match_n[b] = n*,
 * hit_kind[b] = ADAPLD_HIT_LEX.  Without a match: match_n 0, n_cand 0,
 * hit_kind ADAPLD_HIT_NONE.  cand padding is -1.  A length outside [1, ld]
 * is treated as no match.
 *   tokens [B][ld] int32, lengths [B] int32; outputs as in adapld_step_out.
 */
int adapld_lexical_match(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                         int32_t B, int32_t n_max, int32_t k, int32_t *hit_kind,
                         int32_t *match_n, int32_t *cand, int32_t *n_cand, void *ws,
                         size_t ws_bytes, adapld_stream_t stream);

/*
 * Semantic fallback retrieval (Sec. 3.3, Eq. 4-5), capped at k.
 * For every selected sequence (active == NULL selects all; otherwise those
 * with active[b] != 0) with a valid length: score(j) = cos(R_b[j], q_b) for
 * every j in [0, len-2], computed from bf16 inputs with fp32 accumulation;
 * rows with score >= tau are kept and the best min(k, count) are written to
 * cand/score in ranking order, n_cand[b] = count.  Padding: cand -1, score 0.
 * Rows of unselected sequences are left untouched.  A selected sequence with
 * an invalid length gets n_cand 0.
 *   reps  [B][ld][d] bf16 bits, 16-byte aligned, d % 8 == 0
 *   query [B][d]     bf16 bits, 16-byte aligned
 *   active [B] uint8 or NULL
 */
int adapld_semantic_topk(const uint16_t *reps, int64_t ld, int32_t d, const uint16_t *query,
                         const int32_t *lengths, const uint8_t *active, int32_t B, int32_t k,
                         float tau, int32_t *cand, float *score, int32_t *n_cand, void *ws,
                         size_t ws_bytes, adapld_stream_t stream);

/*
 * Rerank and draft-tree construction (Sec. 3.4-3.6, Eq. 6-15, Algorithm 1)
 * from retrieval results already in hit_kind / cand / score / n_cand (as
 * written by the two retrieval entry points).  For a lexical hit the
 * candidates are reranked by Eq. 6 in place (cand and score are rewritten in
 * ranking order; score NaN under ADAPLD_NO_LEX_RERANK); for a semantic hit the
 * Eq. 4 order is kept.  j* = cand[b][0].
 * Branch tokens: if next_topk is non-NULL ([B][ld][Kn] int32, the caller's
 * cached top-Kn next-token ids of the target model at every position, Eq.
 * 10), the first W non-negative ids of row j*; otherwise the first W
 * distinct tokens following the ranked candidates, tokens[c+1] (a model-free
 * reading of the anchor-conditioned next-token distribution).  On a lexical
 * hit the main path's first token is then removed (Eq. 11).
 * Successor drafting (Eq. 13-15) runs for semantic hits (and for lexical
 * ones under ADAPLD_SUCC_ON_STRICT): for branch token b, among the k most
 * recent positions t <= len-2 holding b, pick the one maximising
 * cos(R[t], R[j*+1]) and append tokens[t+1 .. t+succ_len] (clipped at
 * len-1).
 * emb (nullable) selects the two-representation mode: semantic hits are
 * reranked by Eq. 6 as well, and a branch token that never occurs backs off
 * to the embedding fallback with the branch token as the anchor (Sec. 3.5).
 * status [B] may be NULL; its ADAPLD_SEQ_BAD_TOKEN bit is kept, the others
 * are overwritten.
 */
int adapld_build_draft_tree(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                            const uint16_t *reps, int32_t d, const uint16_t *query, int32_t B,
                            const int32_t *hit_kind, int32_t *cand, float *score,
                            const int32_t *n_cand, const int32_t *next_topk, int32_t Kn,
                            const adapld_embeddings *emb, const adapld_params *p,
                            const adapld_tree_out *out, int32_t *status, void *ws,
                            size_t ws_bytes, adapld_stream_t stream);

/*
 * Semantic fallback over token embeddings (Sec. 3.3, Eq. 4 as printed).
 * For every selected sequence (active == NULL selects all) with a valid
 * length: score(j) = cos(E[tokens[j]], E[tokens[len-1]]) for every j in
 * [0, len-2]; rows with score >= tau are kept and the best min(k, count) by
 * (score desc, j desc) are written to cand / score, n_cand[b] = count (the
 * hidden-state rerank of Eq. 6 is adapld_build_draft_tree's).  Unselected
 * rows are left untouched.  status [B] (nullable) receives
 * ADAPLD_SEQ_BAD_TOKEN for a token id outside the table.
 */
int adapld_embedding_topk(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                          const adapld_embeddings *emb, const uint8_t *active, int32_t B,
                          int32_t k, float tau, int32_t *cand, float *score, int32_t *n_cand,
                          int32_t *status, void *ws, size_t ws_bytes, adapld_stream_t stream);

/*
 * One full draft-construction step for B sequences: lexical anchoring, the
 * semantic fallback for the sequences without a lexical hit (unless
 * ADAPLD_NO_SEMANTIC), then rerank and draft-tree construction, enqueued as
 * a chain of kernels with no host synchronisation.  Arguments as above;
 * next_topk may be NULL (then Kn is ignored).
 */
int adapld_step(const int32_t *tokens, int64_t ld, const int32_t *lengths, const uint16_t *reps,
                int32_t d, const uint16_t *query, const int32_t *next_topk, int32_t Kn, int32_t B,
                const adapld_params *p, const adapld_step_out *out, void *ws, size_t ws_bytes,
                adapld_stream_t stream);

/*
 * adapld_step() from HOST inputs to HOST outputs, all on `stream`: copies
 * tokens_h, lengths_h, reps_h and query_h (host memory, page-locked for the
 * copies to be asynchronous) into the caller's device buffers tokens_d,
 * lengths_d, reps_d and query_d (same layouts), runs the step into out_d
 * (device), then copies every non-NULL array of out_h (host; the same
 * shapes as out_d) from out_d.  The host outputs are valid once the stream
 * has been synchronised.  Nothing is allocated; argument errors as for
 * adapld_step() (ADAPLD_ERR_NULL also for a missing host or device input).
 */
int adapld_step_from_host(const int32_t *tokens_h, int64_t ld, const int32_t *lengths_h,
                          const uint16_t *reps_h, int32_t d, const uint16_t *query_h, int32_t B,
                          const adapld_params *p, int32_t *tokens_d, int32_t *lengths_d,
                          uint16_t *reps_d, uint16_t *query_d, const adapld_step_out *out_d,
                          const adapld_step_out *out_h, void *ws, size_t ws_bytes,
                          adapld_stream_t stream);

/*
 * adapld_step() with two options.  emb (nullable) selects the
 * two-representation mode: the fallback scores token embeddings (Eq. 4 as
 * printed), semantic candidates are reranked by the hidden states (Eq. 6),
 * and successor drafting backs off to the embedding fallback for a branch
 * token that never occurs (Sec. 3.5); cand / score then hold the reranked
 * candidates and their Eq. 6 scores.  events (nullable) are CUDA events
 * recorded around the step's kernels.
 */
int adapld_step_ex(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                   const uint16_t *reps, int32_t d, const uint16_t *query,
                   const int32_t *next_topk, int32_t Kn, int32_t B, const adapld_params *p,
                   const adapld_step_out *out, void *ws, size_t ws_bytes,
                   const adapld_embeddings *emb, const adapld_step_events *events,
                   adapld_stream_t stream);

/*
 * adapld_semantic_topk_static(): adapld_semantic_topk() for callers that cannot
 * provide any device memory beyond their inputs and outputs.  The paper has no
 * counterpart; this exists for deployment.  Typical such callers are host
 * libraries embedded in a serving process whose GPU memory is wholly owned by
 * another allocator (a cudaMalloc there would escape that allocator's budget
 * and implicitly synchronise the device), or integrations whose calling
 * convention has no place for a workspace buffer.
 *
 * Arguments, results and errors are those of adapld_semantic_topk() without
 * ws / ws_bytes.  The entry point allocates nothing: its scratch is one
 * file-scope device array of ADAPLD_STATIC_SCRATCH_BYTES (1 MiB), which every
 * GPU that loads the library reserves until the process exits.
 *   - B may be at most ADAPLD_STATIC_MAX_B (1024); larger batches return
 *     ADAPLD_ERR_STATIC_LIMIT without enqueuing anything.
 *   - The first call on each device looks up the array's device address (with
 *     that device current) and caches it; make that first call before any
 *     stream capture.
 *   - All calls on a device share the one array and it keeps the previous
 *     call's contents (each call clears what must start at zero), so calls
 *     that overlap on the GPU -- on different streams, or from different host
 *     threads -- race and must not be issued.  Serialise them.
 *   - The array's device address is cached per device ordinal for the
 *     process.  A context other than the device's primary context, or a
 *     primary context re-created after cudaDeviceReset(), is not supported:
 *     the cached address would belong to the old context.
 *   - A bounded wait that expires inside the kernel sets ADAPLD_DEV_TIMEOUT in
 *     the array's status word and leaves that call's outputs invalid (they
 *     may look like "no candidates").  Read the word with
 *     adapld_semantic_topk_static_status(); adapld_read_device_status() does
 *     not apply to this variant.
 */
#define ADAPLD_STATIC_SCRATCH_BYTES (1u << 20)
#define ADAPLD_STATIC_MAX_B 1024
int adapld_semantic_topk_static(const uint16_t *reps, int64_t ld, int32_t d,
                                const uint16_t *query, const int32_t *lengths,
                                const uint8_t *active, int32_t B, int32_t k, float tau,
                                int32_t *cand, float *score, int32_t *n_cand,
                                adapld_stream_t stream);

/* Synchronises `stream` and returns in *status (host memory) the ADAPLD_DEV_*
 * bits raised by the most recent adapld_semantic_topk_static() call on the
 * current device (0 = none; each call clears the word when it starts).  Pass
 * the stream of that call.  Allocates nothing.  The paper has no counterpart.
 * Errors: ADAPLD_ERR_NULL, ADAPLD_ERR_CUDA. */
int adapld_semantic_topk_static_status(int32_t *status, adapld_stream_t stream);

/* The number of CUDA kernels the library has enqueued in this process since it
 * was loaded, over every entry point, stream and device (an atomic counter;
 * any host thread may read it).  The difference of two readings is the
 * number of kernels the calls between them launched -- a measurement aid
 * (e.g. to count the launches of a timed region).  Never fails.  The paper
 * has no counterpart. */
unsigned long long adapld_kernel_launches(void);

/*
 * Greedy verification of the draft trees and the append to the memory
 * (Sec. 3.6; Appendix C, Eq. 16: at temperature 0 a draft token is accepted
 * iff it equals the target model's greedy choice; Algorithm 1,
 * VerifyAndAccept and the append).  The target model itself is the caller's.
 *   logits [B][N][V] bf16: the target's next-token logits after each tree
 *            node (tree-attention forward); rows of nodes >= n_nodes[b] are
 *            not read.  V % 8 == 0, 16-byte aligned, no NaN.
 *   draft_tokens, parents [B][N], n_nodes [B]: the trees (adapld_tree_out);
 *            node 0 is the root; parents[0] is not read.
 *   The choice at a node is the first index of its maximum logit.  From the
 *   root, the child whose token equals the choice at the current node is
 *   accepted (the first such child in node order), until there is none.
 *   n_accept [B]       accepted draft tokens
 *   new_tokens [B][N]  accepted draft tokens, then the choice after the last
 *                      accepted node (the bonus token); padding -1
 *   n_new [B]          n_accept + 1 (0 for an empty tree)
 * Append (tokens == NULL skips it; tokens and lengths go together): the new
 * tokens go to tokens[b][len_b ..] and lengths[b] grows by n_new.  If
 * node_reps ([B][N][d] bf16: the hidden state after each tree node, from the
 * same forward) is given, reps rows len_b .. len_b+n_new-1 receive the states
 * of the root and of the accepted nodes (row j holds the state after token
 * j-1) and query[b] the state after the last accepted node; reps and query
 * are then required and d valid.  A sequence whose append would pass ld gets
 * ADAPLD_SEQ_FULL in status [B] (nullable) and no append; one with
 * lengths[b] outside [0, ld] gets ADAPLD_SEQ_BAD_LENGTH and no append (the
 * verification outputs are still written).  Uses the verification part of a
 * workspace from adapld_workspace_bytes() for the same B (any ld, d and
 * parameters); N <= 1024.  Calls sharing a workspace must not overlap.
 */
int adapld_accept_greedy(const uint16_t *logits, int32_t V, const int32_t *draft_tokens,
                         const int32_t *parents, const int32_t *n_nodes, int32_t B, int32_t N,
                         int32_t *n_accept, int32_t *new_tokens, int32_t *n_new,
                         int32_t *tokens, int64_t ld, int32_t *lengths,
                         const uint16_t *node_reps, uint16_t *reps, int32_t d,
                         uint16_t *query, int32_t *status, void *ws, size_t ws_bytes,
                         adapld_stream_t stream);

/* Synchronises `stream` and returns in *status the ADAPLD_DEV_* bits raised by
 * the most recent call that used workspace `ws` (0 = none). */
int adapld_read_device_status(const void *ws, int32_t *status, adapld_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* ADAPLD_H */
