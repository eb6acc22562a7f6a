// C ABI of the library (include/adapld.h): argument validation, workspace
// layout and stream-ordered kernel launches.  No entry point allocates memory
// or synchronises the host (except adapld_read_device_status).
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>

#include "checks.h"

using namespace adapld;

namespace {

std::atomic<unsigned long long> g_launches{0};  // kernels enqueued by the library

int cuda_status(cudaError_t e) { return e == cudaSuccess ? ADAPLD_OK : ADAPLD_ERR_CUDA; }

// Bytes from ws.htab that a two-representation call clears before the list
// kernels: the per-sequence hashes and, with the union pass, the bitmap words
// that cover the vocabulary (not the whole bitmap area the workspace holds).
size_t union_clear_bytes(const Workspace &w, int32_t B, int32_t vocab, bool uni) {
    const size_t hashes = sizeof(unsigned long long) * (size_t)B * (size_t)w.H;
    return uni ? hashes + sizeof(uint32_t) * (size_t)(((int64_t)vocab + 31) / 32) : hashes;
}

int record(void *ev, cudaStream_t s) {
    if (!ev) return ADAPLD_OK;
    return cuda_status(cudaEventRecord((cudaEvent_t)ev, s));
}

// Every argument check of a step, on device pointers and sizes only: a step
// fails here, before anything is enqueued, or not at all on the host side.
int check_step_args(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                    const uint16_t *reps, int32_t d, const uint16_t *query,
                    const int32_t *next_topk, int32_t Kn, int32_t B, const adapld_params *p,
                    const adapld_step_out *out, void *ws, size_t ws_bytes,
                    const adapld_embeddings *emb) {
    if (!tokens || !lengths || !reps || !query || !out) return ADAPLD_ERR_NULL;
    if (!out->hit_kind || !out->match_n || !out->cand || !out->score || !out->n_cand)
        return ADAPLD_ERR_NULL;
    const adapld_tree_out &to = out->tree;
    if (!to.anchor || !to.draft_tokens || !to.parents || !to.positions || !to.mask || !to.n_nodes)
        return ADAPLD_ERR_NULL;
    ADAPLD_TRY(check_params(p));
    ADAPLD_TRY(check_shape(B, ld));
    ADAPLD_TRY(check_dim(d));
    if (!aligned16(reps) || !aligned16(query)) return ADAPLD_ERR_ALIGN;
    if (next_topk && (Kn < 1 || Kn > kMaxW)) return ADAPLD_ERR_TOPK_TABLE;
    ADAPLD_TRY(check_emb(emb));
    return check_ws(ws, ws_bytes, B, ld, p->branch_width);
}

}  // namespace

extern "C" {

int32_t adapld_tree_nodes(const adapld_params *p) {
    if (!p) return 0;
    return 1 + p->draft_len + p->branch_width * (1 + p->succ_len);
}

size_t adapld_workspace_bytes(int32_t B, int64_t ld, int32_t d, const adapld_params *p) {
    if (check_shape(B, ld) != ADAPLD_OK || check_dim(d) != ADAPLD_OK) return 0;
    const int32_t W = p ? p->branch_width : 1;
    return layout_workspace(nullptr, B, ld, W).total_bytes;
}

const char *adapld_status_string(int code) {
    switch (code) {
        case ADAPLD_OK: return "ok";
        case ADAPLD_ERR_NULL: return "a required pointer is NULL";
        case ADAPLD_ERR_BATCH: return "batch size B must be in [1, 65535]";
        case ADAPLD_ERR_NMAX: return "n_max must be in [1, 8]";
        case ADAPLD_ERR_K: return "k must be in [1, 32]";
        case ADAPLD_ERR_WIDTH: return "branch_width must be in [0, 64]";
        case ADAPLD_ERR_DRAFT_LEN: return "draft_len must be in [1, 256]";
        case ADAPLD_ERR_DIM: return "d must be a multiple of 8 in [8, 16384]";
        case ADAPLD_ERR_ALIGN: return "reps, query and workspace must be 16-byte aligned";
        case ADAPLD_ERR_WORKSPACE: return "workspace missing or smaller than adapld_workspace_bytes()";
        case ADAPLD_ERR_LD: return "ld must be >= 1";
        case ADAPLD_ERR_TOO_LARGE: return "B*ld must be < 2^31 and the tree at most 1024 nodes";
        case ADAPLD_ERR_SUCC_LEN: return "succ_len must be in [1, 16]";
        case ADAPLD_ERR_TOPK_TABLE: return "next_topk needs Kn in [1, 64]";
        case ADAPLD_ERR_TAU: return "tau must not be NaN";
        case ADAPLD_ERR_STATIC_LIMIT: return "B exceeds ADAPLD_STATIC_MAX_B (1024) for the workspace-free entry point";
        case ADAPLD_ERR_EMBEDDINGS: return "embedding table NULL or misaligned, vocab < 1, or dim not a multiple of 8 in [8, 16384]";
        case ADAPLD_ERR_VOCAB: return "V must be a positive multiple of 8 and logits 16-byte aligned";
        case ADAPLD_ERR_CUDA: return "a CUDA runtime call failed";
        default: return "unknown status";
    }
}

int adapld_lexical_match(const int32_t *tokens, int64_t ld, const int32_t *lengths, int32_t B,
                         int32_t n_max, int32_t k, int32_t *hit_kind, int32_t *match_n,
                         int32_t *cand, int32_t *n_cand, void *ws, size_t ws_bytes,
                         adapld_stream_t stream) {
    if (!tokens || !lengths || !hit_kind || !match_n || !cand || !n_cand) return ADAPLD_ERR_NULL;
    ADAPLD_TRY(check_shape(B, ld));
    if (n_max < 1 || n_max > 8) return ADAPLD_ERR_NMAX;
    ADAPLD_TRY(check_k(k));
    ADAPLD_TRY(check_ws(ws, ws_bytes, B, ld, 1));
    cudaStream_t s = (cudaStream_t)stream;
    Workspace w = layout_workspace(ws, B, ld, 1);
    ADAPLD_TRY(cuda_status(cudaMemsetAsync(w.dev_status, 0, w.counters_bytes, s)));
    LexLaunch a{tokens, ld, lengths, B, n_max, k, hit_kind, match_n, cand, n_cand,
                nullptr, nullptr, nullptr};
    return cuda_status(launch_lexical(a, w, s));
}

int adapld_semantic_topk(const uint16_t *reps, int64_t ld, int32_t d, const uint16_t *query,
                         const int32_t *lengths, const uint8_t *active, int32_t B, int32_t k,
                         float tau, int32_t *cand, float *score, int32_t *n_cand, void *ws,
                         size_t ws_bytes, adapld_stream_t stream) {
    if (!reps || !query || !lengths || !cand || !score || !n_cand) return ADAPLD_ERR_NULL;
    ADAPLD_TRY(check_shape(B, ld));
    ADAPLD_TRY(check_dim(d));
    if (!aligned16(reps) || !aligned16(query)) return ADAPLD_ERR_ALIGN;
    ADAPLD_TRY(check_k(k));
    ADAPLD_TRY(check_tau(tau));
    ADAPLD_TRY(check_ws(ws, ws_bytes, B, ld, 1));
    cudaStream_t s = (cudaStream_t)stream;
    Workspace w = layout_workspace(ws, B, ld, 1);
    ADAPLD_TRY(cuda_status(cudaMemsetAsync(w.dev_status, 0, w.counters_bytes, s)));
    SemLaunch a{reps, ld, d, query, lengths, active, B, k, tau, cand, score, n_cand,
                nullptr, false};
    return cuda_status(launch_semantic(a, w, s));
}

int adapld_embedding_topk(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                          const adapld_embeddings *emb, const uint8_t *active, int32_t B,
                          int32_t k, float tau, int32_t *cand, float *score, int32_t *n_cand,
                          int32_t *status, void *ws, size_t ws_bytes, adapld_stream_t stream) {
    if (!tokens || !lengths || !emb || !cand || !score || !n_cand) return ADAPLD_ERR_NULL;
    ADAPLD_TRY(check_shape(B, ld));
    ADAPLD_TRY(check_emb(emb));
    ADAPLD_TRY(check_k(k));
    ADAPLD_TRY(check_tau(tau));
    ADAPLD_TRY(check_ws(ws, ws_bytes, B, ld, 1));
    cudaStream_t s = (cudaStream_t)stream;
    Workspace w = layout_workspace(ws, B, ld, 1);
    const bool uni = union_applies(B, ld, emb->dim, emb->vocab);  // every table row read once
    ADAPLD_TRY(cuda_status(cudaMemsetAsync(w.dev_status, 0, w.counters_bytes, s)));
    ADAPLD_TRY(cuda_status(
        cudaMemsetAsync(w.htab, 0, union_clear_bytes(w, B, emb->vocab, uni), s)));
    // the distinct tokens of the selected histories and the plan over them,
    // the scores of the distinct tokens, then their positions
    DedupeLaunch da{tokens, ld,   lengths, B,       emb->vocab, active, nullptr, status,
                    false,  true, nullptr, true,    k,          cand,   score,   n_cand};
    da.union_insert = uni;
    ADAPLD_TRY(cuda_status(launch_dedupe(da, w, s)));
    if (uni) {
        UnionLaunch ua{emb->table, emb->vocab, emb->dim, ld,  B,     nullptr, active,
                       k,          tau,        cand,     score, n_cand, status};
        ADAPLD_TRY(cuda_status(launch_union(ua, w, s)));
    } else {
        SemLaunch a{emb->table, ld, emb->dim, nullptr, w.rep_len, active, B, k, tau, cand, score,
                    n_cand, nullptr, true};
        a.tokens = w.rep_tok;
        a.vocab = emb->vocab;
        a.status = status;
        ADAPLD_TRY(cuda_status(launch_semantic(a, w, s)));
    }
    ExpandLaunch ea{tokens, ld,     lengths, emb->vocab, B, nullptr, nullptr, nullptr, cand,
                    score,  n_cand, k,       k,          nullptr, active, w.xticket};
    return cuda_status(launch_expand(ea, w, s));
}

int adapld_build_draft_tree(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                            const uint16_t *reps, int32_t d, const uint16_t *query, int32_t B,
                            const int32_t *hit_kind, int32_t *cand, float *score,
                            const int32_t *n_cand, const int32_t *next_topk, int32_t Kn,
                            const adapld_embeddings *emb, const adapld_params *p,
                            const adapld_tree_out *out, int32_t *status, void *ws,
                            size_t ws_bytes, adapld_stream_t stream) {
    if (!tokens || !lengths || !reps || !query || !hit_kind || !cand || !score || !n_cand || !out)
        return ADAPLD_ERR_NULL;
    if (!out->anchor || !out->draft_tokens || !out->parents || !out->positions || !out->mask ||
        !out->n_nodes)
        return ADAPLD_ERR_NULL;
    ADAPLD_TRY(check_params(p));
    ADAPLD_TRY(check_shape(B, ld));
    ADAPLD_TRY(check_dim(d));
    if (!aligned16(reps) || !aligned16(query)) return ADAPLD_ERR_ALIGN;
    if (next_topk && (Kn < 1 || Kn > kMaxW)) return ADAPLD_ERR_TOPK_TABLE;
    ADAPLD_TRY(check_emb(emb));
    ADAPLD_TRY(check_ws(ws, ws_bytes, B, ld, p->branch_width));
    cudaStream_t s = (cudaStream_t)stream;
    Workspace w = layout_workspace(ws, B, ld, p->branch_width);
    ADAPLD_TRY(cuda_status(cudaMemsetAsync(w.dev_status, 0, w.counters_bytes, s)));
    if (emb)
        ADAPLD_TRY(cuda_status(
            cudaMemsetAsync(w.htab, 0, union_clear_bytes(w, B, emb->vocab, false), s)));
    TreeLaunch a{tokens, ld, lengths, reps, d, query, B, hit_kind, cand, score, n_cand,
                 next_topk, next_topk ? Kn : 0, *p, *out, status};
    if (emb) a.emb = *emb;
    return cuda_status(launch_tree(a, w, s));
}

int adapld_step_ex(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                   const uint16_t *reps, int32_t d, const uint16_t *query,
                   const int32_t *next_topk, int32_t Kn, int32_t B, const adapld_params *p,
                   const adapld_step_out *out, void *ws, size_t ws_bytes,
                   const adapld_embeddings *emb, const adapld_step_events *ev,
                   adapld_stream_t stream) {
    ADAPLD_TRY(check_step_args(tokens, ld, lengths, reps, d, query, next_topk, Kn, B, p, out, ws,
                               ws_bytes, emb));
    const adapld_tree_out &to = out->tree;
    cudaStream_t s = (cudaStream_t)stream;
    Workspace w = layout_workspace(ws, B, ld, p->branch_width);
    const bool semantic = !(p->flags & ADAPLD_NO_SEMANTIC);
    // small batches: the fallback reads each table row of the batch's union
    // once, scored against every fallback query by the tensor cores
    // (csrc/union.cu), instead of once per sequence
    const bool uni = emb && semantic && union_applies(B, ld, emb->dim, emb->vocab);
    // (the workspace counters are zeroed by the lexical kernel)
    if (emb)
        ADAPLD_TRY(cuda_status(
            cudaMemsetAsync(w.htab, 0, union_clear_bytes(w, B, emb->vocab, uni), s)));

    ADAPLD_TRY(record(ev ? ev->lexical_begin : nullptr, s));
    LexLaunch la{tokens, ld, lengths, B, p->n_max, p->k, out->hit_kind, out->match_n, out->cand,
                 out->n_cand, out->score, out->status, to.stats};
    la.zero = w.dev_status;
    la.zero_words = w.counters_bytes / sizeof(int32_t);
    ADAPLD_TRY(cuda_status(launch_lexical(la, w, s)));
    // the semantic plan: derived by the semantic kernel itself for small
    // batches, else by one CTA from the outcomes (with a token-embedding
    // table it is built over the distinct-token lists instead)
    const bool small_plan = B < kPlanInKernelB;
    if (semantic && !emb && !small_plan)
        ADAPLD_TRY(cuda_status(launch_outcome_plan(lengths, ld, B, out->hit_kind, w, s)));
    ADAPLD_TRY(record(ev ? ev->lexical_end : nullptr, s));

    if (semantic) {
        ADAPLD_TRY(record(ev ? ev->semantic_begin : nullptr, s));
        SemLaunch sa{reps, ld, d, query, lengths, nullptr, B, p->k, p->tau, out->cand, out->score,
                     out->n_cand, out->hit_kind, true};
        sa.plan_from_outcome = !emb && small_plan;
        if (emb) {  // Eq. 4 over token embeddings, scored once per distinct token
            // lists for the fallback sequences, and for lexical hits too when
            // those draft successors (their backoff needs them)
            const bool lex_lists = (p->flags & ADAPLD_SUCC_ON_STRICT) != 0;
            DedupeLaunch da{tokens, ld, lengths, B, emb->vocab, nullptr,
                            lex_lists ? nullptr : out->hit_kind, out->status, true, !uni,
                            out->hit_kind, false, p->k, nullptr, nullptr, nullptr};
            da.union_insert = uni;
            ADAPLD_TRY(cuda_status(launch_dedupe(da, w, s)));
            sa.reps = emb->table;
            sa.d = emb->dim;
            sa.query = nullptr;
            sa.lengths = w.rep_len;
            sa.tokens = w.rep_tok;
            sa.vocab = emb->vocab;
            sa.status = out->status;
        }
        if (uni) {
            UnionLaunch ua{emb->table, emb->vocab, emb->dim, ld,         B,
                           out->hit_kind, nullptr,  p->k,     p->tau, out->cand,
                           out->score,    out->n_cand, out->status};
            ADAPLD_TRY(cuda_status(launch_union(ua, w, s)));
        } else {
            ADAPLD_TRY(cuda_status(launch_semantic(sa, w, s)));
        }
        if (emb) {
            ExpandLaunch ea{tokens, ld, lengths, emb->vocab, B, nullptr, nullptr, nullptr,
                            out->cand, out->score, out->n_cand, p->k, p->k, out->hit_kind,
                            nullptr, w.xticket};
            ADAPLD_TRY(cuda_status(launch_expand(ea, w, s)));
        }
        ADAPLD_TRY(record(ev ? ev->semantic_end : nullptr, s));
    }

    ADAPLD_TRY(record(ev ? ev->tree_begin : nullptr, s));
    TreeLaunch ta{tokens, ld, lengths, reps, d, query, B, out->hit_kind, out->cand, out->score,
                  out->n_cand, next_topk, next_topk ? Kn : 0, *p, to, out->status};
    if (emb) ta.emb = *emb;
    ta.lists_ready = emb && semantic;  // the distinct-token lists exist for every sequence
    ADAPLD_TRY(cuda_status(launch_tree(ta, w, s)));
    return record(ev ? ev->tree_end : nullptr, s);
}

int adapld_step(const int32_t *tokens, int64_t ld, const int32_t *lengths, const uint16_t *reps,
                int32_t d, const uint16_t *query, const int32_t *next_topk, int32_t Kn, int32_t B,
                const adapld_params *p, const adapld_step_out *out, void *ws, size_t ws_bytes,
                adapld_stream_t stream) {
    return adapld_step_ex(tokens, ld, lengths, reps, d, query, next_topk, Kn, B, p, out, ws,
                          ws_bytes, nullptr, nullptr, stream);
}

int adapld_step_from_host(const int32_t *tokens_h, int64_t ld, const int32_t *lengths_h,
                          const uint16_t *reps_h, int32_t d, const uint16_t *query_h, int32_t B,
                          const adapld_params *p, int32_t *tokens_d, int32_t *lengths_d,
                          uint16_t *reps_d, uint16_t *query_d, const adapld_step_out *out_d,
                          const adapld_step_out *out_h, void *ws, size_t ws_bytes,
                          adapld_stream_t stream) {
    if (!tokens_h || !lengths_h || !reps_h || !query_h || !out_h) return ADAPLD_ERR_NULL;
    // the step's own checks on the device buffers, before the first copy is
    // enqueued
    ADAPLD_TRY(check_step_args(tokens_d, ld, lengths_d, reps_d, d, query_d, nullptr, 0, B, p,
                               out_d, ws, ws_bytes, nullptr));
    cudaStream_t s = (cudaStream_t)stream;
    auto h2d = [&](void *dst, const void *src, size_t bytes) {
        return cuda_status(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, s));
    };
    const size_t rows = (size_t)B * (size_t)ld;
    ADAPLD_TRY(h2d(tokens_d, tokens_h, sizeof(int32_t) * rows));
    ADAPLD_TRY(h2d(lengths_d, lengths_h, sizeof(int32_t) * (size_t)B));
    ADAPLD_TRY(h2d(reps_d, reps_h, sizeof(uint16_t) * rows * (size_t)d));
    ADAPLD_TRY(h2d(query_d, query_h, sizeof(uint16_t) * (size_t)B * (size_t)d));
    ADAPLD_TRY(adapld_step(tokens_d, ld, lengths_d, reps_d, d, query_d, nullptr, 0, B, p, out_d,
                           ws, ws_bytes, stream));
    // the outputs back, every array the caller asked for
    const size_t N = (size_t)adapld_tree_nodes(p), k = (size_t)p->k, b = (size_t)B;
    struct Copy {
        void *dst;
        const void *src;
        size_t bytes;
    };
    const adapld_tree_out &th = out_h->tree, &td = out_d->tree;
    const Copy copies[] = {
        {out_h->hit_kind, out_d->hit_kind, 4 * b},     {out_h->match_n, out_d->match_n, 4 * b},
        {out_h->cand, out_d->cand, 4 * b * k},         {out_h->score, out_d->score, 4 * b * k},
        {out_h->n_cand, out_d->n_cand, 4 * b},         {out_h->status, out_d->status, 4 * b},
        {th.anchor, td.anchor, 4 * b},                 {th.draft_tokens, td.draft_tokens, 4 * b * N},
        {th.parents, td.parents, 4 * b * N},           {th.positions, td.positions, 4 * b * N},
        {th.mask, td.mask, b * N * N},                 {th.n_nodes, td.n_nodes, 4 * b},
        {th.stats, td.stats, 4 * 4},
    };
    for (const Copy &c : copies) {
        if (!c.dst || !c.src) continue;
        ADAPLD_TRY(cuda_status(cudaMemcpyAsync(c.dst, c.src, c.bytes, cudaMemcpyDeviceToHost, s)));
    }
    return ADAPLD_OK;
}

int adapld_accept_greedy(const uint16_t *logits, int32_t V, const int32_t *draft_tokens,
                         const int32_t *parents, const int32_t *n_nodes, int32_t B, int32_t N,
                         int32_t *n_accept, int32_t *new_tokens, int32_t *n_new,
                         int32_t *tokens, int64_t ld, int32_t *lengths,
                         const uint16_t *node_reps, uint16_t *reps, int32_t d,
                         uint16_t *query, int32_t *status, void *ws, size_t ws_bytes,
                         adapld_stream_t stream) {
    if (!logits || !draft_tokens || !parents || !n_nodes || !n_accept || !new_tokens || !n_new)
        return ADAPLD_ERR_NULL;
    if (B < 1 || B > 65535) return ADAPLD_ERR_BATCH;
    if (N < 1 || N > kMaxNodes) return ADAPLD_ERR_TOO_LARGE;
    if (V < 8 || (V % 8) != 0 || !aligned16(logits)) return ADAPLD_ERR_VOCAB;
    if ((tokens == nullptr) != (lengths == nullptr)) return ADAPLD_ERR_NULL;
    if (tokens && ld < 1) return ADAPLD_ERR_LD;
    if (node_reps) {
        if (!tokens || !reps || !query) return ADAPLD_ERR_NULL;
        ADAPLD_TRY(check_dim(d));
        if (!aligned16(node_reps) || !aligned16(reps) || !aligned16(query)) return ADAPLD_ERR_ALIGN;
    }
    // the layout for ld = 1 and W = 1, which every workspace for this B covers
    ADAPLD_TRY(check_ws(ws, ws_bytes, B, 1, 1));
    const Workspace w = layout_workspace(ws, B, 1, 1);
    cudaStream_t s = (cudaStream_t)stream;
    VerifyLaunch a{logits, V, draft_tokens, parents, n_nodes, B, N, n_accept, new_tokens, n_new,
                   tokens, ld, lengths, node_reps, reps, d, query, status};
    return cuda_status(launch_verify(a, w, s));
}

unsigned long long adapld_kernel_launches(void) {
    return g_launches.load(std::memory_order_relaxed);
}

int adapld_read_device_status(const void *ws, int32_t *status, adapld_stream_t stream) {
    if (!ws || !status) return ADAPLD_ERR_NULL;
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaMemcpyAsync(status, ws, sizeof(int32_t), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return ADAPLD_ERR_CUDA;
    return cuda_status(cudaStreamSynchronize(s));
}

}  // extern "C"

cudaError_t adapld::counted(cudaError_t e) {
    if (e == cudaSuccess) g_launches.fetch_add(1, std::memory_order_relaxed);
    return e;
}
