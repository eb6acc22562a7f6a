// Host-side argument checks shared by every entry point of the C ABI.  Each
// returns ADAPLD_OK or the ADAPLD_ERR_* code that include/adapld.h documents
// for the argument, and none touches the device.
#pragma once

#include <cmath>
#include <cstdint>

#include "common.cuh"

namespace adapld {

inline bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

inline int check_params(const adapld_params *p) {
    if (!p) return ADAPLD_ERR_NULL;
    if (p->n_max < 1 || p->n_max > 8) return ADAPLD_ERR_NMAX;
    if (p->k < 1 || p->k > kMaxK) return ADAPLD_ERR_K;
    if (p->branch_width < 0 || p->branch_width > kMaxW) return ADAPLD_ERR_WIDTH;
    if (p->draft_len < 1 || p->draft_len > 256) return ADAPLD_ERR_DRAFT_LEN;
    if (p->succ_len < 1 || p->succ_len > 16) return ADAPLD_ERR_SUCC_LEN;
    if (std::isnan(p->tau)) return ADAPLD_ERR_TAU;
    if (1 + p->draft_len + p->branch_width * (1 + p->succ_len) > kMaxNodes)
        return ADAPLD_ERR_TOO_LARGE;
    return ADAPLD_OK;
}

inline int check_shape(int32_t B, int64_t ld) {
    if (B < 1 || B > 65535) return ADAPLD_ERR_BATCH;
    if (ld < 1) return ADAPLD_ERR_LD;
    if ((int64_t)B * ld >= ((int64_t)1 << 31)) return ADAPLD_ERR_TOO_LARGE;
    return ADAPLD_OK;
}

inline int check_dim(int32_t d) {
    if (d < 8 || d > 16384 || (d % 8) != 0) return ADAPLD_ERR_DIM;
    return ADAPLD_OK;
}

inline int check_k(int32_t k) { return (k < 1 || k > kMaxK) ? ADAPLD_ERR_K : ADAPLD_OK; }

inline int check_tau(float tau) { return std::isnan(tau) ? ADAPLD_ERR_TAU : ADAPLD_OK; }

inline int check_ws(void *ws, size_t ws_bytes, int32_t B, int64_t ld, int32_t W) {
    if (!ws) return ADAPLD_ERR_WORKSPACE;
    if (!aligned16(ws)) return ADAPLD_ERR_ALIGN;
    if (ws_bytes < layout_workspace(nullptr, B, ld, W).total_bytes) return ADAPLD_ERR_WORKSPACE;
    return ADAPLD_OK;
}

inline int check_emb(const adapld_embeddings *e) {
    if (!e) return ADAPLD_OK;
    if (!e->table || !aligned16(e->table) || e->vocab < 1) return ADAPLD_ERR_EMBEDDINGS;
    if (check_dim(e->dim) != ADAPLD_OK) return ADAPLD_ERR_EMBEDDINGS;
    return ADAPLD_OK;
}

#define ADAPLD_TRY(x)                     \
    do {                                  \
        int rc_ = (x);                    \
        if (rc_ != ADAPLD_OK) return rc_; \
    } while (0)

}  // namespace adapld
