/*
 * AdaPLD draft-construction oracle: a plain, slow, single-threaded CPU
 * restatement of one decoding step of the method, in fp64.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call this file:
 * only the tests, the smoke check and the benchmark's CPU-baseline leg load
 * it.  It shares no source, header or constant with the CUDA library; the two
 * agree only because both follow the paper.
 *
 * Every function follows a passage of the paper (arXiv 2606.05742, "AdaPLD:
 * Adaptive Retrieval and Reuse for Efficient Model-Free Speculative
 * Decoding"):
 *   - lexical anchoring ........ Sec. 3.3, Eq. 3 (generalised from the last
 *                                token to the longest matching suffix n-gram,
 *                                n <= n_max; n_max = 1 is exactly Eq. 3)
 *   - semantic fallback ........ Sec. 3.3, Eq. 4 and the backoff rule Eq. 5
 *   - hidden-state rerank ...... Sec. 3.4, Eq. 6-7
 *   - main span copy ........... Sec. 3.5, Eq. 8-9
 *   - branch tokens ............ Sec. 3.5, Eq. 10-12
 *   - successor drafting ....... Sec. 3.5, Eq. 13-15
 *   - strict vs semantic paths . Algorithm 1 (main copy only when the anchor
 *                                is lexical; successors only for a semantic
 *                                hit; an AR step when nothing is retrieved)
 *   - draft tree ............... Sec. 3.6 (tree attention; the flat layout is
 *                                this library's reading, the paper gives none)
 *
 * Conventions (0-indexed, per sequence): M = tokens[0..len-1]; the query
 * anchor is a = M[len-1].  Row j of the representation cache R belongs to
 * candidate position j (it holds the prefix state h_{j-1} of Eq. 6 in the
 * paper's 1-indexed notation), the query q holds h_{|M|-1}, and the successor
 * reference h_{j*} of Eq. 13 is row j*+1.  Representations are bf16 bit
 * patterns, widened exactly to double.
 *
 * Parity pins: every function here is checked by the CPU test-suite against
 * brute force, closed forms, library routines or the hand-built worked
 * example; the end-to-end acceptance behaviour (verification by the target
 * model) is out of scope and stays parity unpinned.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Retrieval outcome of Eq. 5 / Algorithm 1. */
#define OR_NONE 0
#define OR_LEX 1
#define OR_SEM 2

/* Ablation switches (Table 4 and the readings of the paper). */
#define OR_NO_LEX_RERANK 1u   /* anchor = most recent lexical match        */
#define OR_SUCC_ON_STRICT 2u  /* successors on lexical hits as well (text) */
#define OR_NO_SEMANTIC 4u     /* lexical-only retrieval                    */
#define OR_NO_BRANCH 8u       /* no branch (and hence no successor) paths  */
#define OR_NO_SUCC 16u        /* no successor drafting                     */

static double bf16_bits_to_double(uint16_t h)
{
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* cos(x, y) = <x, y> / (|x| |y|), with the convention cos = 0 when either
 * vector is zero.  Used by Eq. 4, Eq. 6 and Eq. 13. */
double oracle_cosine(const uint16_t *x, const uint16_t *y, int32_t d)
{
    double xy = 0.0, xx = 0.0, yy = 0.0;
    for (int32_t c = 0; c < d; ++c) {
        double a = bf16_bits_to_double(x[c]);
        double b = bf16_bits_to_double(y[c]);
        xy += a * b;
        xx += a * a;
        yy += b * b;
    }
    if (xx == 0.0 || yy == 0.0)
        return 0.0;
    return xy / (sqrt(xx) * sqrt(yy));
}

/* Total order used for every ranking: higher score first, and for equal
 * scores the more recent (larger) position first. */
typedef struct {
    double s;
    int32_t j;
} scored_pos;

static int better(double sa, int32_t ja, double sb, int32_t jb)
{
    return sa > sb || (sa == sb && ja > jb);
}

static int cmp_scored(const void *pa, const void *pb)
{
    const scored_pos *a = (const scored_pos *)pa;
    const scored_pos *b = (const scored_pos *)pb;
    if (better(a->s, a->j, b->s, b->j))
        return -1;
    if (better(b->s, b->j, a->s, a->j))
        return 1;
    return 0;
}

/*
 * Lexical anchoring (Sec. 3.3, Eq. 3), generalised to the longest suffix.
 * For n = min(n_max, len-1) down to 1, C_n = { j : n-1 <= j <= len-2,
 * M[j-n+1 .. j] = M[len-n .. len-1] }.  The first non-empty C_n gives
 * match_n = n and the k most recent members, in descending j.
 * Returns 1 on a hit, 0 otherwise.
 */
int oracle_lexical(const int32_t *M, int32_t len, int32_t n_max, int32_t k,
                   int32_t *match_n, int32_t *cand, int32_t *n_cand)
{
    *match_n = 0;
    *n_cand = 0;
    int32_t top = n_max < len - 1 ? n_max : len - 1;
    for (int32_t n = top; n >= 1; --n) {
        int32_t cnt = 0;
        for (int32_t j = len - 2; j >= n - 1; --j) {
            int same = 1;
            for (int32_t i = 0; i < n; ++i) {
                if (M[j - n + 1 + i] != M[len - n + i]) {
                    same = 0;
                    break;
                }
            }
            if (same) {
                if (cnt < k)
                    cand[cnt] = j;
                ++cnt;
            }
        }
        if (cnt > 0) {
            *match_n = n;
            *n_cand = cnt < k ? cnt : k;
            return 1;
        }
    }
    return 0;
}

/*
 * Semantic fallback (Sec. 3.3, Eq. 4), capped at k.  Every position
 * j in [0, len-2] is scored by cos(R[j], q); those with score >= tau are
 * kept and the best min(k, count) are returned in (score desc, j desc)
 * order.  R points at row 0 of this sequence, rows d elements apart.
 * Returns the number of candidates written.
 */
int32_t oracle_semantic(const uint16_t *R, int32_t d, const uint16_t *q,
                        int32_t len, int32_t k, double tau, int32_t *cand,
                        double *score)
{
    int32_t rows = len - 1;
    if (rows <= 0)
        return 0;
    scored_pos *all = (scored_pos *)malloc(sizeof(scored_pos) * (size_t)rows);
    int32_t cnt = 0;
    for (int32_t j = 0; j < rows; ++j) {
        double s = oracle_cosine(R + (int64_t)j * d, q, d);
        if (s >= tau) {
            all[cnt].s = s;
            all[cnt].j = j;
            ++cnt;
        }
    }
    qsort(all, (size_t)cnt, sizeof(scored_pos), cmp_scored);
    int32_t n = cnt < k ? cnt : k;
    for (int32_t i = 0; i < n; ++i) {
        cand[i] = all[i].j;
        score[i] = all[i].s;
    }
    free(all);
    return n;
}

/*
 * Semantic fallback over token embeddings (Sec. 3.3, Eq. 4 as printed): every
 * position j in [0, len-2] is scored by cos(E[M[j]], E[a]) with a = M[len-1]
 * and E the caller's token-embedding table (rows de elements apart); rows
 * with score >= tau are kept and the best min(k, count) are returned in
 * (score desc, j desc) order.  Returns the number written.
 */
int32_t oracle_semantic_emb(const int32_t *M, int32_t len, const uint16_t *E, int32_t de,
                            int32_t k, double tau, int32_t *cand, double *score)
{
    int32_t rows = len - 1;
    if (rows <= 0)
        return 0;
    const uint16_t *ea = E + (int64_t)M[len - 1] * de;
    scored_pos *all = (scored_pos *)malloc(sizeof(scored_pos) * (size_t)rows);
    int32_t cnt = 0;
    for (int32_t j = 0; j < rows; ++j) {
        double s = oracle_cosine(E + (int64_t)M[j] * de, ea, de);
        if (s >= tau) {
            all[cnt].s = s;
            all[cnt].j = j;
            ++cnt;
        }
    }
    qsort(all, (size_t)cnt, sizeof(scored_pos), cmp_scored);
    int32_t n = cnt < k ? cnt : k;
    for (int32_t i = 0; i < n; ++i) {
        cand[i] = all[i].j;
        score[i] = all[i].s;
    }
    free(all);
    return n;
}

/* All Eq. 4 scores of one sequence, for the tests' tolerance checks. */
void oracle_scores_all(const uint16_t *R, int32_t d, const uint16_t *q,
                       int32_t len, double *out)
{
    for (int32_t j = 0; j + 1 < len; ++j)
        out[j] = oracle_cosine(R + (int64_t)j * d, q, d);
}

/*
 * Hidden-state rerank (Sec. 3.4, Eq. 6-7) of lexical candidates:
 * s(j) = cos(R[j], q), candidates re-sorted by (s desc, j desc); the first
 * is j*.  Sorts cand[] in place and fills score[].
 */
void oracle_rerank(const uint16_t *R, int32_t d, const uint16_t *q,
                   int32_t *cand, double *score, int32_t n)
{
    scored_pos *tmp = (scored_pos *)malloc(sizeof(scored_pos) * (size_t)(n > 0 ? n : 1));
    for (int32_t i = 0; i < n; ++i) {
        tmp[i].j = cand[i];
        tmp[i].s = oracle_cosine(R + (int64_t)cand[i] * d, q, d);
    }
    qsort(tmp, (size_t)n, sizeof(scored_pos), cmp_scored);
    for (int32_t i = 0; i < n; ++i) {
        cand[i] = tmp[i].j;
        score[i] = tmp[i].s;
    }
    free(tmp);
}

/*
 * Successor candidates (Sec. 3.5, Eq. 13-14) for one branch token b: the k
 * most recent positions t in [0, len-2] with M[t] = b (positions that have
 * an observed following token), each scored by cos(R[t], R[j*+1]).
 * Written in descending t.  Returns the count.
 */
int32_t oracle_successor_candidates(const int32_t *M, int32_t len,
                                    const uint16_t *R, int32_t d,
                                    int32_t j_star, int32_t b, int32_t k,
                                    int32_t *t_out, double *s_out)
{
    int32_t cnt = 0;
    const uint16_t *ref = R + (int64_t)(j_star + 1) * d;
    for (int32_t t = len - 2; t >= 0 && cnt < k; --t) {
        if (M[t] == b) {
            t_out[cnt] = t;
            s_out[cnt] = oracle_cosine(R + (int64_t)t * d, ref, d);
            ++cnt;
        }
    }
    return cnt;
}

/*
 * Successor candidates with the lexical-first backoff of Sec. 3.5 applied to
 * the branch token b: the k most recent lexical occurrences of b; if there
 * are none and an embedding table E is given, the semantic fallback of
 * Eq. 4 with b as the query anchor (positions t in [0, len-2] with
 * cos(E[M[t]], E[b]) >= tau, best k by (score desc, t desc)).  Each is then
 * scored by Eq. 13 against R[j*+1].  Returns the count.
 */
int32_t oracle_successor_candidates_emb(const int32_t *M, int32_t len, const uint16_t *R,
                                        int32_t d, const uint16_t *E, int32_t de,
                                        double tau, int32_t j_star, int32_t b, int32_t k,
                                        int32_t *t_out, double *s_out)
{
    int32_t cnt = oracle_successor_candidates(M, len, R, d, j_star, b, k, t_out, s_out);
    if (cnt > 0 || E == NULL || len < 2)
        return cnt;
    const uint16_t *eb = E + (int64_t)b * de;
    scored_pos *all = (scored_pos *)malloc(sizeof(scored_pos) * (size_t)(len - 1));
    int32_t m = 0;
    for (int32_t t = 0; t + 1 < len; ++t) {
        double s = oracle_cosine(E + (int64_t)M[t] * de, eb, de);
        if (s >= tau) {
            all[m].s = s;
            all[m].j = t;
            ++m;
        }
    }
    qsort(all, (size_t)m, sizeof(scored_pos), cmp_scored);
    const uint16_t *ref = R + (int64_t)(j_star + 1) * d;
    for (int32_t i = 0; i < m && i < k; ++i) {
        t_out[cnt] = all[i].j;
        s_out[cnt] = oracle_cosine(R + (int64_t)all[i].j * d, ref, d);
        ++cnt;
    }
    free(all);
    return cnt;
}

/*
 * Draft-tree construction (Sec. 3.5 and Algorithm 1) from a retrieval
 * outcome and its ranked candidate list (cand[0] is j*).
 *
 *   node 0            : the anchor a = M[len-1], parent -1, depth 0
 *   main chain (LEX)  : M[j*+1 .. j*+l], l = min(D, len-1-j*)      Eq. 8-9
 *   branches          : B~ = first W distinct M[c+1] over the ranked
 *                       candidates (or the first W ids of the caller's
 *                       next-token table row at j*, when given); on a
 *                       lexical hit main[0] is removed          Eq. 10-11
 *   successors        : for SEM (or any hit with SUCC_ON_STRICT), per
 *                       branch b: j_b* = argmax over the k most recent
 *                       occurrences of b of cos(R[t], R[j*+1]); append
 *                       M[j_b*+1 .. j_b*+succ_len], clipped at len-1
 *                                                                Eq. 13-15
 * position id = len-1+depth; mask[i][j] = 1 iff j is i or an ancestor of i.
 * Unused slots: token/parent/position -1, mask 0.
 *
 * Returns the number of branches that received at least one successor.
 */
int32_t oracle_tree_from_emb(const int32_t *M, int32_t len, const uint16_t *R,
                             int32_t d, const uint16_t *E, int32_t de, double tau,
                             int32_t hit, const int32_t *cand,
                             int32_t n_cand, const int32_t *topk_row, int32_t Kn,
                             int32_t k, int32_t W, int32_t D, int32_t succ_len,
                             uint32_t flags, int32_t nmax, int32_t *anchor,
                             int32_t *tok, int32_t *par, int32_t *pos,
                             uint8_t *mask, int32_t *n_nodes)
{
    int32_t *depth = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nmax > 0 ? nmax : 1));
    int32_t n = 0;
    int32_t succ_ext = 0;
    for (int32_t i = 0; i < nmax; ++i) {
        tok[i] = -1;
        par[i] = -1;
        pos[i] = -1;
    }
    memset(mask, 0, (size_t)nmax * (size_t)nmax);
    *anchor = -1;

    /* the root: the last observed token */
    tok[0] = M[len - 1];
    par[0] = -1;
    depth[0] = 0;
    n = 1;

    if ((hit == OR_LEX || hit == OR_SEM) && n_cand > 0) {
        int32_t js = cand[0];
        *anchor = js;
        int32_t main0 = -1;
        if (hit == OR_LEX) {
            int32_t l = len - 1 - js;
            if (l > D)
                l = D;
            for (int32_t i = 0; i < l; ++i) {
                tok[n] = M[js + 1 + i];
                par[n] = (i == 0) ? 0 : n - 1;
                depth[n] = i + 1;
                ++n;
            }
            main0 = M[js + 1];
        }
        if (!(flags & OR_NO_BRANCH) && W > 0) {
            int32_t br[64];
            int32_t nb = 0;
            if (topk_row != NULL) {
                for (int32_t r = 0; r < Kn && nb < W; ++r)
                    if (topk_row[r] >= 0)
                        br[nb++] = topk_row[r];
            } else {
                for (int32_t r = 0; r < n_cand && nb < W; ++r) {
                    int32_t t = M[cand[r] + 1];
                    int dup = 0;
                    for (int32_t e = 0; e < nb; ++e)
                        if (br[e] == t)
                            dup = 1;
                    if (!dup)
                        br[nb++] = t;
                }
            }
            if (hit == OR_LEX) { /* Eq. 11 */
                int32_t m = 0;
                for (int32_t e = 0; e < nb; ++e)
                    if (br[e] != main0)
                        br[m++] = br[e];
                nb = m;
            }
            int want_succ = !(flags & OR_NO_SUCC) &&
                            (hit == OR_SEM || (flags & OR_SUCC_ON_STRICT));
            int32_t *tc = (int32_t *)malloc(sizeof(int32_t) * (size_t)k);
            double *sc = (double *)malloc(sizeof(double) * (size_t)k);
            for (int32_t e = 0; e < nb; ++e) {
                int32_t bnode = n;
                tok[n] = br[e];
                par[n] = 0;
                depth[n] = 1;
                ++n;
                if (!want_succ)
                    continue;
                int32_t c = oracle_successor_candidates_emb(M, len, R, d, E, de, tau,
                                                            js, br[e], k, tc, sc);
                if (c == 0)
                    continue;
                int32_t best = 0;
                for (int32_t i = 1; i < c; ++i)
                    if (better(sc[i], tc[i], sc[best], tc[best]))
                        best = i;
                int32_t tb = tc[best];
                int32_t prev = bnode;
                int32_t added = 0;
                for (int32_t i = 1; i <= succ_len && tb + i <= len - 1; ++i) {
                    tok[n] = M[tb + i];
                    par[n] = prev;
                    depth[n] = depth[prev] + 1;
                    prev = n;
                    ++n;
                    ++added;
                }
                if (added > 0)
                    ++succ_ext;
            }
            free(tc);
            free(sc);
        }
    }

    for (int32_t i = 0; i < n; ++i) {
        pos[i] = len - 1 + depth[i];
        for (int32_t a = i; a >= 0; a = par[a])
            mask[(size_t)i * nmax + a] = 1;
    }
    *n_nodes = n;
    free(depth);
    return succ_ext;
}

/* The draft tree of the single-cache reading (no embedding table). */
int32_t oracle_tree_from(const int32_t *M, int32_t len, const uint16_t *R,
                         int32_t d, int32_t hit, const int32_t *cand,
                         int32_t n_cand, const int32_t *topk_row, int32_t Kn,
                         int32_t k, int32_t W, int32_t D, int32_t succ_len,
                         uint32_t flags, int32_t nmax, int32_t *anchor,
                         int32_t *tok, int32_t *par, int32_t *pos,
                         uint8_t *mask, int32_t *n_nodes)
{
    return oracle_tree_from_emb(M, len, R, d, NULL, 0, 0.0, hit, cand, n_cand, topk_row, Kn,
                                k, W, D, succ_len, flags, nmax, anchor, tok, par, pos, mask,
                                n_nodes);
}

/*
 * One full draft-construction step for B sequences laid out as the library
 * lays them out: tokens[B][ld], reps[B][ld][d], query[B][d],
 * next_topk[B][ld][Kn] (may be NULL), and optionally a token-embedding table
 * E[V][de] (may be NULL).  Per sequence: Eq. 3 -> (if empty and the fallback
 * is on) Eq. 4 -> Eq. 5 -> Eq. 6-7 -> Eq. 8-15 -> tree.
 *
 * Without E the fallback scores the representation cache itself (the
 * single-cache reading: row j against the query), and those scores are also
 * the rerank scores.  With E the fallback scores token embeddings as Eq. 4
 * prints it, cos(E[M[j]], E[a]), keeps the best k, and Eq. 6 then reranks
 * them by cos(R[j], q); successor drafting backs off to the same embedding
 * fallback for a branch token that never occurs (Sec. 3.5).
 *
 * Outputs per sequence b: hit[b], match_n[b], anchor[b], cand[b][k],
 * score[b][k] (the ranking scores; padding -1 / 0), n_cand[b], tree arrays
 * [b][nmax] (mask [b][nmax][nmax]) and n_nodes[b]; stats[4] = lexical,
 * semantic and empty retrievals and successor extensions.  A sequence whose
 * length is outside [1, ld] gets hit NONE and n_nodes 0.  With
 * NO_LEX_RERANK the lexical scores are NaN (not computed).
 */
void oracle_step_emb(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                     const uint16_t *reps, int32_t d, const uint16_t *query,
                     const uint16_t *E, int32_t de,
                     const int32_t *next_topk, int32_t Kn, int32_t B,
                     int32_t n_max, int32_t k, int32_t W, int32_t D,
                     int32_t succ_len, double tau, uint32_t flags, int32_t nmax,
                     int32_t *hit, int32_t *match_n, int32_t *anchor,
                     int32_t *cand, double *score, int32_t *n_cand, int32_t *tok,
                     int32_t *par, int32_t *pos, uint8_t *mask, int32_t *n_nodes,
                     int64_t *stats)
{
    for (int32_t s = 0; s < 4; ++s)
        stats[s] = 0;
    for (int32_t b = 0; b < B; ++b) {
        const int32_t *M = tokens + (int64_t)b * ld;
        const uint16_t *R = reps + (int64_t)b * ld * d;
        const uint16_t *q = query + (int64_t)b * d;
        int32_t len = lengths[b];
        int32_t *cb = cand + (int64_t)b * k;
        double *sb = score + (int64_t)b * k;
        for (int32_t i = 0; i < k; ++i) {
            cb[i] = -1;
            sb[i] = 0.0;
        }
        hit[b] = OR_NONE;
        match_n[b] = 0;
        anchor[b] = -1;
        n_cand[b] = 0;
        int32_t *tb = tok + (int64_t)b * nmax;
        int32_t *pb = par + (int64_t)b * nmax;
        int32_t *ob = pos + (int64_t)b * nmax;
        uint8_t *mb = mask + (int64_t)b * nmax * nmax;
        if (len < 1 || len > ld) {
            for (int32_t i = 0; i < nmax; ++i)
                tb[i] = pb[i] = ob[i] = -1;
            memset(mb, 0, (size_t)nmax * (size_t)nmax);
            n_nodes[b] = 0;
            stats[2]++;
            continue;
        }
        int32_t nc = 0;
        if (oracle_lexical(M, len, n_max, k, &match_n[b], cb, &nc)) {
            hit[b] = OR_LEX;
            if (flags & OR_NO_LEX_RERANK) {
                for (int32_t i = 0; i < nc; ++i)
                    sb[i] = NAN;
            } else {
                oracle_rerank(R, d, q, cb, sb, nc);
            }
        } else if (!(flags & OR_NO_SEMANTIC)) {
            if (E != NULL) {
                nc = oracle_semantic_emb(M, len, E, de, k, tau, cb, sb);
                oracle_rerank(R, d, q, cb, sb, nc);
            } else {
                nc = oracle_semantic(R, d, q, len, k, tau, cb, sb);
            }
            hit[b] = nc > 0 ? OR_SEM : OR_NONE;
        }
        n_cand[b] = nc;
        const int32_t *row = NULL;
        if (next_topk != NULL && nc > 0)
            row = next_topk + ((int64_t)b * ld + cb[0]) * Kn;
        int32_t ext = oracle_tree_from_emb(M, len, R, d, E, de, tau, hit[b], cb, nc, row, Kn,
                                           k, W, D, succ_len, flags, nmax,
                                           &anchor[b], tb, pb, ob, mb, &n_nodes[b]);
        if (hit[b] == OR_LEX)
            stats[0]++;
        else if (hit[b] == OR_SEM)
            stats[1]++;
        else
            stats[2]++;
        stats[3] += ext;
    }
}

/* oracle_step_emb without an embedding table (the single-cache reading). */
void oracle_step(const int32_t *tokens, int64_t ld, const int32_t *lengths,
                 const uint16_t *reps, int32_t d, const uint16_t *query,
                 const int32_t *next_topk, int32_t Kn, int32_t B,
                 int32_t n_max, int32_t k, int32_t W, int32_t D,
                 int32_t succ_len, double tau, uint32_t flags, int32_t nmax,
                 int32_t *hit, int32_t *match_n, int32_t *anchor,
                 int32_t *cand, double *score, int32_t *n_cand, int32_t *tok,
                 int32_t *par, int32_t *pos, uint8_t *mask, int32_t *n_nodes,
                 int64_t *stats)
{
    oracle_step_emb(tokens, ld, lengths, reps, d, query, NULL, 0, next_topk, Kn, B, n_max, k,
                    W, D, succ_len, tau, flags, nmax, hit, match_n, anchor, cand, score,
                    n_cand, tok, par, pos, mask, n_nodes, stats);
}

/*
 * Greedy verification of one draft tree (Sec. 3.6; Appendix C, Eq. 16: at
 * temperature 0 a draft token is accepted iff it equals the target model's
 * greedy choice).  logits[i][v] (bf16 bits, rows V apart) are the target's
 * next-token logits after tree node i; its choice there is the first index
 * of the maximum.  From the root, the child of the current node whose token
 * equals the choice at the current node is accepted, until there is none.
 * The new tokens are the accepted draft tokens followed by the choice after
 * the last accepted node (the bonus token of Algorithm 1); path[0] is the
 * root and path[i] the i-th accepted node.  Returns the number of accepted
 * draft tokens; *n_new is that plus one (0 for an empty tree).
 */
int32_t oracle_verify_greedy(const uint16_t *logits, int32_t V, const int32_t *tok,
                             const int32_t *par, int32_t n_nodes, int32_t *new_tokens,
                             int32_t *path, int32_t *n_new)
{
    *n_new = 0;
    if (n_nodes < 1)
        return 0;
    int32_t cur = 0, n_acc = 0;
    for (;;) {
        const uint16_t *row = logits + (int64_t)cur * V;
        int32_t best = 0;
        for (int32_t v = 1; v < V; ++v)
            if (bf16_bits_to_double(row[v]) > bf16_bits_to_double(row[best]))
                best = v;
        path[n_acc] = cur;
        int32_t next = -1;
        for (int32_t i = 1; i < n_nodes; ++i)
            if (par[i] == cur && tok[i] == best) {
                next = i;
                break;
            }
        if (next < 0) {
            new_tokens[n_acc] = best;  /* the bonus token */
            *n_new = n_acc + 1;
            return n_acc;
        }
        new_tokens[n_acc] = tok[next];
        ++n_acc;
        cur = next;
    }
}

/*
 * Verification and the memory append for B sequences (Algorithm 1: append
 * the accepted tokens and the bonus token, update the context).  Per
 * sequence: oracle_verify_greedy on logits[b] ([N][V]); then, if
 * len + n_new <= ld, tokens[b][len + i] = new_tokens[i], lengths[b] += n_new
 * and, when node_reps ([B][N][d]) is given, reps[b][len + i] =
 * node_reps[b][path[i]] (the hidden state after each new position's
 * predecessor) and query[b] = node_reps[b][path[n_new - 1]]; otherwise
 * full[b] = 1 and nothing is appended.  n_accept[b], new_tokens[b][N]
 * (padding -1) and n_new[b] are always written.
 */
void oracle_accept_greedy(const uint16_t *logits, int32_t V, const int32_t *tok,
                          const int32_t *par, const int32_t *n_nodes, int32_t B, int32_t N,
                          int32_t *n_accept, int32_t *new_tokens, int32_t *n_new,
                          int32_t *tokens, int64_t ld, int32_t *lengths,
                          const uint16_t *node_reps, uint16_t *reps, int32_t d,
                          uint16_t *query, int32_t *full)
{
    int32_t *path = (int32_t *)malloc(sizeof(int32_t) * (size_t)(N > 0 ? N : 1));
    for (int32_t b = 0; b < B; ++b) {
        int32_t *nt = new_tokens + (int64_t)b * N;
        for (int32_t i = 0; i < N; ++i)
            nt[i] = -1;
        full[b] = 0;
        n_accept[b] = oracle_verify_greedy(logits + (int64_t)b * N * V, V,
                                           tok + (int64_t)b * N, par + (int64_t)b * N,
                                           n_nodes[b], nt, path, &n_new[b]);
        if (tokens == NULL || n_new[b] == 0)
            continue;
        int32_t len = lengths[b];
        if (len + n_new[b] > ld) {
            full[b] = 1;
            continue;
        }
        for (int32_t i = 0; i < n_new[b]; ++i)
            tokens[(int64_t)b * ld + len + i] = nt[i];
        if (node_reps != NULL) {
            for (int32_t i = 0; i < n_new[b]; ++i)
                memcpy(reps + ((int64_t)b * ld + len + i) * d,
                       node_reps + ((int64_t)b * N + path[i]) * d, sizeof(uint16_t) * (size_t)d);
            memcpy(query + (int64_t)b * d, node_reps + ((int64_t)b * N + path[n_new[b] - 1]) * d,
                   sizeof(uint16_t) * (size_t)d);
        }
        lengths[b] = len + n_new[b];
    }
    free(path);
}
