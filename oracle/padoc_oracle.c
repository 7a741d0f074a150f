/*
 * padoc_oracle.c -- plain, slow fp64 CPU oracle for PaDoc ancestor-masked attention.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may include, link, load or call this
 * file: only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference leg use it.
 * It shares no header, helper, table or constant with the CUDA library; its page description is
 * its own flat int32 layout.
 *
 * What it computes (paper, Sec. 3.2 "Training Paradigm", Eq. for Anc(B_k) and Anc(Y_k);
 * App. C.1 "Attention Backends", the relation Q_M -> K_M and Q_{Y_k} -> [K_{M<=f_k}; K_{Y_k}];
 * App. E.1, the additive-bias softmax Attn(Q) = softmax(QK^T/sqrt(d) + A_M) V and Algorithm 1):
 *
 *   A page is the packed sequence [ X (P tokens) | layout stream B (L tokens) | Y_1 | ... | Y_N ].
 *   Node X and the layout stream are each causal; the layout stream sees all of X
 *   (Anc(B_k) = {X, B_<k} and causal inside B_k make the layout stream one causal sequence after X).
 *   Branch Y_k sees all of X, the first f_k layout tokens (B_<=k at its fork) and its own non-future
 *   tokens (Anc(Y_k) = {X, B_<=k}). Tokens of different pages never see each other.
 *
 *   For every query and head h (KV head g = h / (Hq/Hkv)):
 *     s_j = scale * sum_c Q[c] K_j[c]  over visible j,  lse = ln sum_j exp(s_j),
 *     O   = sum_j exp(s_j - lse) V_j.
 *
 * Two independent formulations are given, as the paper gives two realizations that expose the
 * same visibility (App. C.1): a dense visibility test written from node membership
 * ("Dense SDPA", the paper's reference implementation), and a per-branch gather of
 * [M_<=f_k ; Y_k] with bottom-right-aligned causal attention ("Tree-varlen").
 *
 * The backward (oracle_prefill_bwd) is the chain rule of that softmax attention for an upstream
 * gradient dO: dQ, dK, dV under the same visibility, with every shared-stream key's gradient summed
 * over all queries that see it (the scatter-add of the tree-varlen gather's backward, App. C.1).
 *
 * Readings of the paper used here (each also listed in the design notes):
 *   - f_k is the number of layout-stream tokens visible to branch k (Alg. 1 copies the layout
 *     row before the boundary output is appended; Sec. E.1). Any f_k in [0, L], in any order.
 *   - the prefix X is causal (App. C.1 states Q_M -> K_M causal, M contains the image).
 *   - every branch has >= 1 token (its branch-start token, Sec. 3.2), so no row is empty.
 *   - decode: a stream's private history includes the token being decoded (Alg. 1 appends the
 *     live streams' inputs before decoding them).
 *   - LSE is the natural-log log-sum-exp of the scaled scores.
 *
 * Floating point: every input (fp32 holding bf16 or fp32 values) is converted exactly to double
 * and all arithmetic is double. Each query's softmax is evaluated in key order j ascending.
 *
 * Page description (flat int32): pln[3*p + 0] = P, pln[3*p + 1] = L, pln[3*p + 2] = N;
 * fork[] and blen[] hold f_k and n_k of all pages' branches back to back in page order.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------------------------ */
/* Page bookkeeping                                                                             */
/* ------------------------------------------------------------------------------------------ */

static int64_t page_tokens(const int32_t *pln, const int32_t *blen, int64_t branch_off, int p)
{
    int64_t s = (int64_t)pln[3 * p] + pln[3 * p + 1];
    for (int k = 0; k < pln[3 * p + 2]; ++k) s += blen[branch_off + k];
    return s;
}

/* Total packed tokens over all pages. */
int64_t oracle_total_tokens(const int32_t *pln, int32_t num_pages, const int32_t *blen)
{
    int64_t t = 0, boff = 0;
    for (int p = 0; p < num_pages; ++p) {
        t += page_tokens(pln, blen, boff, p);
        boff += pln[3 * p + 2];
    }
    return t;
}

/* Node of a page-local position: kind 0 = image/prompt node X (index i), 1 = layout stream
 * (index l), 2 = content node Y_k (branch k, index i). */
typedef struct { int kind, branch, index; } node_pos;

static node_pos node_of(const int32_t *pln_p, const int32_t *fork_p, const int32_t *blen_p, int64_t pos)
{
    (void)fork_p;
    node_pos r;
    const int64_t P = pln_p[0], L = pln_p[1];
    const int N = pln_p[2];
    if (pos < P) { r.kind = 0; r.branch = -1; r.index = (int)pos; return r; }
    if (pos < P + L) { r.kind = 1; r.branch = -1; r.index = (int)(pos - P); return r; }
    int64_t base = P + L;
    for (int k = 0; k < N; ++k) {
        if (pos < base + blen_p[k]) { r.kind = 2; r.branch = k; r.index = (int)(pos - base); return r; }
        base += blen_p[k];
    }
    r.kind = -1; r.branch = -1; r.index = -1;
    return r;
}

/* Visibility from the ancestor sets (Sec. 3.2): may the token at page-local position q attend to
 * the token at page-local position j? */
static int visible_by_ancestors(const int32_t *pln_p, const int32_t *fork_p, const int32_t *blen_p,
                                int64_t q, int64_t j)
{
    node_pos a = node_of(pln_p, fork_p, blen_p, q);
    node_pos b = node_of(pln_p, fork_p, blen_p, j);
    if (a.kind == 0) {                       /* X: causal inside X */
        return b.kind == 0 && b.index <= a.index;
    }
    if (a.kind == 1) {                       /* layout stream: all of X, causal inside the stream */
        if (b.kind == 0) return 1;
        return b.kind == 1 && b.index <= a.index;
    }
    /* content node Y_k: X, B_<=k (the first f_k layout tokens) and its own non-future tokens */
    if (b.kind == 0) return 1;
    if (b.kind == 1) return b.index < fork_p[a.branch];
    if (b.kind == 2) return b.branch == a.branch && b.index <= a.index;
    return 0;
}

/* Dense Boolean visibility of one page, row-major [S_p][S_p] (Sec. 3.2 / App. C.1 "Dense SDPA"). */
void oracle_dense_mask(const int32_t *pln, int32_t num_pages, const int32_t *fork, const int32_t *blen,
                       int32_t page, uint8_t *mask)
{
    int64_t boff = 0;
    for (int p = 0; p < page; ++p) boff += pln[3 * p + 2];
    (void)num_pages;
    const int32_t *pp = pln + 3 * page;
    const int64_t S = page_tokens(pln, blen, boff, page);
    for (int64_t q = 0; q < S; ++q)
        for (int64_t j = 0; j < S; ++j)
            mask[q * S + j] = (uint8_t)visible_by_ancestors(pp, fork + boff, blen + boff, q, j);
}

/* Per-query visible spans in absolute packed indices, [T][4] = {kv0_begin, kv0_end, kv1_begin,
 * kv1_end}, read off the ancestor sets: X token i sees [X_0, X_i]; layout token l sees X and
 * [B_0, B_l], which is one contiguous run; branch token (k, i) sees X followed by f_k layout tokens,
 * and [Y_k,0 .. Y_k,i]. An empty second span is written as {kv0_end, kv0_end}. */
void oracle_spans(const int32_t *pln, int32_t num_pages, const int32_t *fork, const int32_t *blen,
                  int32_t *spans)
{
    int64_t pbase = 0, boff = 0;
    for (int p = 0; p < num_pages; ++p) {
        const int32_t *pp = pln + 3 * p;
        const int64_t S = page_tokens(pln, blen, boff, p);
        for (int64_t q = 0; q < S; ++q) {
            node_pos a = node_of(pp, fork + boff, blen + boff, q);
            int32_t *o = spans + 4 * (pbase + q);
            if (a.kind == 0 || a.kind == 1) {
                o[0] = (int32_t)pbase;
                o[1] = (int32_t)(pbase + q + 1);
                o[2] = o[1];
                o[3] = o[1];
            } else {
                int64_t ybase = pp[0] + pp[1];
                for (int k = 0; k < a.branch; ++k) ybase += blen[boff + k];
                o[0] = (int32_t)pbase;
                o[1] = (int32_t)(pbase + pp[0] + fork[boff + a.branch]);
                o[2] = (int32_t)(pbase + ybase);
                o[3] = (int32_t)(pbase + q + 1);
            }
        }
        pbase += S;
        boff += pp[2];
    }
}

/* ------------------------------------------------------------------------------------------ */
/* Softmax attention of one query row over an explicit list of key rows                        */
/* ------------------------------------------------------------------------------------------ */

/* o[d] = sum_j softmax(scale * q.k_j) v_j over keys[0..nk); returns lse (natural log).
 * k_rows[j] / v_rows[j] point at float[d]. nk == 0 gives o = 0, lse = -inf. */
static double attend_rows(const float *q, const float *const *k_rows, const float *const *v_rows,
                          int64_t nk, int d, double scale, double *s_buf, double *o)
{
    for (int c = 0; c < d; ++c) o[c] = 0.0;
    if (nk == 0) return -INFINITY;
    double mx = -INFINITY;
    for (int64_t j = 0; j < nk; ++j) {
        double acc = 0.0;
        for (int c = 0; c < d; ++c) acc += (double)q[c] * (double)k_rows[j][c];
        s_buf[j] = scale * acc;
        if (s_buf[j] > mx) mx = s_buf[j];
    }
    double sum = 0.0;
    for (int64_t j = 0; j < nk; ++j) sum += exp(s_buf[j] - mx);
    const double lse = mx + log(sum);
    for (int64_t j = 0; j < nk; ++j) {
        const double w = exp(s_buf[j] - lse);
        for (int c = 0; c < d; ++c) o[c] += w * (double)v_rows[j][c];
    }
    return lse;
}

/* ------------------------------------------------------------------------------------------ */
/* Packed prefill, formulation 1: dense visibility from node membership                          */
/* ------------------------------------------------------------------------------------------ */

/* q: [T][Hq][d], k, v: [T][Hkv][d] (packed order), o: [T][Hq][d], lse: [T][Hq]. */
void oracle_prefill_dense(const int32_t *pln, int32_t num_pages, const int32_t *fork, const int32_t *blen,
                          const float *q, const float *k, const float *v, int32_t Hq, int32_t Hkv, int32_t d,
                          double scale, double *o, double *lse)
{
    int64_t pbase = 0, boff = 0;
    const int group = Hq / Hkv;
    for (int p = 0; p < num_pages; ++p) {
        const int32_t *pp = pln + 3 * p;
        const int64_t S = page_tokens(pln, blen, boff, p);
        const int32_t *fk = fork + boff, *bl = blen + boff;
#pragma omp parallel
        {
            const float **kr = (const float **)malloc(sizeof(float *) * (size_t)(S > 0 ? S : 1));
            const float **vr = (const float **)malloc(sizeof(float *) * (size_t)(S > 0 ? S : 1));
            double *sb = (double *)malloc(sizeof(double) * (size_t)(S > 0 ? S : 1));
#pragma omp for schedule(dynamic, 4)
            for (int64_t qi = 0; qi < S; ++qi) {
                int64_t nk = 0;
                int64_t *vis = (int64_t *)sb; /* visible page-local key positions, ascending */
                for (int64_t j = 0; j < S; ++j)
                    if (visible_by_ancestors(pp, fk, bl, qi, j)) vis[nk++] = j;
                int64_t *visc = (int64_t *)malloc(sizeof(int64_t) * (size_t)(nk > 0 ? nk : 1));
                memcpy(visc, vis, sizeof(int64_t) * (size_t)nk);
                for (int h = 0; h < Hq; ++h) {
                    const int g = h / group;
                    for (int64_t c = 0; c < nk; ++c) {
                        kr[c] = k + ((pbase + visc[c]) * Hkv + g) * d;
                        vr[c] = v + ((pbase + visc[c]) * Hkv + g) * d;
                    }
                    const int64_t row = (pbase + qi) * Hq + h;
                    lse[row] = attend_rows(q + row * d, kr, vr, nk, d, scale, sb, o + row * d);
                }
                free(visc);
            }
            free(kr); free(vr); free(sb);
        }
        pbase += S;
        boff += pp[2];
    }
}

/* The dense formulation on selected query rows only (sampled checks of large packed batches):
 * rows[i] is an absolute packed row; q_sel: [n_rows][Hq][d] holds those rows' queries; k, v the whole
 * packed [T][Hkv][d]; o: [n_rows][Hq][d], lse: [n_rows][Hq]. Each row's visible keys come from
 * visible_by_ancestors exactly as in oracle_prefill_dense, so a selected row's result is that
 * function's row bit for bit. */
void oracle_prefill_dense_rows(const int32_t *pln, int32_t num_pages, const int32_t *fork, const int32_t *blen,
                               const float *q_sel, const float *k, const float *v, int32_t Hq, int32_t Hkv, int32_t d,
                               double scale, int64_t n_rows, const int64_t *rows, double *o, double *lse)
{
    const int group = Hq / Hkv;
    /* page of each row: page starts and branch offsets */
    int64_t *pstart = (int64_t *)malloc(sizeof(int64_t) * (size_t)(num_pages + 1));
    int64_t *bstart = (int64_t *)malloc(sizeof(int64_t) * (size_t)(num_pages + 1));
    pstart[0] = 0; bstart[0] = 0;
    for (int p = 0; p < num_pages; ++p) {
        pstart[p + 1] = pstart[p] + page_tokens(pln, blen, bstart[p], p);
        bstart[p + 1] = bstart[p] + pln[3 * p + 2];
    }
#pragma omp parallel
    {
        int64_t cap = 0;
        const float **kr = NULL, **vr = NULL;
        double *sb = NULL;
        int64_t *vis = NULL;
#pragma omp for schedule(dynamic, 1)
        for (int64_t i = 0; i < n_rows; ++i) {
            int p = 0;
            while (p + 1 < num_pages && rows[i] >= pstart[p + 1]) ++p;
            const int64_t S = pstart[p + 1] - pstart[p], qi = rows[i] - pstart[p];
            if (S > cap) {
                cap = S;
                kr = (const float **)realloc((void *)kr, sizeof(float *) * (size_t)cap);
                vr = (const float **)realloc((void *)vr, sizeof(float *) * (size_t)cap);
                sb = (double *)realloc(sb, sizeof(double) * (size_t)cap);
                vis = (int64_t *)realloc(vis, sizeof(int64_t) * (size_t)cap);
            }
            int64_t nk = 0;
            for (int64_t j = 0; j < S; ++j)
                if (visible_by_ancestors(pln + 3 * p, fork + bstart[p], blen + bstart[p], qi, j)) vis[nk++] = j;
            for (int h = 0; h < Hq; ++h) {
                const int g = h / group;
                for (int64_t c = 0; c < nk; ++c) {
                    kr[c] = k + ((pstart[p] + vis[c]) * Hkv + g) * d;
                    vr[c] = v + ((pstart[p] + vis[c]) * Hkv + g) * d;
                }
                lse[i * Hq + h] = attend_rows(q_sel + (i * Hq + h) * d, kr, vr, nk, d, scale, sb, o + (i * Hq + h) * d);
            }
        }
        free((void *)kr); free((void *)vr); free(sb); free(vis);
    }
    free(pstart); free(bstart);
}

/* ------------------------------------------------------------------------------------------ */
/* Packed prefill, formulation 2: tree-varlen gather with bottom-right causal alignment          */
/* ------------------------------------------------------------------------------------------ */

/* The shared stream M = [X | B] is one causal problem. Branch k gathers the key/value rows
 * [M_0 .. M_{P+f_k-1}] followed by Y_k, and its i-th query sees gathered rows c <= i + (P + f_k)
 * (FlashAttention's bottom-right alignment of an n_k-query, (P+f_k+n_k)-key causal problem). */
void oracle_prefill_gather(const int32_t *pln, int32_t num_pages, const int32_t *fork, const int32_t *blen,
                           const float *q, const float *k, const float *v, int32_t Hq, int32_t Hkv, int32_t d,
                           double scale, double *o, double *lse)
{
    int64_t pbase = 0, boff = 0;
    const int group = Hq / Hkv;
    for (int p = 0; p < num_pages; ++p) {
        const int32_t *pp = pln + 3 * p;
        const int64_t P = pp[0], L = pp[1];
        const int N = pp[2];
        const int64_t S = page_tokens(pln, blen, boff, p);
        const int64_t M = P + L;
        /* causal problem over M */
#pragma omp parallel
        {
            const float **kr = (const float **)malloc(sizeof(float *) * (size_t)(S > 0 ? S : 1));
            const float **vr = (const float **)malloc(sizeof(float *) * (size_t)(S > 0 ? S : 1));
            double *sb = (double *)malloc(sizeof(double) * (size_t)(S > 0 ? S : 1));
#pragma omp for schedule(dynamic, 4) collapse(2)
            for (int64_t qi = 0; qi < M; ++qi) {
                for (int h = 0; h < Hq; ++h) {
                    const int g = h / group;
                    for (int64_t j = 0; j <= qi; ++j) {
                        kr[j] = k + ((pbase + j) * Hkv + g) * d;
                        vr[j] = v + ((pbase + j) * Hkv + g) * d;
                    }
                    const int64_t row = (pbase + qi) * Hq + h;
                    lse[row] = attend_rows(q + row * d, kr, vr, qi + 1, d, scale, sb, o + row * d);
                }
            }
            free(kr); free(vr); free(sb);
        }
        /* one causal problem per branch over the gathered [M_<f_k ; Y_k] */
        int64_t ybase = M;
        for (int b = 0; b < N; ++b) {
            const int64_t n = blen[boff + b];
            const int64_t vis_prefix = P + fork[boff + b];
            const int64_t lkv = vis_prefix + n;
            /* gather (row pointers into packed K/V; no arithmetic is shared with formulation 1) */
            int64_t *gidx = (int64_t *)malloc(sizeof(int64_t) * (size_t)(lkv > 0 ? lkv : 1));
            for (int64_t c = 0; c < vis_prefix; ++c) gidx[c] = pbase + c;
            for (int64_t c = 0; c < n; ++c) gidx[vis_prefix + c] = pbase + ybase + c;
#pragma omp parallel
            {
                const float **kr = (const float **)malloc(sizeof(float *) * (size_t)(lkv > 0 ? lkv : 1));
                const float **vr = (const float **)malloc(sizeof(float *) * (size_t)(lkv > 0 ? lkv : 1));
                double *sb = (double *)malloc(sizeof(double) * (size_t)(lkv > 0 ? lkv : 1));
#pragma omp for schedule(dynamic, 4) collapse(2)
                for (int64_t i = 0; i < n; ++i) {
                    for (int h = 0; h < Hq; ++h) {
                        const int g = h / group;
                        const int64_t last = i + (lkv - n); /* bottom-right alignment */
                        for (int64_t c = 0; c <= last; ++c) {
                            kr[c] = k + (gidx[c] * Hkv + g) * d;
                            vr[c] = v + (gidx[c] * Hkv + g) * d;
                        }
                        const int64_t row = (pbase + ybase + i) * Hq + h;
                        lse[row] = attend_rows(q + row * d, kr, vr, last + 1, d, scale, sb, o + row * d);
                    }
                }
                free(kr); free(vr); free(sb);
            }
            free(gidx);
            ybase += n;
        }
        pbase += S;
        boff += N;
    }
}

/* ------------------------------------------------------------------------------------------ */
/* Decode step (Algorithm 1): one query per live stream over its mask row                       */
/* ------------------------------------------------------------------------------------------ */

/* Logical (unpaged) cache: page p's shared stream K/V rows are stream_k/v[page_off[p] ..
 * page_off[p] + page_len[p]) as [rows][Hkv][d]; stream s's private history (its own tokens,
 * including the one being decoded) is priv_k/v[priv_off[s] .. priv_off[s] + priv_len[s]).
 * Stream s of page stream_page[s] sees shared rows [0, shared_len[s]) and all its private rows.
 * q: [S][Hq][d]; o: [S][Hq][d]; lse: [S][Hq]. */
void oracle_decode(int32_t num_streams, const int32_t *stream_page, const int32_t *shared_len,
                   const int32_t *priv_len, const int64_t *page_off, const int64_t *priv_off,
                   const float *stream_k, const float *stream_v, const float *priv_k, const float *priv_v,
                   const float *q, int32_t Hq, int32_t Hkv, int32_t d, double scale, double *o, double *lse)
{
    const int group = Hq / Hkv;
#pragma omp parallel
    {
        int64_t cap = 0;
        const float **kr = NULL, **vr = NULL;
        double *sb = NULL;
#pragma omp for schedule(dynamic, 1) collapse(2)
        for (int s = 0; s < num_streams; ++s) {
            for (int h = 0; h < Hq; ++h) {
                const int g = h / group;
                const int64_t nk = (int64_t)shared_len[s] + priv_len[s];
                if (nk > cap) {
                    cap = nk;
                    kr = (const float **)realloc((void *)kr, sizeof(float *) * (size_t)cap);
                    vr = (const float **)realloc((void *)vr, sizeof(float *) * (size_t)cap);
                    sb = (double *)realloc(sb, sizeof(double) * (size_t)cap);
                }
                int64_t c = 0;
                const int64_t po = page_off[stream_page[s]];
                for (int64_t j = 0; j < shared_len[s]; ++j, ++c) {
                    kr[c] = stream_k + ((po + j) * Hkv + g) * d;
                    vr[c] = stream_v + ((po + j) * Hkv + g) * d;
                }
                for (int64_t j = 0; j < priv_len[s]; ++j, ++c) {
                    kr[c] = priv_k + ((priv_off[s] + j) * Hkv + g) * d;
                    vr[c] = priv_v + ((priv_off[s] + j) * Hkv + g) * d;
                }
                const int64_t row = (int64_t)s * Hq + h;
                lse[row] = attend_rows(q + row * d, kr, vr, nk, d, scale, sb, o + row * d);
            }
        }
        free((void *)kr); free((void *)vr); free(sb);
    }
}

/* The same decode step over fp64 K/V rows (a dequantized cache, whose values code_value * scale
 * need more bits than fp32 holds); q stays fp32. Arguments as oracle_decode. */
static double attend_rows_f64(const float *q, const double *const *k_rows, const double *const *v_rows, int64_t nk,
                              int d, double scale, double *s_buf, double *o)
{
    for (int c = 0; c < d; ++c) o[c] = 0.0;
    if (nk == 0) return -INFINITY;
    double mx = -INFINITY;
    for (int64_t j = 0; j < nk; ++j) {
        double acc = 0.0;
        for (int c = 0; c < d; ++c) acc += (double)q[c] * k_rows[j][c];
        s_buf[j] = scale * acc;
        if (s_buf[j] > mx) mx = s_buf[j];
    }
    double sum = 0.0;
    for (int64_t j = 0; j < nk; ++j) sum += exp(s_buf[j] - mx);
    const double lse = mx + log(sum);
    for (int64_t j = 0; j < nk; ++j) {
        const double w = exp(s_buf[j] - lse);
        for (int c = 0; c < d; ++c) o[c] += w * v_rows[j][c];
    }
    return lse;
}

void oracle_decode_f64(int32_t num_streams, const int32_t *stream_page, const int32_t *shared_len,
                       const int32_t *priv_len, const int64_t *page_off, const int64_t *priv_off,
                       const double *stream_k, const double *stream_v, const double *priv_k, const double *priv_v,
                       const float *q, int32_t Hq, int32_t Hkv, int32_t d, double scale, double *o, double *lse)
{
    const int group = Hq / Hkv;
#pragma omp parallel
    {
        int64_t cap = 0;
        const double **kr = NULL, **vr = NULL;
        double *sb = NULL;
#pragma omp for schedule(dynamic, 1) collapse(2)
        for (int s = 0; s < num_streams; ++s) {
            for (int h = 0; h < Hq; ++h) {
                const int g = h / group;
                const int64_t nk = (int64_t)shared_len[s] + priv_len[s];
                if (nk > cap) {
                    cap = nk;
                    kr = (const double **)realloc((void *)kr, sizeof(double *) * (size_t)cap);
                    vr = (const double **)realloc((void *)vr, sizeof(double *) * (size_t)cap);
                    sb = (double *)realloc(sb, sizeof(double) * (size_t)cap);
                }
                int64_t c = 0;
                const int64_t po = page_off[stream_page[s]];
                for (int64_t j = 0; j < shared_len[s]; ++j, ++c) {
                    kr[c] = stream_k + ((po + j) * Hkv + g) * d;
                    vr[c] = stream_v + ((po + j) * Hkv + g) * d;
                }
                for (int64_t j = 0; j < priv_len[s]; ++j, ++c) {
                    kr[c] = priv_k + ((priv_off[s] + j) * Hkv + g) * d;
                    vr[c] = priv_v + ((priv_off[s] + j) * Hkv + g) * d;
                }
                const int64_t row = (int64_t)s * Hq + h;
                lse[row] = attend_rows_f64(q + row * d, kr, vr, nk, d, scale, sb, o + row * d);
            }
        }
        free((void *)kr); free((void *)vr); free(sb);
    }
}

/* ------------------------------------------------------------------------------------------ */
/* Merge of partial softmax results over a partition of the visible set                         */
/* ------------------------------------------------------------------------------------------ */

/* Softmax over a union of disjoint key sets: with per-part (O_s, lse_s),
 *   lse = ln sum_s exp(lse_s),  O = sum_s exp(lse_s - lse) O_s;  a part with lse_s = -inf weighs 0.
 * part_o: [S][rows][d], part_lse: [S][rows]; out_o: [rows][d]; out_lse: [rows]. */
void oracle_merge(const double *part_o, const double *part_lse, int32_t num_parts, int64_t rows, int32_t d,
                  double *out_o, double *out_lse)
{
    for (int64_t r = 0; r < rows; ++r) {
        double mx = -INFINITY;
        for (int s = 0; s < num_parts; ++s)
            if (part_lse[s * rows + r] > mx) mx = part_lse[s * rows + r];
        for (int c = 0; c < d; ++c) out_o[r * d + c] = 0.0;
        if (mx == -INFINITY) { out_lse[r] = -INFINITY; continue; }
        double sum = 0.0;
        for (int s = 0; s < num_parts; ++s) sum += exp(part_lse[s * rows + r] - mx);
        const double tot = mx + log(sum);
        for (int s = 0; s < num_parts; ++s) {
            const double w = exp(part_lse[s * rows + r] - tot);
            if (w == 0.0) continue;
            for (int c = 0; c < d; ++c) out_o[r * d + c] += w * part_o[(s * rows + r) * d + c];
        }
        out_lse[r] = tot;
    }
}

/* ------------------------------------------------------------------------------------------ */
/* Brute-force tile classification (prefill work list)                                          */
/* ------------------------------------------------------------------------------------------ */

/* For q-tile rows [qt*qb, min(T,(qt+1)*qb)) and k-tile columns [kt*kb, (kt+1)*kb), counts visible
 * (row, column) pairs by testing every pair against the ancestor rule (tokens of different pages
 * never see each other). kind[qt * num_kt + kt] = 0 if no pair is visible, 2 (FULL) if every
 * existing row sees all kb columns (so a tile reaching past T is never FULL), else 1 (PARTIAL).
 * Quadratic in T: small inputs only. */
void oracle_tile_kinds(const int32_t *pln, int32_t num_pages, const int32_t *fork, const int32_t *blen,
                       int32_t qb, int32_t kb, int8_t *kind)
{
    const int64_t T = oracle_total_tokens(pln, num_pages, blen);
    const int64_t nqt = (T + qb - 1) / qb, nkt = (T + kb - 1) / kb;
    /* page of every packed token and its page-local position */
    int32_t *pg = (int32_t *)malloc(sizeof(int32_t) * (size_t)(T > 0 ? T : 1));
    int64_t *loc = (int64_t *)malloc(sizeof(int64_t) * (size_t)(T > 0 ? T : 1));
    int64_t *boffs = (int64_t *)malloc(sizeof(int64_t) * (size_t)(num_pages > 0 ? num_pages : 1));
    int64_t t = 0, boff = 0;
    for (int p = 0; p < num_pages; ++p) {
        boffs[p] = boff;
        const int64_t S = page_tokens(pln, blen, boff, p);
        for (int64_t i = 0; i < S; ++i) { pg[t] = p; loc[t] = i; ++t; }
        boff += pln[3 * p + 2];
    }
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int64_t qt = 0; qt < nqt; ++qt) {
        for (int64_t kt = 0; kt < nkt; ++kt) {
            const int64_t r0 = qt * qb, r1 = (r0 + qb < T) ? r0 + qb : T;
            int64_t cnt = 0;
            for (int64_t r = r0; r < r1; ++r) {
                for (int64_t c = kt * kb; c < kt * kb + kb; ++c) {
                    if (c >= T || pg[c] != pg[r]) continue;
                    const int p = pg[r];
                    cnt += visible_by_ancestors(pln + 3 * p, fork + boffs[p], blen + boffs[p], loc[r], loc[c]);
                }
            }
            kind[qt * nkt + kt] = (int8_t)(cnt == 0 ? 0 : (cnt == (r1 - r0) * (int64_t)kb ? 2 : 1));
        }
    }
    free(pg); free(loc); free(boffs);
}

/* ------------------------------------------------------------------------------------------ */
/* Packed prefill backward: gradients of the ancestor-masked attention                          */
/* ------------------------------------------------------------------------------------------ */

/* The forward of every query row and head is s_j = scale * q.k_j over its visible keys j,
 * P_j = exp(s_j - lse), O = sum_j P_j v_j (Sec. 3.2 visibility, App. E.1 softmax). For an upstream
 * gradient dO of O, the chain rule through the softmax gives, per query row and head,
 *   dP_j = dO . v_j,   D = sum_j P_j dP_j,   dS_j = P_j (dP_j - D),   dQ = scale * sum_j dS_j k_j,
 * and every key j of KV head g collects over the queries i that see it and the query heads h that
 * read KV head g:
 *   dK_j = scale * sum_{i,h} dS_ij q_ih,   dV_j = sum_{i,h} P_ij dO_ih.
 * A shared-stream key is seen by the stream's later tokens and by every branch forked after it, so
 * its dK and dV sum over all of them: the scatter-add back onto the shared rows that the backward
 * of the tree-varlen gather performs (App. C.1). Visibility is the dense ancestor test above; lse
 * and D are recomputed here in fp64 from the inputs (nothing is taken from a forward output).
 *
 * q: [T][Hq][d], k, v: [T][Hkv][d], dout: [T][Hq][d] (packed order, fp32 holding exact values).
 * Only the selected rows are produced: q_sel[0..nq) (packed query rows) -> dq [nq][Hq][d];
 * k_sel[0..nk) (packed key rows) -> dk, dv [nk][Hkv][d]. Sums run over keys (dQ) or queries then
 * heads (dK, dV) in ascending order. */

typedef struct {
    int32_t *pg;        /* page of each packed token */
    int64_t *loc;       /* page-local position */
    int64_t *pbase;     /* first packed token of each page */
    int64_t *boffs;     /* first branch of each page in fork[] / blen[] */
    int64_t *ptok;      /* tokens of each page */
} page_index;

static void page_index_build(const int32_t *pln, int32_t num_pages, const int32_t *blen, int64_t T, page_index *ix)
{
    ix->pg = (int32_t *)malloc(sizeof(int32_t) * (size_t)(T > 0 ? T : 1));
    ix->loc = (int64_t *)malloc(sizeof(int64_t) * (size_t)(T > 0 ? T : 1));
    ix->pbase = (int64_t *)malloc(sizeof(int64_t) * (size_t)(num_pages > 0 ? num_pages : 1));
    ix->boffs = (int64_t *)malloc(sizeof(int64_t) * (size_t)(num_pages > 0 ? num_pages : 1));
    ix->ptok = (int64_t *)malloc(sizeof(int64_t) * (size_t)(num_pages > 0 ? num_pages : 1));
    int64_t t = 0, boff = 0;
    for (int p = 0; p < num_pages; ++p) {
        ix->pbase[p] = t;
        ix->boffs[p] = boff;
        ix->ptok[p] = page_tokens(pln, blen, boff, p);
        for (int64_t i = 0; i < ix->ptok[p]; ++i) { ix->pg[t] = p; ix->loc[t] = i; ++t; }
        boff += pln[3 * p + 2];
    }
}

static void page_index_free(page_index *ix)
{
    free(ix->pg); free(ix->loc); free(ix->pbase); free(ix->boffs); free(ix->ptok);
}

static double dot_fd(const float *a, const float *b, int d)
{
    double acc = 0.0;
    for (int c = 0; c < d; ++c) acc += (double)a[c] * (double)b[c];
    return acc;
}

/* Softmax statistics of query (page p, local qi), head h: lse and D = sum_j P_j dP_j. With dq
 * non-null, also dq[c] = scale * sum_j dS_j k_j[c]. sbuf/pbuf: scratch of the page's size. */
static void row_backward(const int32_t *pln, const int32_t *fork, const int32_t *blen, const page_index *ix, int p,
                         int64_t qi, int h, const float *q, const float *k, const float *v, const float *dout,
                         int32_t Hq, int32_t Hkv, int32_t d, double scale, int64_t *vis, double *sbuf,
                         double *dpbuf, double *lse_out, double *D_out, double *dq)
{
    const int32_t *pp = pln + 3 * p;
    const int32_t *fk = fork + ix->boffs[p], *bl = blen + ix->boffs[p];
    const int64_t S = ix->ptok[p], pb = ix->pbase[p];
    const int g = h / (Hq / Hkv);
    const float *qr = q + ((pb + qi) * Hq + h) * d;
    const float *gr = dout + ((pb + qi) * Hq + h) * d;
    int64_t nv = 0;
    double mx = -INFINITY;
    for (int64_t j = 0; j < S; ++j) {
        if (!visible_by_ancestors(pp, fk, bl, qi, j)) continue;
        vis[nv] = j;
        sbuf[nv] = scale * dot_fd(qr, k + ((pb + j) * Hkv + g) * d, d);
        if (sbuf[nv] > mx) mx = sbuf[nv];
        ++nv;
    }
    double sum = 0.0;
    for (int64_t c = 0; c < nv; ++c) sum += exp(sbuf[c] - mx);
    const double lse = nv ? mx + log(sum) : -INFINITY;
    double D = 0.0;
    for (int64_t c = 0; c < nv; ++c) {
        sbuf[c] = exp(sbuf[c] - lse);                                   /* P_j */
        dpbuf[c] = dot_fd(gr, v + ((pb + vis[c]) * Hkv + g) * d, d);    /* dP_j */
        D += sbuf[c] * dpbuf[c];
    }
    *lse_out = lse;
    *D_out = D;
    if (dq) {
        for (int c = 0; c < d; ++c) dq[c] = 0.0;
        for (int64_t c = 0; c < nv; ++c) {
            const double ds = sbuf[c] * (dpbuf[c] - D);
            const float *kr = k + ((pb + vis[c]) * Hkv + g) * d;
            for (int e = 0; e < d; ++e) dq[e] += ds * (double)kr[e];
        }
        for (int c = 0; c < d; ++c) dq[c] *= scale;
    }
}

void oracle_prefill_bwd(const int32_t *pln, int32_t num_pages, const int32_t *fork, const int32_t *blen,
                        const float *q, const float *k, const float *v, const float *dout, int32_t Hq, int32_t Hkv,
                        int32_t d, double scale, int64_t nq, const int64_t *q_sel, int64_t nk, const int64_t *k_sel,
                        double *dq, double *dk, double *dv)
{
    const int64_t T = oracle_total_tokens(pln, num_pages, blen);
    page_index ix;
    page_index_build(pln, num_pages, blen, T, &ix);
    int64_t smax = 1;
    for (int p = 0; p < num_pages; ++p) if (ix.ptok[p] > smax) smax = ix.ptok[p];

    /* dQ of the selected query rows */
#pragma omp parallel
    {
        int64_t *vis = (int64_t *)malloc(sizeof(int64_t) * (size_t)smax);
        double *sb = (double *)malloc(sizeof(double) * (size_t)smax);
        double *db = (double *)malloc(sizeof(double) * (size_t)smax);
#pragma omp for collapse(2) schedule(dynamic, 4)
        for (int64_t r = 0; r < nq; ++r) {
            for (int h = 0; h < Hq; ++h) {
                const int64_t t = q_sel[r];
                double lse, D;
                row_backward(pln, fork, blen, &ix, ix.pg[t], ix.loc[t], h, q, k, v, dout, Hq, Hkv, d, scale, vis, sb,
                             db, &lse, &D, dq + (r * Hq + h) * d);
            }
        }
        free(vis); free(sb); free(db);
    }

    /* dK, dV of the selected key rows: the softmax statistics of every query of a touched page */
    uint8_t *touched = (uint8_t *)calloc((size_t)(num_pages > 0 ? num_pages : 1), 1);
    for (int64_t r = 0; r < nk; ++r) touched[ix.pg[k_sel[r]]] = 1;
    double *lse_all = (double *)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1) * (size_t)Hq);
    double *D_all = (double *)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1) * (size_t)Hq);
    for (int p = 0; p < num_pages; ++p) {
        if (!touched[p]) continue;
        const int64_t S = ix.ptok[p];
#pragma omp parallel
        {
            int64_t *vis = (int64_t *)malloc(sizeof(int64_t) * (size_t)smax);
            double *sb = (double *)malloc(sizeof(double) * (size_t)smax);
            double *db = (double *)malloc(sizeof(double) * (size_t)smax);
#pragma omp for collapse(2) schedule(dynamic, 4)
            for (int64_t qi = 0; qi < S; ++qi) {
                for (int h = 0; h < Hq; ++h) {
                    const int64_t row = (ix.pbase[p] + qi) * Hq + h;
                    row_backward(pln, fork, blen, &ix, p, qi, h, q, k, v, dout, Hq, Hkv, d, scale, vis, sb, db,
                                 &lse_all[row], &D_all[row], NULL);
                }
            }
            free(vis); free(sb); free(db);
        }
    }
    const int group = Hq / Hkv;
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int64_t r = 0; r < nk; ++r) {
        for (int g = 0; g < Hkv; ++g) {
            const int64_t t = k_sel[r];
            const int p = ix.pg[t];
            const int64_t j = ix.loc[t], pb = ix.pbase[p], S = ix.ptok[p];
            const int32_t *pp = pln + 3 * p;
            const int32_t *fk = fork + ix.boffs[p], *bl = blen + ix.boffs[p];
            const float *kr = k + (t * Hkv + g) * d, *vr = v + (t * Hkv + g) * d;
            double *dkr = dk + (r * Hkv + g) * d, *dvr = dv + (r * Hkv + g) * d;
            for (int c = 0; c < d; ++c) { dkr[c] = 0.0; dvr[c] = 0.0; }
            for (int64_t qi = 0; qi < S; ++qi) {
                if (!visible_by_ancestors(pp, fk, bl, qi, j)) continue;
                for (int h = g * group; h < (g + 1) * group; ++h) {
                    const int64_t row = (pb + qi) * Hq + h;
                    const float *qr = q + row * d, *gr = dout + row * d;
                    const double pij = exp(scale * dot_fd(qr, kr, d) - lse_all[row]);
                    const double ds = pij * (dot_fd(gr, vr, d) - D_all[row]);
                    for (int c = 0; c < d; ++c) {
                        dkr[c] += ds * (double)qr[c];
                        dvr[c] += pij * (double)gr[c];
                    }
                }
            }
            for (int c = 0; c < d; ++c) dkr[c] *= scale;
        }
    }
    free(touched); free(lse_all); free(D_all);
    page_index_free(&ix);
}

/* ============================================================================================
 * FP8 (E4M3) KV cache. The paper serves a bf16 cache; this is the definition the FP8 cache
 * variant of the decode step is checked against: K and V stored as E4M3 codes with one fp32 scale
 * per (block, KV head), and attention over the dequantized values code_value * scale.
 *
 * E4M3 (the OCP 8-bit floating point format): sign bit, 4 exponent bits with bias 7, 3 mantissa
 * bits; exponent field 0 is subnormal (value m * 2^-9); no infinities; S.1111.111 is NaN, so the
 * largest finite magnitude is 1.75 * 2^8 = 448.
 * ========================================================================================== */

double oracle_e4m3_value(uint8_t code)
{
    const int s = code >> 7, e = (code >> 3) & 15, m = code & 7;
    if (e == 15 && m == 7) return NAN;
    const double v = e == 0 ? ldexp((double)m, -9) : ldexp((double)(8 + m), e - 10);
    return s ? -v : v;
}

/* Nearest E4M3 code to x, ties to the even code (the one whose mantissa's last bit is 0),
 * magnitudes of 448 and above saturated to 448, NaN to the NaN code 0x7F. The search runs over
 * every finite positive code, which is slow and plainly correct. */
uint8_t oracle_e4m3_encode_one(double x)
{
    if (isnan(x)) return 0x7F;
    const int s = signbit(x) ? 1 : 0;
    const double a = fabs(x);
    int best = 0;
    if (a >= 448.0) {
        best = 0x7E;
    } else {
        double best_err = INFINITY;
        for (int c = 0; c <= 0x7E; ++c) {
            const double err = fabs(oracle_e4m3_value((uint8_t)c) - a);
            if (err < best_err || (err == best_err && (c & 1) == 0)) {
                best_err = err;
                best = c;
            }
        }
    }
    return (uint8_t)(best | (s << 7));
}

void oracle_e4m3_encode(const float *x, int64_t n, uint8_t *codes)
{
    for (int64_t i = 0; i < n; ++i) codes[i] = oracle_e4m3_encode_one((double)x[i]);
}

void oracle_e4m3_decode(const uint8_t *codes, int64_t n, double *x)
{
    for (int64_t i = 0; i < n; ++i) x[i] = oracle_e4m3_value(codes[i]);
}

/* Quantizes a pool [num_blocks][hkv][bs][d] of fp32 K or V: per (block, head) the scale is
 * amax / 448 in fp32 and each element's code is the E4M3 code of x / scale, the division taken in
 * fp32, the precision a kernel that quantizes on write uses. An all-zero (block, head) gets scale 0
 * and codes 0: a zero scale marks a (block, head) that holds no nonzero value, the state the
 * row-by-row append below starts from, so a block quantized whole and then extended row by row
 * follows one rule. */
void oracle_quantize_kv_blocks(const float *x, int64_t num_blocks, int32_t hkv, int32_t bs, int32_t d, uint8_t *codes,
                               float *scales)
{
    const int64_t per = (int64_t)bs * d;
    for (int64_t u = 0; u < num_blocks * hkv; ++u) {
        const float *src = x + u * per;
        float amax = 0.0f;
        for (int64_t i = 0; i < per; ++i) amax = fmaxf(amax, fabsf(src[i]));
        const float scale = amax / 448.0f;
        scales[u] = scale;
        for (int64_t i = 0; i < per; ++i) {
            if (scale == 0.0f) { codes[u * per + i] = 0; continue; }
            const float y = src[i] / scale;
            codes[u * per + i] = oracle_e4m3_encode_one((double)y);
        }
    }
}

/* Appends rows to a quantized pool one at a time, in the order given, as a decoding loop writes
 * its cache (Algorithm 1 appends one input per live stream per step). Row i, for every KV head g,
 * goes to block b = slots[i] / bs, row r = slots[i] % bs:
 *   1. a = max_c |x_c| over the new row (fp32); s_old = the block's scale, taken as 0 when r = 0
 *      (a block's first row starts it afresh: a block handed out again keeps a former owner's
 *      scale and rows, which no one reads);
 *   2. s_new = max(s_old, a / 448), the division in fp32: the scale stays amax / 448 over the rows
 *      written so far;
 *   3. if s_new > s_old > 0, each earlier row r' < r is re-encoded against the new scale: the value
 *      its code stood for, code_value * s_old (fp32 product), divided by s_new (fp32), is encoded
 *      again (nearest even, saturating);
 *   4. the new row's codes are the codes of x_c / s_new (fp32 division), or 0 when s_new = 0;
 *   5. the block's scale becomes s_new.
 * Rows r' > r are left as they are. rows: [count][hkv][d] fp32; codes [num_blocks][hkv][bs][d];
 * scales [num_blocks][hkv]. */
void oracle_append_kv_quantized(uint8_t *codes, float *scales, int64_t num_blocks, int32_t hkv, int32_t bs, int32_t d,
                                const int32_t *slots, int32_t count, const float *rows)
{
    for (int32_t i = 0; i < count; ++i) {
        const int64_t b = slots[i] / bs;
        const int32_t r = slots[i] % bs;
        if (b < 0 || b >= num_blocks) continue;
        for (int32_t g = 0; g < hkv; ++g) {
            const float *x = rows + ((int64_t)i * hkv + g) * d;
            uint8_t *blk = codes + (b * hkv + g) * (int64_t)bs * d;
            float *sc = scales + b * hkv + g;
            float a = 0.0f;
            for (int32_t c = 0; c < d; ++c) a = fmaxf(a, fabsf(x[c]));
            const float s_old = r == 0 ? 0.0f : *sc;
            const float cand = a / 448.0f;
            const float s_new = cand > s_old ? cand : s_old;
            if (s_new > s_old && s_old > 0.0f) {
                for (int32_t rr = 0; rr < r; ++rr)
                    for (int32_t c = 0; c < d; ++c) {
                        uint8_t *cp = blk + (int64_t)rr * d + c;
                        const float y = (float)oracle_e4m3_value(*cp) * s_old;
                        const float z = y / s_new;
                        *cp = oracle_e4m3_encode_one((double)z);
                    }
            }
            for (int32_t c = 0; c < d; ++c) {
                uint8_t *cp = blk + (int64_t)r * d + c;
                if (s_new == 0.0f) { *cp = 0; continue; }
                const float z = x[c] / s_new;
                *cp = oracle_e4m3_encode_one((double)z);
            }
            *sc = s_new;
        }
    }
}

/* The dequantized pool: code_value * scale, exact in fp64. */
void oracle_dequantize_kv_blocks(const uint8_t *codes, const float *scales, int64_t num_blocks, int32_t hkv,
                                 int32_t bs, int32_t d, double *x)
{
    const int64_t per = (int64_t)bs * d;
    for (int64_t u = 0; u < num_blocks * hkv; ++u)
        for (int64_t i = 0; i < per; ++i) x[u * per + i] = oracle_e4m3_value(codes[u * per + i]) * (double)scales[u];
}
