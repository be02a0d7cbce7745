/*
 * CacheBack oracle: a plain, slow fp64 CPU restatement of the score -> select
 * -> compact path of receiver-conditioned KV filtering.
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only the tests, the smoke check and
 * the benchmark's CPU-baseline / reference leg may load this library.  It
 * shares no code, header, table or helper with the CUDA path.
 *
 * Notation (App. C.1, "General scoring rule"):
 *   l   scored layer, h query head, r query token (m of them), t sender position (T of them)
 *   a_{l,h,r,t}  attention from query token r in head h of layer l to position t
 *   s = (l, g)   KV-head group: the G = Hq/Hkv query heads h with h / G == g share KV head g
 *   b_{s,r,t}    mean of a over the query heads of group s
 *   Pool_w       max over the w positions centred on t, clipped at 0 and T-1
 *
 * Readings of points the paper leaves open (each is listed with its reason in
 * the design notes):
 *   - the softmax runs over the T sender positions only (the keys the sender holds);
 *   - the logit scale is a parameter (1/sqrt(d) by default);
 *   - query head h belongs to KV head h / G (consecutive grouping);
 *   - C = 1 wherever the denominator sum is 0.
 *
 * Every sum is in double, in a fixed order, so results do not depend on the
 * thread count.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#else
static int omp_get_max_threads(void) { return 1; }
#endif

#define CBO_OK 0
#define CBO_EINVAL 1
#define CBO_ESHAPE 2
#define CBO_EBUDGET 3
#define CBO_ENOMEM 4

typedef struct {
    int32_t n_layers;   /* |L| */
    int32_t n_q_heads;  /* Hq */
    int32_t n_kv_heads; /* Hkv */
    int32_t head_dim;   /* d */
    int32_t m;          /* query tokens */
    int64_t T;          /* sender positions */
    int64_t k_layer, k_head, k_pos; /* element strides of K and V, dim stride 1 */
    int64_t q_layer, q_tok, q_head; /* element strides of Q, dim stride 1 */
    int64_t s_layer, s_tok, s_head; /* element strides of the query's own keys Ks[l][u][g][:], if given */
} cbo_dims;

/* bf16 bit pattern -> double, exact. */
static double bf16_to_double(uint16_t bits) {
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static int check_dims(const cbo_dims *dm) {
    if (!dm) return CBO_EINVAL;
    if (dm->n_layers < 1 || dm->n_q_heads < 1 || dm->n_kv_heads < 1 || dm->head_dim < 1 ||
        dm->m < 1 || dm->T < 1)
        return CBO_ESHAPE;
    if (dm->n_q_heads % dm->n_kv_heads) return CBO_ESHAPE;
    return CBO_OK;
}

/*
 * Pool_w (App. C.1): y_t = max of x_u over u in [t - w/2, t + w/2], clipped to
 * [0, T).  Pooling runs over sender positions only.  w = 1 is the identity.
 */
void cbo_pool(const double *x, double *y, int64_t T, int32_t w) {
    int64_t half = w / 2;
    for (int64_t t = 0; t < T; ++t) {
        int64_t lo = t - half < 0 ? 0 : t - half;
        int64_t hi = t + half > T - 1 ? T - 1 : t + half;
        double mx = x[lo];
        for (int64_t u = lo + 1; u <= hi; ++u)
            if (x[u] > mx) mx = x[u];
        y[t] = mx;
    }
}

/* K slice of group (l, g) as doubles, transposed to [d][T] so the logit loop
 * below accumulates each z_t over the head dimension in index order. */
static double *load_keys_transposed(const cbo_dims *dm, const uint16_t *K, int l, int g) {
    int64_t T = dm->T;
    int d = dm->head_dim;
    double *kt = (double *)malloc(sizeof(double) * (size_t)d * (size_t)T);
    if (!kt) return NULL;
    const uint16_t *base = K + (int64_t)l * dm->k_layer + (int64_t)g * dm->k_head;
    for (int64_t t = 0; t < T; ++t)
        for (int k = 0; k < d; ++k) kt[(int64_t)k * T + t] = bf16_to_double(base[t * dm->k_pos + k]);
    return kt;
}

/* scale * <q, ks_{l,u,g}>: logit of a query token against query token u's own key. */
static double self_logit(const cbo_dims *dm, const uint16_t *q, const uint16_t *Ks, int l, int u, int g,
                         double scale) {
    const uint16_t *k = Ks + (int64_t)l * dm->s_layer + (int64_t)u * dm->s_tok + (int64_t)g * dm->s_head;
    double z = 0.0;
    for (int i = 0; i < dm->head_dim; ++i) z += bf16_to_double(q[i]) * bf16_to_double(k[i]);
    return z * scale;
}

/*
 * One attention row a_{l,h,r,.} (App. C.1, "Adapting SnapKV"): the sender
 * attends from query token r, head h, to its cached positions:
 *   z_t = scale * <q_{l,r,h}, k_{l,g(h),t}>,   a_t = exp(z_t - M) / sum_u exp(z_u - M),
 * with M = max_t z_t (the shift leaves a unchanged).  z is scratch of length T.
 * With the query tokens' own keys Ks (not NULL) the softmax also runs over the keys of query
 * tokens 0..r (the causal prefix of the query in a real forward pass); a still covers the
 * sender positions only, so it sums to less than one.
 */
static void attention_row(const cbo_dims *dm, const double *kt, const uint16_t *Q, const uint16_t *Ks, int l,
                          int h, int r, double scale, double *z, double *a) {
    int64_t T = dm->T;
    int d = dm->head_dim;
    const uint16_t *q = Q + (int64_t)l * dm->q_layer + (int64_t)r * dm->q_tok + (int64_t)h * dm->q_head;
    for (int64_t t = 0; t < T; ++t) z[t] = 0.0;
    for (int k = 0; k < d; ++k) {
        double qk = bf16_to_double(q[k]);
        const double *row = kt + (int64_t)k * T;
        for (int64_t t = 0; t < T; ++t) z[t] += qk * row[t];
    }
    double M = -INFINITY;
    for (int64_t t = 0; t < T; ++t) {
        z[t] *= scale;
        if (z[t] > M) M = z[t];
    }
    const int g = h / (dm->n_q_heads / dm->n_kv_heads);
    if (Ks)
        for (int u = 0; u <= r; ++u) {
            const double zs = self_logit(dm, q, Ks, l, u, g, scale);
            if (zs > M) M = zs;
        }
    double Z = 0.0;
    for (int64_t t = 0; t < T; ++t) {
        a[t] = exp(z[t] - M);
        Z += a[t];
    }
    if (Ks)
        for (int u = 0; u <= r; ++u) Z += exp(self_logit(dm, q, Ks, l, u, g, scale) - M);
    for (int64_t t = 0; t < T; ++t) a[t] /= Z;
}

/*
 * Attention weights of every scored layer: a[l][h][r][t] (nL*Hq*m*T doubles).
 * Exposed so tests can check the softmax and the head-to-KV-head mapping
 * against a library attention routine.
 */
int cbo_attention_self(const cbo_dims *dm, const uint16_t *K, const uint16_t *Q, const uint16_t *Ks, double scale,
                       double *a) {
    int st = check_dims(dm);
    if (st) return st;
    if (!K || !Q || !a) return CBO_EINVAL;
    int64_t T = dm->T;
    int G = dm->n_q_heads / dm->n_kv_heads;
    double *z = (double *)malloc(sizeof(double) * (size_t)T);
    if (!z) return CBO_ENOMEM;
    for (int l = 0; l < dm->n_layers; ++l)
        for (int h = 0; h < dm->n_q_heads; ++h) {
            double *kt = load_keys_transposed(dm, K, l, h / G);
            if (!kt) { free(z); return CBO_ENOMEM; }
            for (int r = 0; r < dm->m; ++r)
                attention_row(dm, kt, Q, Ks, l, h, r, scale,
                              z, a + (((int64_t)l * dm->n_q_heads + h) * dm->m + r) * T);
            free(kt);
        }
    free(z);
    return CBO_OK;
}

int cbo_attention(const cbo_dims *dm, const uint16_t *K, const uint16_t *Q, double scale, double *a) {
    return cbo_attention_self(dm, K, Q, NULL, scale, a);
}

/*
 * Score every sender position (App. C.1 and App. D.2); Ks (may be NULL) are the query tokens'
 * own keys, joining each query token's softmax causally (see attention_row):
 *
 *   Q_t   = Pool( sum_l 1/(m |H_l|) sum_r sum_{h in H_l} a_{l,h,r,t} )          (mean query attention)
 *   C_p,t = ( sum_s mean_r[Pool(b_{s,r,.})_t^p] / sum_s Pool(mean_r b_{s,r,.})_t^p )^(1/(p-1))
 *   S_t   = Q_t * C_p,t^alpha                                                     (CacheBack: p = alpha = 2)
 *
 * with C = 1 where the denominator is zero.  p = +infinity takes the limit (App. D.2, parameter
 * sensitivity: the largest pooled query-token attention against the largest pooled mean):
 *   C_inf,t = max_{s,r} Pool(b_{s,r,.})_t / max_s Pool(mean_r b_{s,r,.})_t
 * (the 1/m factor and the sums over s become 1 and maxima in the limit of the 1/(p-1) power);
 * then N and D hold those maxima.  Outputs (any may be NULL), each [T]:
 *   S, Qt, C, U (the layer sum inside Pool, before pooling), N and D (numerator
 *   and denominator sums of C).
 * The work is split over the groups s = (l, g); each group's contributions are
 * kept apart and added in the order s = 0, 1, ... at the end.
 */
int cbo_score_self(const cbo_dims *dm, const uint16_t *K, const uint16_t *Q, const uint16_t *Ks, double scale,
                   double p, double alpha, int32_t pool_w, int32_t n_threads, double *S, double *Qt, double *C,
                   double *U, double *N, double *D) {
    int st = check_dims(dm);
    if (st) return st;
    if (!K || !Q) return CBO_EINVAL;
    if (!(p > 1.0) || alpha < 0.0 || pool_w < 1 || (pool_w % 2) == 0) return CBO_EINVAL;
    const int p_inf = isinf(p);
    const int64_t T = dm->T;
    const int m = dm->m, Hq = dm->n_q_heads, Hkv = dm->n_kv_heads, G = Hq / Hkv;
    const int nS = dm->n_layers * Hkv;

    double *part = (double *)calloc((size_t)nS * 3 * (size_t)T, sizeof(double)); /* U_s, N_s, D_s */
    if (!part) return CBO_ENOMEM;
    int failed = 0;

#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads > 0 ? n_threads : omp_get_max_threads())
    for (int s = 0; s < nS; ++s) {
        const int l = s / Hkv, g = s % Hkv;
        double *Us = part + ((int64_t)s * 3 + 0) * T;
        double *Ns = part + ((int64_t)s * 3 + 1) * T;
        double *Ds = part + ((int64_t)s * 3 + 2) * T;
        double *kt = load_keys_transposed(dm, K, l, g);
        double *b = (double *)calloc((size_t)m * (size_t)T, sizeof(double));
        double *z = (double *)malloc(sizeof(double) * (size_t)T);
        double *a = (double *)malloc(sizeof(double) * (size_t)T);
        double *pooled = (double *)malloc(sizeof(double) * (size_t)T);
        double *bbar = (double *)calloc((size_t)T, sizeof(double));
        if (!kt || !b || !z || !a || !pooled || !bbar) {
#pragma omp atomic write
            failed = 1;
        } else {
            for (int r = 0; r < m; ++r) {
                double *br = b + (int64_t)r * T;
                for (int j = 0; j < G; ++j) {
                    const int h = g * G + j;
                    attention_row(dm, kt, Q, Ks, l, h, r, scale, z, a);
                    for (int64_t t = 0; t < T; ++t) {
                        br[t] += a[t] / G;                 /* b_{s,r,t}: mean over the group's heads */
                        Us[t] += a[t] / ((double)m * Hq);  /* this group's share of the layer term of Q_t */
                    }
                }
            }
            /* numerator: mean over r of Pool(b_{s,r,.})^p */
            for (int r = 0; r < m; ++r) {
                const double *br = b + (int64_t)r * T;
                cbo_pool(br, pooled, T, pool_w);
                if (p_inf)
                    for (int64_t t = 0; t < T; ++t) Ns[t] = pooled[t] > Ns[t] ? pooled[t] : Ns[t];
                else
                    for (int64_t t = 0; t < T; ++t) Ns[t] += pow(pooled[t], p) / m;
            }
            /* denominator: Pool(mean over r of b_{s,r,.})^p */
            for (int r = 0; r < m; ++r) {
                const double *br = b + (int64_t)r * T;
                for (int64_t t = 0; t < T; ++t) bbar[t] += br[t] / m;
            }
            cbo_pool(bbar, pooled, T, pool_w);
            for (int64_t t = 0; t < T; ++t) Ds[t] = p_inf ? pooled[t] : pow(pooled[t], p);
        }
        free(kt); free(b); free(z); free(a); free(pooled); free(bbar);
    }
    if (failed) { free(part); return CBO_ENOMEM; }

    double *Usum = (double *)calloc((size_t)T, sizeof(double));
    double *Nsum = (double *)calloc((size_t)T, sizeof(double));
    double *Dsum = (double *)calloc((size_t)T, sizeof(double));
    double *Qv = (double *)malloc(sizeof(double) * (size_t)T);
    if (!Usum || !Nsum || !Dsum || !Qv) {
        free(part); free(Usum); free(Nsum); free(Dsum); free(Qv);
        return CBO_ENOMEM;
    }
    for (int s = 0; s < nS; ++s)
        for (int64_t t = 0; t < T; ++t) {
            const double n_s = part[((int64_t)s * 3 + 1) * T + t], d_s = part[((int64_t)s * 3 + 2) * T + t];
            Usum[t] += part[((int64_t)s * 3 + 0) * T + t];
            if (p_inf) {   /* maxima over the groups; every partial is >= 0 and the sums start at 0 */
                Nsum[t] = n_s > Nsum[t] ? n_s : Nsum[t];
                Dsum[t] = d_s > Dsum[t] ? d_s : Dsum[t];
            } else {
                Nsum[t] += n_s;
                Dsum[t] += d_s;
            }
        }
    cbo_pool(Usum, Qv, T, pool_w);
    for (int64_t t = 0; t < T; ++t) {
        double c = Dsum[t] > 0.0 ? (p_inf ? Nsum[t] / Dsum[t] : pow(Nsum[t] / Dsum[t], 1.0 / (p - 1.0))) : 1.0;
        if (S) S[t] = Qv[t] * pow(c, alpha);
        if (Qt) Qt[t] = Qv[t];
        if (C) C[t] = c;
        if (U) U[t] = Usum[t];
        if (N) N[t] = Nsum[t];
        if (D) D[t] = Dsum[t];
    }
    free(part); free(Usum); free(Nsum); free(Dsum); free(Qv);
    return CBO_OK;
}

int cbo_score(const cbo_dims *dm, const uint16_t *K, const uint16_t *Q, double scale, double p, double alpha,
              int32_t pool_w, int32_t n_threads, double *S, double *Qt, double *C, double *U, double *N, double *D) {
    return cbo_score_self(dm, K, Q, NULL, scale, p, alpha, pool_w, n_threads, S, Qt, C, U, N, D);
}

/* ---------------------------------------------------------------------------
 * Selection (App. C.2, "Budgets and position selection")
 * ------------------------------------------------------------------------- */

typedef struct {
    double mean;
    int64_t j;
} span_rank;

/* Higher mean first; equal means favour the earlier span. */
static int span_cmp(const void *x, const void *y) {
    const span_rank *a = (const span_rank *)x, *b = (const span_rank *)y;
    if (a->mean > b->mean) return -1;
    if (a->mean < b->mean) return 1;
    return a->j < b->j ? -1 : (a->j > b->j ? 1 : 0);
}

typedef struct {
    int64_t dist, t;
} near_pos;

static int near_cmp(const void *x, const void *y) {
    const near_pos *a = (const near_pos *)x, *b = (const near_pos *)y;
    if (a->dist != b->dist) return a->dist < b->dist ? -1 : 1;
    return a->t < b->t ? -1 : (a->t > b->t ? 1 : 0);
}

/*
 * Span selection of B positions out of T (App. C.2):
 *   1. keep the first n_sink positions and the last n_latent (latent) positions;
 *      they count toward B;
 *   2. set the first position's score to the maximum position score;
 *   3. spans [w j, min(T, w j + w)) are ranked by their mean score (a shorter
 *      last span is averaged over its own length), equal means favouring the
 *      earlier span;
 *   4. walking the ranking, add each span's not-yet-selected positions while
 *      they fit; when the next span does not fit, add the positions of that
 *      span nearest to its highest-scoring unselected position (ties: lower
 *      index), up to the budget;
 *   5. return the selected positions in source order.
 * `sf` (fp32 scores) or `sd` (fp64 scores) supplies S; with fp32 scores every
 * span mean is formed in fp32 (positions added in index order, then divided by
 * the span length) so ranking decisions are taken in the scores' precision.
 * Returns the count written to idx (== B) or a negative error.
 */
static int64_t select_impl(int64_t T, const double *sd, const float *sf, int64_t B, int32_t n_sink,
                           int32_t n_latent, int32_t span_w, int32_t *idx) {
    if (T < 1 || span_w < 1 || n_sink < 0 || n_latent < 0 || !idx || (!sd && !sf)) return -CBO_EINVAL;
    unsigned char *sel = (unsigned char *)calloc((size_t)T, 1);
    double *Sp = (double *)malloc(sizeof(double) * (size_t)T);
    int64_t nspan = (T + span_w - 1) / span_w;
    span_rank *rank = (span_rank *)malloc(sizeof(span_rank) * (size_t)nspan);
    near_pos *near = (near_pos *)malloc(sizeof(near_pos) * (size_t)span_w);
    if (!sel || !Sp || !rank || !near) {
        free(sel); free(Sp); free(rank); free(near);
        return -CBO_ENOMEM;
    }
    int64_t count = 0;
    for (int64_t t = 0; t < T; ++t)
        if (t < n_sink || t >= T - n_latent) { sel[t] = 1; ++count; }
    if (B < count || B > T) {
        free(sel); free(Sp); free(rank); free(near);
        return -CBO_EBUDGET;
    }
    /* S' : the first position takes the maximum score */
    for (int64_t t = 0; t < T; ++t) Sp[t] = sd ? sd[t] : (double)sf[t];
    if (n_sink > 0) {
        double mx = Sp[0];
        for (int64_t t = 1; t < T; ++t)
            if (Sp[t] > mx) mx = Sp[t];
        Sp[0] = mx;
    }
    for (int64_t j = 0; j < nspan; ++j) {
        int64_t lo = j * span_w, hi = lo + span_w < T ? lo + span_w : T;
        if (sf) {
            float acc = 0.0f;
            for (int64_t t = lo; t < hi; ++t) acc += (float)Sp[t];
            rank[j].mean = (double)(acc / (float)(hi - lo));
        } else {
            double acc = 0.0;
            for (int64_t t = lo; t < hi; ++t) acc += Sp[t];
            rank[j].mean = acc / (double)(hi - lo);
        }
        rank[j].j = j;
    }
    qsort(rank, (size_t)nspan, sizeof(span_rank), span_cmp);
    for (int64_t k = 0; k < nspan && count < B; ++k) {
        int64_t lo = rank[k].j * span_w, hi = lo + span_w < T ? lo + span_w : T;
        int64_t nu = 0;
        for (int64_t t = lo; t < hi; ++t) nu += !sel[t];
        if (nu == 0) continue;
        if (count + nu <= B) {
            for (int64_t t = lo; t < hi; ++t)
                if (!sel[t]) { sel[t] = 1; ++count; }
        } else {
            int64_t c = -1;
            for (int64_t t = lo; t < hi; ++t)
                if (!sel[t] && (c < 0 || Sp[t] > Sp[c])) c = t;
            int64_t n = 0;
            for (int64_t t = lo; t < hi; ++t)
                if (!sel[t]) { near[n].dist = t > c ? t - c : c - t; near[n].t = t; ++n; }
            qsort(near, (size_t)n, sizeof(near_pos), near_cmp);
            for (int64_t i = 0; count < B; ++i) { sel[near[i].t] = 1; ++count; }
        }
    }
    int64_t n = 0;
    for (int64_t t = 0; t < T; ++t)
        if (sel[t]) idx[n++] = (int32_t)t;
    free(sel); free(Sp); free(rank); free(near);
    return n;
}

int64_t cbo_select_f64(int64_t T, const double *S, int64_t B, int32_t n_sink, int32_t n_latent,
                       int32_t span_w, int32_t *idx) {
    return select_impl(T, S, NULL, B, n_sink, n_latent, span_w, idx);
}

int64_t cbo_select_f32(int64_t T, const float *S, int64_t B, int32_t n_sink, int32_t n_latent,
                       int32_t span_w, int32_t *idx) {
    return select_impl(T, NULL, S, B, n_sink, n_latent, span_w, idx);
}

/*
 * Gather-compact (the message of selected positions): for every layer l and KV
 * head g, row j of the output at sequence offset `off` is the source row idx[j]:
 *   out[l][g][off + j][:] = src[l][g][idx[j]][:]      for K and for V,
 * copied as raw bf16 bits.  Output strides o_layer / o_head are in elements;
 * positions are contiguous rows of d elements.
 */
int cbo_compact(const cbo_dims *dm, const uint16_t *K, const uint16_t *V, const int32_t *idx, int64_t B,
                uint16_t *k_out, uint16_t *v_out, int64_t off, int64_t o_layer, int64_t o_head) {
    int st = check_dims(dm);
    if (st) return st;
    if (!K || !V || !idx || !k_out || !v_out || B < 0) return CBO_EINVAL;
    const int d = dm->head_dim;
    for (int64_t j = 0; j < B; ++j)
        if (idx[j] < 0 || idx[j] >= dm->T) return CBO_EINVAL;
    for (int l = 0; l < dm->n_layers; ++l)
        for (int g = 0; g < dm->n_kv_heads; ++g)
            for (int64_t j = 0; j < B; ++j) {
                int64_t src = (int64_t)l * dm->k_layer + (int64_t)g * dm->k_head + (int64_t)idx[j] * dm->k_pos;
                int64_t dst = (int64_t)l * o_layer + (int64_t)g * o_head + (off + j) * d;
                memcpy(k_out + dst, K + src, sizeof(uint16_t) * (size_t)d);
                memcpy(v_out + dst, V + src, sizeof(uint16_t) * (size_t)d);
            }
    return CBO_OK;
}

/*
 * Message rows (Sec. 3.1 "State Representation", App. C.3 "Message encoding"): the
 * continuous-row encoding sends the sender's per-position row (hidden state) of every selected
 * position, the token-ID encoding the token ID (a 4-byte row) of every selected source position:
 *   out row (off + j) = src row idx[j],   j < count,
 * rows of row_bytes raw bytes, row t of src at src + t * src_stride, row r of out at
 * out + r * out_stride.
 */
int cbo_gather(const uint8_t *src, int64_t T, int64_t src_stride, int64_t row_bytes, const int32_t *idx,
               int64_t count, uint8_t *out, int64_t off, int64_t out_stride) {
    if (!src || !out || (count > 0 && !idx) || T < 1 || count < 0 || row_bytes < 1) return CBO_EINVAL;
    for (int64_t j = 0; j < count; ++j)
        if (idx[j] < 0 || idx[j] >= T) return CBO_EINVAL;
    for (int64_t j = 0; j < count; ++j)
        memcpy(out + (off + j) * out_stride, src + (int64_t)idx[j] * src_stride, (size_t)row_bytes);
    return CBO_OK;
}

/*
 * Paged (block-table) cache layout (App. F: the agents are served by vLLM, whose KV cache is
 * kept in fixed-size pages named by a per-sequence block table).  Position t of the sender is
 * row (t mod P) of page pages[floor(t / P)], the same page in every layer and KV head:
 *   out[l][g][t][k] = pool[l * s_layer + pages[t / P] * s_page + (t mod P) * s_pos + g * s_head + k]
 * for t < T.  The result is the contiguous [nL][Hkv][T][d] cache the other routines read.
 * Returns CBO_EINVAL (writing nothing) when a page entry lies outside [0, n_pages).
 */
int cbo_unpage(const uint16_t *pool, int32_t nL, int32_t Hkv, int32_t d, int64_t T, const int32_t *pages,
               int64_t P, int64_t n_pages, int64_t s_layer, int64_t s_page, int64_t s_pos, int64_t s_head,
               uint16_t *out) {
    if (!pool || !out || (T > 0 && !pages) || nL < 1 || Hkv < 1 || d < 1 || T < 0 || P < 1) return CBO_EINVAL;
    const int64_t n_used = (T + P - 1) / P;
    for (int64_t b = 0; b < n_used; ++b)
        if (pages[b] < 0 || pages[b] >= n_pages) return CBO_EINVAL;
    for (int32_t l = 0; l < nL; ++l)
        for (int32_t g = 0; g < Hkv; ++g)
            for (int64_t t = 0; t < T; ++t) {
                const int64_t page = pages[t / P], row = t % P;
                const uint16_t *src = pool + l * s_layer + page * s_page + row * s_pos + g * s_head;
                uint16_t *dst = out + (((int64_t)l * Hkv + g) * T + t) * d;
                for (int32_t k = 0; k < d; ++k) dst[k] = src[k];
            }
    return CBO_OK;
}

/* double -> bf16 bits, rounded once to nearest (ties to even); finite normal inputs. */
static uint16_t double_to_bf16(double x) {
    if (x == 0.0) return signbit(x) ? 0x8000u : 0u;
    int e;
    const double m = frexp(x, &e);                 /* |m| in [0.5, 1) */
    const double r = nearbyint(ldexp(m, 8));       /* 8 significant bits, ties to even */
    const float f = (float)ldexp(r, e - 8);         /* exact: a bf16 value */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(u >> 16);
}

/*
 * Compaction with the positional re-index direct K/V transfer needs (App. C.3: a receiver that
 * takes the sender's K rows as they are must move them from sender position t to its own
 * position p).  Rotary embeddings rotate each pair of K's dimensions by angle pos * theta_k with
 * theta_k = base^(-2k/d), k < d/2, so a row rotated for t becomes the row for p by one more
 * rotation by (p - t) * theta_k:
 *   (x_a, x_b) -> (x_a cos phi - x_b sin phi, x_b cos phi + x_a sin phi),  phi = (p - t) theta_k,
 * pairs (a, b) = (k, k + d/2) for style 0 (halves) or (2k, 2k + 1) for style 1 (interleaved).
 * Row j of the output (at out offset off) sits at receiver position p = pos0 + off + j.
 * K is rotated in double and rounded once to bf16; V is copied as in cbo_compact.
 */
int cbo_compact_rope(const cbo_dims *dm, const uint16_t *K, const uint16_t *V, const int32_t *idx, int64_t B,
                     uint16_t *k_out, uint16_t *v_out, int64_t off, int64_t o_layer, int64_t o_head, double base,
                     int32_t style, int64_t pos0) {
    int st = check_dims(dm);
    if (st) return st;
    if (!K || !V || !idx || !k_out || !v_out || B < 0 || !(base > 0.0) || (style != 0 && style != 1)) return CBO_EINVAL;
    const int d = dm->head_dim, half = d / 2;
    if (d % 2) return CBO_ESHAPE;
    for (int64_t j = 0; j < B; ++j)
        if (idx[j] < 0 || idx[j] >= dm->T) return CBO_EINVAL;
    for (int l = 0; l < dm->n_layers; ++l)
        for (int g = 0; g < dm->n_kv_heads; ++g)
            for (int64_t j = 0; j < B; ++j) {
                const int64_t src = (int64_t)l * dm->k_layer + (int64_t)g * dm->k_head + (int64_t)idx[j] * dm->k_pos;
                const int64_t dst = (off + j) * d + (int64_t)g * o_head + (int64_t)l * o_layer;
                const double delta = (double)(pos0 + off + j - idx[j]);
                for (int k = 0; k < half; ++k) {
                    const int a = style == 0 ? k : 2 * k, b = style == 0 ? k + half : 2 * k + 1;
                    const double phi = delta * pow(base, -2.0 * k / d);
                    const double xa = bf16_to_double(K[src + a]), xb = bf16_to_double(K[src + b]);
                    k_out[dst + a] = double_to_bf16(xa * cos(phi) - xb * sin(phi));
                    k_out[dst + b] = double_to_bf16(xb * cos(phi) + xa * sin(phi));
                }
                memcpy(&v_out[dst], &V[src], sizeof(uint16_t) * (size_t)d);
            }
    return CBO_OK;
}

int cbo_max_threads(void) { return omp_get_max_threads(); }
