/*
 * mla_oracle.c -- plain, slow, fp64 CPU oracle for the absorbed multi-head
 * latent attention (MLA) decode step of a converted MLA draft model.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, __graft_entry__.smoke() and the
 * CPU-baseline / reference arm of bench.py load this file.  The CUDA library
 * never links, includes or calls it, and the two share no code, header,
 * table or constant.
 *
 * Conventions
 *   - bf16 inputs are read as their exact values (a bf16 is the top half of
 *     an IEEE binary32), all arithmetic is fp64, nothing is rounded in
 *     between.  The only roundings are the cache writes of
 *     orc_cache_append() and orc_project_append(), which must store bf16
 *     into the cache like the GPU does; each rounds the exact fp64 value
 *     (rotation, projection) once, to nearest-even.
 *   - The attention is computed in its plain, NON-absorbed form: every cached
 *     latent c_j is up-projected to an explicit key k_j^nope = W_UK[g] c_j and
 *     value v_j = W_UV[g] c_j (Sec. 3.2, Eq. 5), and the scaled causal softmax
 *     attention of Sec. 3.1 (Eqs. 2-4) is evaluated with the score routing of
 *     Sec. 3.3 (a non-positional part plus a rotated positional part, both
 *     under one scale).  The latent-weighted average o_lat = sum_j a_j c_j is
 *     reported as well, because the absorbed GPU path exposes it.
 *
 * Readings of points the paper leaves open (each is stated once more at its
 * function):
 *   - RoPE (Sec. 3.1, R_t): frequency theta_k = base^(-2k/d_rope); style 0
 *     pairs element k with k + d_rope/2 ("rotate half"), style 1 pairs 2k with
 *     2k+1.  The rotation by angle t*theta_k maps (a, b) to
 *     (a cos - b sin, b cos + a sin).
 *   - Positions: the n_new appended entries of sequence b go to
 *     start_pos[b] + k; with kv_len[b] entries in the cache (after the append)
 *     query i of a q_len chunk sits at position kv_len[b] - q_len + i and sees
 *     keys 0 .. kv_len[b] - q_len + i (causal inside the chunk).
 *   - The positional cache k_rope stores keys already rotated to their own
 *     position, so a score is dot(R_p q_pe, k_rope_j) = q_pe^T R_pj k_pe_j.
 *   - Head h uses KV group g(h) = h / (H / G).
 *   - Output projection: out = W_O * concat_h o_h, concat index h*d_v + e.
 *
 * Pins (tests that tie this file to the paper and to mathematics, not to
 * itself) live in tests/test_oracle_pins.py; every function below has at
 * least one.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int32_t num_heads;     /* H  : query heads                        */
    int32_t num_kv_groups; /* G  : KV groups, H % G == 0              */
    int32_t d_nope;        /* non-positional query/key width          */
    int32_t d_rope;        /* decoupled positional key width (even)   */
    int32_t d_v;           /* value width per head                    */
    int32_t rank;          /* r  : latent rank                        */
    int32_t hidden;        /* D  : model width, 0 = no W_O            */
    double sm_scale;       /* softmax scale (1/sqrt(d_k))             */
    int32_t rope_style;    /* 0 rotate-half, 1 interleaved            */
    double rope_base;      /* RoPE base                               */
} orc_dims;

typedef struct {
    uint16_t *c_kv;        /* bf16 latent cache                        */
    uint16_t *k_rope;      /* bf16 rotated positional-key cache        */
    int64_t c_tok_stride;  /* elements between consecutive tokens      */
    int64_t r_tok_stride;
    int64_t c_blk_stride;  /* elements between blocks (seq or page)    */
    int64_t r_blk_stride;
    const int32_t *block_table; /* [batch, bt_stride] or NULL          */
    int32_t bt_stride;
    int32_t page_size;
    int32_t num_pages;
    int32_t capacity;      /* tokens a sequence may hold               */
} orc_cache;

enum { ORC_OK = 0, ORC_BAD_ARG = 1, ORC_BAD_POSITION = 2, ORC_BAD_PAGE = 3, ORC_NO_MEMORY = 4 };

int orc_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Exact value of a bf16 bit pattern. */
double orc_bf16_value(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round an fp64 value once to bf16, to nearest with ties to even.  bf16 keeps
 * 8 significant bits; below 2^-126 the spacing is fixed at 2^-133. */
uint16_t orc_bf16_round(double x)
{
    if (isnan(x)) return 0x7fc0;
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    if (isinf(x)) return (uint16_t)(sign | 0x7f80);
    double ax = fabs(x);
    if (ax == 0.0) return sign;
    int e;
    (void)frexp(ax, &e);               /* ax in [2^(e-1), 2^e) */
    int ulp_exp = e - 8;
    if (ulp_exp < -133) ulp_exp = -133;
    double r = nearbyint(ldexp(ax, -ulp_exp)); /* default mode: ties to even */
    double v = ldexp(r, ulp_exp);
    float f = (float)v;                /* exact, or +inf past the bf16 range */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7fffffffu) > 0x7f7f0000u) u = 0x7f800000u; /* past bf16 max */
    return (uint16_t)(sign | (u >> 16));
}

/* RoPE rotation R_pos of Sec. 3.1 applied to x (length d_rope), written to y
 * (y may alias x).  theta_k = base^(-2k/d_rope). */
void orc_rope(const double *x, double *y, int d_rope, int64_t pos, double base, int style)
{
    int half = d_rope / 2;
    for (int k = 0; k < half; ++k) {
        double theta = pow(base, -2.0 * (double)k / (double)d_rope);
        double ang = (double)pos * theta;
        double cs = cos(ang), sn = sin(ang);
        int i0 = style == 0 ? k : 2 * k;
        int i1 = style == 0 ? k + half : 2 * k + 1;
        double a = x[i0], b = x[i1];
        y[i0] = a * cs - b * sn;
        y[i1] = b * cs + a * sn;
    }
}

/* Element offsets of token t of sequence b in the two caches.  Contiguous
 * layout: block b.  Paged layout: page block_table[b][t / page_size], slot
 * t % page_size. */
static int tok_offsets(const orc_cache *c, int b, int64_t t, int64_t *co, int64_t *ro)
{
    if (t < 0 || t >= c->capacity) return ORC_BAD_POSITION;
    int64_t blk, slot;
    if (c->block_table) {
        int32_t page = c->block_table[(int64_t)b * c->bt_stride + t / c->page_size];
        if (page < 0 || page >= c->num_pages) return ORC_BAD_PAGE;
        blk = page;
        slot = t % c->page_size;
    } else {
        blk = b;
        slot = t;
    }
    *co = blk * c->c_blk_stride + slot * c->c_tok_stride;
    *ro = blk * c->r_blk_stride + slot * c->r_tok_stride;
    return ORC_OK;
}

static int check_dims(const orc_dims *d)
{
    if (d->num_heads <= 0 || d->num_kv_groups <= 0) return ORC_BAD_ARG;
    if (d->num_heads % d->num_kv_groups) return ORC_BAD_ARG;
    if (d->d_nope < 0 || d->d_rope < 0 || (d->d_rope & 1)) return ORC_BAD_ARG;
    if (d->d_v <= 0 || d->rank <= 0 || d->hidden < 0) return ORC_BAD_ARG;
    return ORC_OK;
}

/* Cache append (Sec. 3.2 latent cache c_j = W^DKV h_j with its positional key
 * k^PE_j; Sec. 3.1 rotation R_j).  Entry k of sequence b goes to position
 * start_pos[b] + k: the latent row is copied bit for bit, the positional key
 * is rotated to that position in fp64 and rounded once to bf16.
 *   c_new  [batch, n_new, rank]   bf16
 *   kr_new [batch, n_new, d_rope] bf16 (not yet rotated) */
int orc_cache_append(const orc_dims *d, const orc_cache *c, int batch, int n_new,
                     const uint16_t *c_new, const uint16_t *kr_new, const int32_t *start_pos)
{
    if (check_dims(d) || batch < 0 || n_new < 0) return ORC_BAD_ARG;
    const int r = d->rank, dr = d->d_rope;
    double *tmp = (double *)malloc(sizeof(double) * (size_t)(dr > 0 ? dr : 1));
    if (!tmp) return ORC_NO_MEMORY;
    int err = ORC_OK;
    for (int b = 0; b < batch && !err; ++b) {
        for (int k = 0; k < n_new && !err; ++k) {
            int64_t pos = (int64_t)start_pos[b] + k, co, ro;
            err = tok_offsets(c, b, pos, &co, &ro);
            if (err) break;
            const uint16_t *src_c = c_new + ((int64_t)b * n_new + k) * r;
            for (int e = 0; e < r; ++e) c->c_kv[co + e] = src_c[e];
            const uint16_t *src_r = kr_new + ((int64_t)b * n_new + k) * dr;
            for (int e = 0; e < dr; ++e) tmp[e] = orc_bf16_value(src_r[e]);
            orc_rope(tmp, tmp, dr, pos, d->rope_base, d->rope_style);
            for (int e = 0; e < dr; ++e) c->k_rope[ro + e] = orc_bf16_round(tmp[e]);
        }
    }
    free(tmp);
    return err;
}

/* Query absorption (Sec. 1: attention "through absorbed projections"; the
 * algebra is Eq. 5 read right to left): since the non-positional score is
 * q_nope . (W_UK[g] c_j) = (W_UK[g]^T q_nope) . c_j, the latent query is
 * q_lat = W_UK[g]^T q_nope (length rank).  The positional query is rotated to
 * the query's own position kv_len - q_len + i.
 *   q_nope [batch, q_len, H, d_nope], q_pe [batch, q_len, H, d_rope]
 *   w_uk   [G, d_nope, rank]
 *   q_lat  [batch, q_len, H, rank] (out), q_pe_rot [batch, q_len, H, d_rope] */
int orc_absorb_q(const orc_dims *d, int batch, int q_len, const uint16_t *q_nope,
                 const uint16_t *q_pe, const int32_t *kv_len, const uint16_t *w_uk,
                 double *q_lat, double *q_pe_rot)
{
    if (check_dims(d) || batch < 0 || q_len <= 0) return ORC_BAD_ARG;
    const int H = d->num_heads, hpg = d->num_heads / d->num_kv_groups;
    const int dn = d->d_nope, dr = d->d_rope, r = d->rank;
    for (int b = 0; b < batch; ++b)
        if (kv_len[b] < q_len) return ORC_BAD_POSITION;
    int64_t rows = (int64_t)batch * q_len * H;
#pragma omp parallel for schedule(static)
    for (int64_t row = 0; row < rows; ++row) {
        int h = (int)(row % H);
        int i = (int)((row / H) % q_len);
        int b = (int)(row / ((int64_t)H * q_len));
        int g = h / hpg;
        const uint16_t *qn = q_nope + row * dn;
        double *ql = q_lat + row * r;
        for (int rho = 0; rho < r; ++rho) {
            double acc = 0.0;
            for (int dd = 0; dd < dn; ++dd)
                acc += orc_bf16_value(qn[dd]) * orc_bf16_value(w_uk[((int64_t)g * dn + dd) * r + rho]);
            ql[rho] = acc;
        }
        double *qr = q_pe_rot + row * dr;
        for (int e = 0; e < dr; ++e) qr[e] = orc_bf16_value(q_pe[row * dr + e]);
        orc_rope(qr, qr, dr, (int64_t)kv_len[b] - q_len + i, d->rope_base, d->rope_style);
    }
    return ORC_OK;
}

/* One decode step of MLA attention, in the plain non-absorbed form.
 *
 * For every requested sequence b, group g, head h with g(h) = g, and query i
 * at position p = kv_len[b] - q_len + i (Sec. 3.1 Eqs. 2-4 with the Sec. 3.2
 * up-projection of Eq. 5 and the Sec. 3.3 score routing):
 *     k_j = W_UK[g] c_j,  v_j = W_UV[g] c_j                  (j = 0 .. p)
 *     s_j = sm_scale * ( q_nope . k_j + (R_p q_pe) . k_rope_j )
 *     a_j = exp(s_j) / sum_{u <= p} exp(s_u)
 *     o   = sum_j a_j v_j,  o_lat = sum_j a_j c_j,  lse = ln sum_{u <= p} exp(s_u)
 * and, when w_o is given and hidden > 0 (Sec. 4.1, the block output "after its
 * fixed output projection"):  out = W_O concat_h o_h.
 *
 *   seqs   : indices of the sequences to compute (NULL = all); outputs of the
 *            other sequences are left untouched
 *   o_lat  [batch, q_len, H, rank], lse [batch, q_len, H], o [batch, q_len, H, d_v],
 *   out    [batch, q_len, hidden] (may be NULL); any output pointer may be NULL. */
int orc_mla_decode(const orc_dims *d, const orc_cache *c, int batch, int q_len,
                   const int32_t *kv_len, const uint16_t *q_nope, const uint16_t *q_pe,
                   const uint16_t *w_uk, const uint16_t *w_uv, const uint16_t *w_o,
                   const int32_t *seqs, int n_seqs,
                   double *o_lat, double *lse, double *o, double *out)
{
    if (check_dims(d) || batch < 0 || q_len <= 0) return ORC_BAD_ARG;
    if (!seqs) n_seqs = batch;
    const int H = d->num_heads, G = d->num_kv_groups, hpg = H / G;
    const int dn = d->d_nope, dr = d->d_rope, dv = d->d_v, r = d->rank;
    for (int s = 0; s < n_seqs; ++s) {
        int b = seqs ? seqs[s] : s;
        if (b < 0 || b >= batch) return ORC_BAD_ARG;
        if (kv_len[b] < q_len || kv_len[b] > c->capacity) return ORC_BAD_POSITION;
        for (int64_t t = 0; t < kv_len[b]; ++t) {  /* every key must be addressable */
            int64_t co, ro;
            int e = tok_offsets(c, b, t, &co, &ro);
            if (e) return e;
        }
    }
    int err = ORC_OK;
    int64_t tasks = (int64_t)n_seqs * G;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t task = 0; task < tasks; ++task) {
        int b = seqs ? seqs[task / G] : (int)(task / G);
        int g = (int)(task % G);
        int64_t kv = kv_len[b];
        double *K = (double *)malloc(sizeof(double) * (size_t)(kv * (dn > 0 ? dn : 1)));
        double *V = (double *)malloc(sizeof(double) * (size_t)(kv * dv));
        double *KR = (double *)malloc(sizeof(double) * (size_t)(kv * (dr > 0 ? dr : 1)));
        double *cj = (double *)malloc(sizeof(double) * (size_t)r);
        double *s = (double *)malloc(sizeof(double) * (size_t)kv);
        double *qr = (double *)malloc(sizeof(double) * (size_t)(dr > 0 ? dr : 1));
        if (!K || !V || !KR || !cj || !s || !qr) {
#pragma omp atomic write
            err = ORC_NO_MEMORY;
        } else {
            /* explicit keys and values of group g (Eq. 5) */
            for (int64_t j = 0; j < kv; ++j) {
                int64_t co = 0, ro = 0;
                tok_offsets(c, b, j, &co, &ro);
                for (int rho = 0; rho < r; ++rho) cj[rho] = orc_bf16_value(c->c_kv[co + rho]);
                for (int dd = 0; dd < dn; ++dd) {
                    const uint16_t *w = w_uk + ((int64_t)g * dn + dd) * r;
                    double acc = 0.0;
                    for (int rho = 0; rho < r; ++rho) acc += orc_bf16_value(w[rho]) * cj[rho];
                    K[j * dn + dd] = acc;
                }
                for (int e = 0; e < dv; ++e) {
                    const uint16_t *w = w_uv + ((int64_t)g * dv + e) * r;
                    double acc = 0.0;
                    for (int rho = 0; rho < r; ++rho) acc += orc_bf16_value(w[rho]) * cj[rho];
                    V[j * dv + e] = acc;
                }
                for (int e = 0; e < dr; ++e) KR[j * dr + e] = orc_bf16_value(c->k_rope[ro + e]);
            }
            for (int h = g * hpg; h < (g + 1) * hpg; ++h) {
                for (int i = 0; i < q_len; ++i) {
                    int64_t row = ((int64_t)b * q_len + i) * H + h;
                    int64_t p = kv - q_len + i; /* query position; keys 0..p visible */
                    const uint16_t *qn = q_nope + row * dn;
                    for (int e = 0; e < dr; ++e) qr[e] = orc_bf16_value(q_pe[row * dr + e]);
                    orc_rope(qr, qr, dr, p, d->rope_base, d->rope_style);
                    double m = -INFINITY;
                    for (int64_t j = 0; j <= p; ++j) {
                        double acc = 0.0;
                        for (int dd = 0; dd < dn; ++dd) acc += orc_bf16_value(qn[dd]) * K[j * dn + dd];
                        double accr = 0.0;
                        for (int e = 0; e < dr; ++e) accr += qr[e] * KR[j * dr + e];
                        s[j] = d->sm_scale * (acc + accr);
                        if (s[j] > m) m = s[j];
                    }
                    double z = 0.0;
                    for (int64_t j = 0; j <= p; ++j) z += exp(s[j] - m);
                    if (lse) lse[row] = m + log(z);
                    for (int64_t j = 0; j <= p; ++j) s[j] = exp(s[j] - m) / z; /* now a_j */
                    if (o) {
                        for (int e = 0; e < dv; ++e) {
                            double acc = 0.0;
                            for (int64_t j = 0; j <= p; ++j) acc += s[j] * V[j * dv + e];
                            o[row * dv + e] = acc;
                        }
                    }
                    if (o_lat) {
                        double *ol = o_lat + row * r;
                        for (int rho = 0; rho < r; ++rho) ol[rho] = 0.0;
                        for (int64_t j = 0; j <= p; ++j) {
                            int64_t co = 0, ro = 0;
                            tok_offsets(c, b, j, &co, &ro);
                            for (int rho = 0; rho < r; ++rho) ol[rho] += s[j] * orc_bf16_value(c->c_kv[co + rho]);
                        }
                    }
                }
            }
        }
        free(K); free(V); free(KR); free(cj); free(s); free(qr);
    }
    if (err) return err;
    if (out && w_o && o && d->hidden > 0) {
        const int D = d->hidden;
        int64_t rows = (int64_t)n_seqs * q_len;
#pragma omp parallel for schedule(static)
        for (int64_t t = 0; t < rows; ++t) {
            int b = seqs ? seqs[t / q_len] : (int)(t / q_len);
            int i = (int)(t % q_len);
            int64_t row0 = ((int64_t)b * q_len + i) * H; /* first head of (b, i) */
            for (int n = 0; n < D; ++n) {
                const uint16_t *w = w_o + (int64_t)n * H * dv;
                double acc = 0.0;
                for (int h = 0; h < H; ++h)
                    for (int e = 0; e < dv; ++e)
                        acc += orc_bf16_value(w[h * dv + e]) * o[(row0 + h) * dv + e];
                out[((int64_t)b * q_len + i) * D + n] = acc;
            }
        }
    }
    return ORC_OK;
}

/* Projection of new hidden states into the cache and the queries, ahead of
 * the decode step (Sec. 3.2: the latent c_j = W^DKV h_j and a positional key
 * k^PE_j that is kept on the rotary path; Sec. 3.1 Eq. 1: q_{t,i} = W^Q_i h_t).
 * Readings: k^PE_j = R_j (W^KR h_j), one positional key shared by every head;
 * the converted query of head i is [q_nope (d_nope) ; q_pe (d_rope)], the
 * first part on the non-positional path and the second on the rotary path
 * (Sec. 3.3 routing).  Entry k of sequence b sits at position
 * start_pos[b] + k.  Every projection is an exact fp64 dot product of the
 * bf16 values; the cache receives the latent and the rotated positional key
 * each rounded once to bf16 (the rotation is applied to the exact fp64
 * projection), the queries are returned unrounded and unrotated.
 *   h      [batch, n_new, D] bf16, D = d->hidden (> 0)
 *   w_dkv  [rank, D], w_kr [d_rope, D], w_q [H (d_nope + d_rope), D] bf16
 *          (w_q may be NULL: no query projection)
 *   q_nope [batch, n_new, H, d_nope], q_pe [batch, n_new, H, d_rope] fp64 out
 *          (ignored when w_q is NULL) */
int orc_project_append(const orc_dims *d, const orc_cache *c, int batch, int n_new, const uint16_t *h,
                       const uint16_t *w_dkv, const uint16_t *w_kr, const uint16_t *w_q,
                       const int32_t *start_pos, double *q_nope, double *q_pe)
{
    if (check_dims(d) || batch < 0 || n_new < 0 || d->hidden <= 0) return ORC_BAD_ARG;
    const int D = d->hidden, r = d->rank, dr = d->d_rope, dn = d->d_nope, H = d->num_heads;
    const int dq = dn + dr;
    /* positions and pages first, so that a bad entry leaves the cache untouched */
    for (int b = 0; b < batch; ++b)
        for (int k = 0; k < n_new; ++k) {
            int64_t co, ro;
            int err = tok_offsets(c, b, (int64_t)start_pos[b] + k, &co, &ro);
            if (err) return err;
        }
    const int64_t rows = (int64_t)batch * n_new;
    int err = ORC_OK;
#pragma omp parallel for schedule(static)
    for (int64_t row = 0; row < rows; ++row) {
        const int b = (int)(row / (n_new > 0 ? n_new : 1)), k = (int)(row % (n_new > 0 ? n_new : 1));
        const int64_t pos = (int64_t)start_pos[b] + k;
        int64_t co, ro;
        tok_offsets(c, b, pos, &co, &ro);
        double *x = (double *)malloc(sizeof(double) * (size_t)(D + dr + 1));
        if (!x) {
#pragma omp critical
            err = ORC_NO_MEMORY;
            continue;
        }
        double *kr = x + D;
        for (int e = 0; e < D; ++e) x[e] = orc_bf16_value(h[row * D + e]);
        for (int e = 0; e < r; ++e) {  /* c = W^DKV h */
            double acc = 0.0;
            for (int t = 0; t < D; ++t) acc += orc_bf16_value(w_dkv[(int64_t)e * D + t]) * x[t];
            c->c_kv[co + e] = orc_bf16_round(acc);
        }
        for (int e = 0; e < dr; ++e) {  /* k^PE = R_pos W^KR h */
            double acc = 0.0;
            for (int t = 0; t < D; ++t) acc += orc_bf16_value(w_kr[(int64_t)e * D + t]) * x[t];
            kr[e] = acc;
        }
        orc_rope(kr, kr, dr, pos, d->rope_base, d->rope_style);
        for (int e = 0; e < dr; ++e) c->k_rope[ro + e] = orc_bf16_round(kr[e]);
        if (w_q) {  /* q_i = W^Q_i h, split into the two paths */
            for (int hd = 0; hd < H; ++hd)
                for (int e = 0; e < dq; ++e) {
                    const uint16_t *w = w_q + ((int64_t)hd * dq + e) * D;
                    double acc = 0.0;
                    for (int t = 0; t < D; ++t) acc += orc_bf16_value(w[t]) * x[t];
                    if (e < dn)
                        q_nope[(row * H + hd) * dn + e] = acc;
                    else
                        q_pe[(row * H + hd) * dr + (e - dn)] = acc;
                }
        }
        free(x);
    }
    return err;
}

/* Acceptance statistics of a draft against its target at the same contexts
 * (Sec. 3.3, Eqs. 9-10), one row per context, over the vocabulary:
 *   p_D = softmax(draft row), p_T = softmax(target row)   (temperature 1)
 *   alpha_sample = sum_y min(p_D(y), p_T(y))              (Eq. 9)
 *   argmax_D, argmax_T: index of the largest logit, the lowest index among
 *   equal maxima (the paper does not say how ties break); the decision is
 *   taken on the logits themselves, softmax being monotone
 *   greedy = [argmax_D == argmax_T]                        (Eq. 10)
 * Logits are given as exact fp64 values; every sum is fp64.
 *   draft, target [rows, vocab]; outputs [rows] (any may be NULL). */
int orc_acceptance(int rows, int vocab, const double *draft, const double *target, double *alpha,
                   int32_t *argmax_d, int32_t *argmax_t, int32_t *greedy)
{
    if (rows < 0 || vocab <= 0) return ORC_BAD_ARG;
#pragma omp parallel for schedule(static)
    for (int r = 0; r < rows; ++r) {
        const double *d = draft + (int64_t)r * vocab, *t = target + (int64_t)r * vocab;
        int ad = 0, at = 0;
        for (int y = 1; y < vocab; ++y) {
            if (d[y] > d[ad]) ad = y;
            if (t[y] > t[at]) at = y;
        }
        const double md = d[ad], mt = t[at];
        double zd = 0.0, zt = 0.0;
        for (int y = 0; y < vocab; ++y) {
            zd += exp(d[y] - md);
            zt += exp(t[y] - mt);
        }
        double acc = 0.0;
        for (int y = 0; y < vocab; ++y) {
            const double pd = exp(d[y] - md) / zd, pt = exp(t[y] - mt) / zt;
            acc += pd < pt ? pd : pt;
        }
        if (alpha) alpha[r] = acc;
        if (argmax_d) argmax_d[r] = ad;
        if (argmax_t) argmax_t[r] = at;
        if (greedy) greedy[r] = ad == at;
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------ original GQA
 * The unconverted draft the paper compares against (Sec. 3.1, Eqs. 1-4): each
 * KV group g keeps its own key and value cache.  Keys are stored rotated to
 * their own position (R_j k_j), so the score of query q at position p with key
 * j is (R_p q) . (R_j k_j) = q^T R_pj k_j.  Cache blocks: sequence b, group g
 * is block b * G + g (contiguous) or block-table row b * G + g (paged); in
 * orc_cache, c_kv holds the values (d_v per token) and k_rope the keys (d_k). */
typedef struct {
    int32_t num_heads;     /* H                                        */
    int32_t num_kv_groups; /* G, H % G == 0                            */
    int32_t d_k;           /* key / query width per head (even)       */
    int32_t d_v;           /* value width per head                    */
    double sm_scale;       /* 1/sqrt(d_k)                             */
    int32_t rope_style;
    double rope_base;
} orc_gqa_dims;

/* New keys and values of every (sequence, group) at positions start_pos[b] + k:
 * the key rotated in fp64 and rounded once to bf16, the value copied.
 *   k_new [batch, n_new, G, d_k], v_new [batch, n_new, G, d_v] bf16 */
int orc_gqa_append(const orc_gqa_dims *d, const orc_cache *c, int batch, int n_new, const uint16_t *k_new,
                   const uint16_t *v_new, const int32_t *start_pos)
{
    const int G = d->num_kv_groups, dk = d->d_k, dv = d->d_v;
    if (G <= 0 || dk <= 0 || (dk & 1) || dv <= 0 || batch < 0 || n_new < 0) return ORC_BAD_ARG;
    double *tmp = (double *)malloc(sizeof(double) * (size_t)dk);
    if (!tmp) return ORC_NO_MEMORY;
    int err = ORC_OK;
    for (int b = 0; b < batch && !err; ++b)
        for (int g = 0; g < G && !err; ++g)
            for (int k = 0; k < n_new && !err; ++k) {
                const int64_t pos = (int64_t)start_pos[b] + k, e0 = ((int64_t)b * n_new + k) * G + g;
                int64_t co, ro;
                err = tok_offsets(c, b * G + g, pos, &co, &ro);
                if (err) break;
                for (int e = 0; e < dv; ++e) c->c_kv[co + e] = v_new[e0 * dv + e];
                for (int e = 0; e < dk; ++e) tmp[e] = orc_bf16_value(k_new[e0 * dk + e]);
                orc_rope(tmp, tmp, dk, pos, d->rope_base, d->rope_style);
                for (int e = 0; e < dk; ++e) c->k_rope[ro + e] = orc_bf16_round(tmp[e]);
            }
    free(tmp);
    return err;
}

/* One decode step of GQA attention: for b, query i at p = kv_len[b] - q_len + i,
 * head h of group g = h / (H / G):
 *   s_j = sm_scale * (R_p q[b, i, h]) . K[b, g, j]   (j = 0 .. p)
 *   o[b, i, h] = sum_j softmax(s)_j V[b, g, j],  lse = ln sum_j exp(s_j)
 *   q [batch, q_len, H, d_k] bf16 (not rotated); o [batch, q_len, H, d_v], lse [batch, q_len, H] */
int orc_gqa_decode(const orc_gqa_dims *d, const orc_cache *c, int batch, int q_len, const int32_t *kv_len,
                   const uint16_t *q, double *o, double *lse)
{
    const int H = d->num_heads, G = d->num_kv_groups, dk = d->d_k, dv = d->d_v;
    if (H <= 0 || G <= 0 || H % G || dk <= 0 || (dk & 1) || dv <= 0 || batch < 0 || q_len <= 0) return ORC_BAD_ARG;
    const int hpg = H / G;
    for (int b = 0; b < batch; ++b)
        if (kv_len[b] < q_len || kv_len[b] > c->capacity) return ORC_BAD_POSITION;
    const int64_t rows = (int64_t)batch * q_len * H;
    int err = ORC_OK;
#pragma omp parallel for schedule(dynamic)
    for (int64_t row = 0; row < rows; ++row) {
        const int h = (int)(row % H), i = (int)((row / H) % q_len), b = (int)(row / ((int64_t)H * q_len));
        const int g = h / hpg;
        const int64_t p = (int64_t)kv_len[b] - q_len + i;
        double *qr = (double *)malloc(sizeof(double) * (size_t)(dk + p + 1));
        if (!qr) {
#pragma omp critical
            err = ORC_NO_MEMORY;
            continue;
        }
        double *s = qr + dk;
        for (int e = 0; e < dk; ++e) qr[e] = orc_bf16_value(q[row * dk + e]);
        orc_rope(qr, qr, dk, p, d->rope_base, d->rope_style);
        double m = -INFINITY;
        for (int64_t j = 0; j <= p; ++j) {
            int64_t co, ro;
            tok_offsets(c, b * G + g, j, &co, &ro);
            double acc = 0.0;
            for (int e = 0; e < dk; ++e) acc += qr[e] * orc_bf16_value(c->k_rope[ro + e]);
            s[j] = d->sm_scale * acc;
            if (s[j] > m) m = s[j];
        }
        double z = 0.0;
        for (int64_t j = 0; j <= p; ++j) z += exp(s[j] - m);
        for (int e = 0; e < dv; ++e) {
            double acc = 0.0;
            for (int64_t j = 0; j <= p; ++j) {
                int64_t co, ro;
                tok_offsets(c, b * G + g, j, &co, &ro);
                acc += exp(s[j] - m) * orc_bf16_value(c->c_kv[co + e]);
            }
            o[row * dv + e] = acc / z;
        }
        if (lse) lse[row] = m + log(z);
        free(qr);
    }
    return err;
}

/* Forward value of the E2E functional-reconstruction loss of one layer
 * (Sec. 4.1): the masked mean-squared error between the converted MLA
 * block's post-W_O output and the frozen original block's,
 *   L = sum_t M_t sum_d (A_MLA[t, d] - A_orig[t, d])^2 / (D sum_t M_t),
 * over rows t (tokens) with mask M_t in {0, 1} (mask NULL: every row counts).
 * A row set with no counted row gives 0.  a_mla, a_orig [rows, D] fp64. */
int orc_e2e_loss(int rows, int hidden, const double *a_mla, const double *a_orig, const uint8_t *mask,
                 double *loss)
{
    if (rows < 0 || hidden <= 0 || !loss) return ORC_BAD_ARG;
    double num = 0.0, den = 0.0;
    for (int t = 0; t < rows; ++t) {
        if (mask && !mask[t]) continue;
        for (int e = 0; e < hidden; ++e) {
            const double d = a_mla[(int64_t)t * hidden + e] - a_orig[(int64_t)t * hidden + e];
            num += d * d;
        }
        den += 1.0;
    }
    *loss = den > 0.0 ? num / ((double)hidden * den) : 0.0;
    return ORC_OK;
}
