/*
 * kvx_oracle.c -- CPU oracle for cross-model KV translation.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline leg of bench.py may load this code.  The product path (the CUDA
 * library under paper_2608_30963_gb300/) never calls it and shares no code,
 * header, table or constant with it.
 *
 * What it computes (paper Section 4, translation operator KV^_B = T_{A->B}(KV_A),
 * and Section 5, parameterised translator T_theta, at the granularities
 * Section 5 lists: individual KV heads, individual layers, groups of layers,
 * low-dimensional latent adapters).  For every target layer j, target KV head
 * h, K or V, and target token t of sequence b:
 *
 *   1. source layers    l_k = layer_map[j][k], k < k_layers (one: nearest
 *                       relative depth; several: a group of source layers)
 *   2. source span      [lo_t, hi_t) of the source tokens of sequence b
 *   3. for every s in the span, every source layer l_k and every source head
 *      g feeding target head h (its GQA group, or all heads in the dense
 *      per-layer form):
 *        K: u = R_{d_s,base_s}(-p_s) K[l_k,b,g,s]   (undo the source RoPE)
 *        V: u = V[l_k,b,g,s]
 *      concatenated layer by layer, heads ascending within a layer (length in)
 *   4. xbar = (1/|span|) sum_s u                      (span mean)
 *   5. y = xbar . W[j,h]      with W[j,h] of shape [in, out=d_t]; for a
 *      low-rank latent adapter, z = xbar . A[j,h] ([in, rank]) and then
 *      y = z . B[j,h] ([rank, out])
 *   6. K: y <- R_{d_t,base_t}(+p_t) y                 (apply the target RoPE)
 *
 * R_{d,base}(p) is the half-split rotary map: channel pairs (i, i+d/2) for
 * i < d/2 are rotated by the angle p * theta_i, theta_i = base^(-2i/d) or its
 * rescaled form under the model's frequency schedule (kvxo_theta).  The angle
 * is taken in exact (double) arithmetic.  A base <= 0 means "no RoPE".
 *
 * Everything runs in double precision, in the order above, with no blocking,
 * fusion or reordering.  Inputs are float32 arrays (bf16 storage is widened
 * exactly by the caller).
 */
#define _DEFAULT_SOURCE
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define KVXO_API __attribute__((visibility("default")))

/* ---------------------------------------------------------------------- */
/* Layer alignment: target layer j draws from the source layer nearest to it
 * in relative depth, depth(j) = j/(L_t-1), depth(s) = s/(L_s-1).  Ties round
 * to the deeper layer.  Implemented as an explicit argmin over all source
 * layers with exact integer cross-multiplication. */
KVXO_API int kvxo_layer_map_nearest(int Ls, int Lt, int32_t* out)
{
    if (Ls < 1 || Lt < 1 || !out) return 1;
    for (int j = 0; j < Lt; ++j) {
        if (Lt == 1 || Ls == 1) { out[j] = 0; continue; }
        /* |s/(Ls-1) - j/(Lt-1)| compared as |s*(Lt-1) - j*(Ls-1)| */
        int best = 0;
        int64_t best_d = INT64_MAX;
        for (int s = 0; s < Ls; ++s) {
            int64_t d = (int64_t)s * (Lt - 1) - (int64_t)j * (Ls - 1);
            if (d < 0) d = -d;
            if (d <= best_d) { best = s; best_d = d; }   /* '<=': ties go deeper */
        }
        out[j] = best;
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Token-span alignment between two tokenisations of the same byte string
 * (the paper names tokenizer differences among the model differences the
 * translator must bridge, Sections 1 and 4).
 *
 * Byte-end offsets per sequence are strictly increasing and relative to the
 * sequence start.  Source token s covers bytes [src_end[s-1], src_end[s]);
 * target token t covers [tgt_end[t-1], tgt_end[t]).  Source token s belongs to
 * the target token whose byte range holds s's last byte.  A target token that
 * receives no source token takes the single source token holding its own last
 * byte.  Output spans are within-sequence source indices [lo, hi).
 *
 * Walks both sequences with one merge pointer.  Returns the number of target
 * tokens whose span had to be clamped because the source text ended first. */
KVXO_API int kvxo_build_alignment(int batch,
                                  const int32_t* src_seq_off, const int32_t* src_end,
                                  const int32_t* tgt_seq_off, const int32_t* tgt_end,
                                  int32_t* span_lo, int32_t* span_hi)
{
    int clamped = 0;
    for (int b = 0; b < batch; ++b) {
        const int32_t* se = src_end + src_seq_off[b];
        const int32_t* te = tgt_end + tgt_seq_off[b];
        int S = src_seq_off[b + 1] - src_seq_off[b];
        int T = tgt_seq_off[b + 1] - tgt_seq_off[b];
        int s = 0;                       /* first source token not yet assigned */
        for (int t = 0; t < T; ++t) {
            int lo = s;
            while (s < S && se[s] <= te[t]) ++s;   /* last byte se[s]-1 < te[t] */
            int hi = s;
            if (hi == lo) {              /* empty: source token holding byte te[t]-1 */
                hi = lo + 1;
                if (lo >= S) { lo = S - 1; hi = S; ++clamped; }
            }
            span_lo[tgt_seq_off[b] + t] = lo;
            span_hi[tgt_seq_off[b] + t] = hi;
        }
    }
    return clamped;
}

/* ---------------------------------------------------------------------- */
/* Rotary frequency schedule of one model.  type 0: the plain RoFormer
 * frequencies theta_i = base^(-2i/d).  type 1: linear position interpolation,
 * the angle of position p is that of p / factor.  type 2: the Llama-3.1
 * frequency-dependent rescaling: a pair whose wavelength 2 pi / theta_i is
 * shorter than orig_ctx / high keeps theta_i, one longer than orig_ctx / low
 * gets theta_i / factor, and in between the two are mixed with weight
 * m = (orig_ctx / wavelength - low) / (high - low) on the unscaled frequency. */
typedef struct {
    double base;          /* <= 0: no rotary encoding */
    int32_t type;
    double factor, low, high;
    int32_t orig_ctx;
    int32_t rot;          /* channels that rotate (partial rotary: the first rot); 0 = all d */
} kvxo_rope_sched;

static double kvxo_theta(const kvxo_rope_sched* r, int i, int d)
{
    double theta = pow(r->base, -2.0 * (double)i / (double)d);
    if (r->type == 1) return theta / r->factor;
    if (r->type == 2) {
        double wavelength = 2.0 * M_PI / theta;
        double short_edge = (double)r->orig_ctx / r->high;   /* below: high-frequency band */
        double long_edge = (double)r->orig_ctx / r->low;     /* above: low-frequency band */
        if (wavelength < short_edge) return theta;
        if (wavelength > long_edge) return theta / r->factor;
        double m = ((double)r->orig_ctx / wavelength - r->low) / (r->high - r->low);
        return m * theta + (1.0 - m) * theta / r->factor;
    }
    return theta;
}

/* Half-split rotary map on one head vector of length d (d even).  With n rotated
 * channels (n = r->rot, or d when 0; a partial rotary head rotates only its first
 * n channels and passes the rest through) and h = n/2:
 * x'[i] = x[i] cos a - x[i+h] sin a,  x'[i+h] = x[i+h] cos a + x[i] sin a  (i < h),
 * a = sign * pos * theta_i, theta_i taken over the n rotated channels (base^(-2i/n)).
 * sign = +1 applies the RoPE, -1 undoes it. */
KVXO_API void kvxo_rope_sched_apply(double* x, int d, const kvxo_rope_sched* r, double pos, int sign)
{
    if (r->base <= 0.0) return;
    int n = r->rot > 0 ? r->rot : d;
    int h = n / 2;
    for (int i = 0; i < h; ++i) {
        double a = (double)sign * pos * kvxo_theta(r, i, n);
        double c = cos(a), sn = sin(a);
        double x0 = x[i], x1 = x[i + h];
        x[i]     = x0 * c - x1 * sn;
        x[i + h] = x1 * c + x0 * sn;
    }
}

/* The plain schedule (type 0) with the given base. */
KVXO_API void kvxo_rope(double* x, int d, double base, double pos, int sign)
{
    kvxo_rope_sched r = {base, 0, 1.0, 1.0, 1.0, 1, 0};
    kvxo_rope_sched_apply(x, d, &r, pos, sign);
}

/* ---------------------------------------------------------------------- */
typedef struct {
    int32_t Ls, Hs, ds; kvxo_rope_sched rope_s;   /* source geometry */
    int32_t Lt, Ht, dt; kvxo_rope_sched rope_t;   /* target geometry */
    const int32_t* layer_map;                 /* [Lt] */
    int32_t batch, s_max, t_max;
    const int32_t* src_len;                   /* [B] */
    const int32_t* tgt_seq_off;               /* [B+1] packed target offsets */
    const int32_t* span_lo;                   /* [T_total] or NULL (identity) */
    const int32_t* span_hi;
    const int32_t* src_pos;                   /* [B*s_max] or NULL (= index) */
    const int32_t* tgt_pos;                   /* [T_total] or NULL (= index) */
    const float* const* src_k;                /* [Ls] -> [B][Hs][s_max][ds] */
    const float* const* src_v;
    const float* w_k;                         /* [Lt][Ht][in][dt] (full-rank form) */
    const float* w_v;
    int32_t form;                             /* 0: GQA group of source heads, 1: all source heads */
    int32_t k_layers;                         /* source layers per target layer (layer_map [Lt][k]) */
    int32_t rank;                             /* > 0: latent adapter A [Lt][Ht][in][rank], B [Lt][Ht][rank][dt] */
    const float* a_k; const float* b_k;
    const float* a_v; const float* b_v;
} kvxo_problem;

/* Source heads per source layer that feed one target head. */
static int heads_per_layer(const kvxo_problem* p)
{
    if (p->form == 1) return p->Hs;
    return p->Hs >= p->Ht ? p->Hs / p->Ht : 1;
}

static int layers_per_target(const kvxo_problem* p) { return p->k_layers > 0 ? p->k_layers : 1; }

static int group_in(const kvxo_problem* p)
{
    return layers_per_target(p) * heads_per_layer(p) * p->ds;
}

KVXO_API int kvxo_group_in(const kvxo_problem* p) { return group_in(p); }

/* Steps 1-4 for one target token: the translator's input row xbar (length
 * group_in) of target layer j, head h, kv (0 = K, 1 = V), packed target token
 * tp.  Returns nonzero on a geometry it cannot place. */
KVXO_API int kvxo_input_row(const kvxo_problem* p, int j, int h, int kv, int tp, double* sum)
{
    if (p->Hs % p->Ht != 0 && p->Ht % p->Hs != 0) return 1;
    if (p->form != 0 && p->form != 1) return 1;
    int b = 0;
    while (b < p->batch - 1 && p->tgt_seq_off[b + 1] <= tp) ++b;
    int t = tp - p->tgt_seq_off[b];
    int K = layers_per_target(p);
    int lo = p->span_lo ? p->span_lo[tp] : t;                  /* step 2 */
    int hi = p->span_hi ? p->span_hi[tp] : t + 1;
    int in = group_in(p);
    int nh = heads_per_layer(p);
    int g0 = p->form == 1 ? 0 : (p->Hs >= p->Ht ? h * nh : h / (p->Ht / p->Hs));

    for (int i = 0; i < in; ++i) sum[i] = 0.0;
    double* u = (double*)malloc(sizeof(double) * (size_t)p->ds);
    for (int s = lo; s < hi; ++s) {                            /* step 3 */
        double ps = p->src_pos ? (double)p->src_pos[(size_t)b * p->s_max + s] : (double)s;
        for (int k = 0; k < K; ++k) {
            int l = p->layer_map[j * K + k];                   /* step 1 */
            const float* src = kv == 0 ? p->src_k[l] : p->src_v[l];
            for (int q = 0; q < nh; ++q) {
                int g = g0 + q;
                const float* row = src + (((size_t)b * p->Hs + g) * p->s_max + s) * p->ds;
                for (int e = 0; e < p->ds; ++e) u[e] = (double)row[e];
                if (kv == 0) kvxo_rope_sched_apply(u, p->ds, &p->rope_s, ps, -1);
                for (int e = 0; e < p->ds; ++e) sum[(k * nh + q) * p->ds + e] += u[e];
            }
        }
    }
    double n = (double)(hi - lo);                              /* step 4 */
    for (int i = 0; i < in; ++i) sum[i] /= n;
    free(u);
    return 0;
}

/* One output row: target layer j, target head h, kv (0 = K, 1 = V), packed
 * target token index tp.  Writes d_t doubles.  Returns nonzero on a
 * geometry it cannot place. */
KVXO_API int kvxo_translate_row(const kvxo_problem* p, int j, int h, int kv, int tp, double* out)
{
    int in = group_in(p);
    double* sum = (double*)malloc(sizeof(double) * (size_t)in);
    if (kvxo_input_row(p, j, h, kv, tp, sum)) { free(sum); return 1; }
    int b = 0;
    while (b < p->batch - 1 && p->tgt_seq_off[b + 1] <= tp) ++b;
    int t = tp - p->tgt_seq_off[b];

    if (p->rank > 0) {                                         /* step 5, latent adapter */
        size_t jh = (size_t)j * p->Ht + h;
        const float* A = (kv == 0 ? p->a_k : p->a_v) + jh * (size_t)in * p->rank;
        const float* B = (kv == 0 ? p->b_k : p->b_v) + jh * (size_t)p->rank * p->dt;
        double* z = (double*)malloc(sizeof(double) * (size_t)p->rank);
        for (int c = 0; c < p->rank; ++c) {
            double acc = 0.0;
            for (int i = 0; i < in; ++i) acc += sum[i] * (double)A[(size_t)i * p->rank + c];
            z[c] = acc;
        }
        for (int o = 0; o < p->dt; ++o) {
            double acc = 0.0;
            for (int c = 0; c < p->rank; ++c) acc += z[c] * (double)B[(size_t)c * p->dt + o];
            out[o] = acc;
        }
        free(z);
    } else {                                                   /* step 5 */
        const float* W = (kv == 0 ? p->w_k : p->w_v) + ((size_t)j * p->Ht + h) * (size_t)in * p->dt;
        for (int o = 0; o < p->dt; ++o) {
            double acc = 0.0;
            for (int i = 0; i < in; ++i) acc += sum[i] * (double)W[(size_t)i * p->dt + o];
            out[o] = acc;
        }
    }
    if (kv == 0) {                                             /* step 6 */
        double pt = p->tgt_pos ? (double)p->tgt_pos[tp] : (double)t;
        kvxo_rope_sched_apply(out, p->dt, &p->rope_t, pt, +1);
    }
    free(sum);
    return 0;
}

/* Whole translation.  out_k / out_v: [Lt][Ht][T_total][dt] doubles. */
KVXO_API int kvxo_translate(const kvxo_problem* p, double* out_k, double* out_v)
{
    int T = p->tgt_seq_off[p->batch];
    for (int j = 0; j < p->Lt; ++j)
        for (int h = 0; h < p->Ht; ++h)
            for (int tp = 0; tp < T; ++tp) {
                size_t o = (((size_t)j * p->Ht + h) * T + tp) * p->dt;
                if (kvxo_translate_row(p, j, h, 0, tp, out_k + o)) return 1;
                if (kvxo_translate_row(p, j, h, 1, tp, out_v + o)) return 1;
            }
    return 0;
}

/* Apply (sign=+1) or undo (sign=-1) the RoPE on every row of a KV cache laid
 * out [B][H][S][d] (float32 in place, arithmetic in double).  pos: [B*S]
 * positions or NULL (= token index).  Used to synthesise post-RoPE source
 * caches the way a source model's prefill would have stored them. */
KVXO_API void kvxo_rope_cache(float* x, int B, int H, int S, int d, const kvxo_rope_sched* r,
                              const int32_t* pos, int sign)
{
    double* row = (double*)malloc(sizeof(double) * (size_t)d);
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h)
            for (int s = 0; s < S; ++s) {
                float* xr = x + (((size_t)b * H + h) * S + s) * d;
                for (int e = 0; e < d; ++e) row[e] = (double)xr[e];
                double p = pos ? (double)pos[(size_t)b * S + s] : (double)s;
                kvxo_rope_sched_apply(row, d, r, p, sign);
                for (int e = 0; e < d; ++e) xr[e] = (float)row[e];
            }
    free(row);
}

/* ---------------------------------------------------------------------- */
/* Closed-form fit of the linear translator.  Section 5 gives the objective
 * L_KV = D(T_theta(KV_A(C)), KV_B(C)), the distance between the translated
 * cache and the cache the target's own prefill builds.  With D the squared
 * Euclidean distance summed over target tokens, plus a ridge term
 * lambda |W|^2, and T_theta linear in W, each (target layer j, head h, K|V)
 * is an independent least-squares problem:
 *
 *   W = argmin_W  sum_t |x_t W - y_t|^2 + lambda |W|^2,
 *   i.e. the normal equations (X^T X + lambda I) W = X^T Y,
 *
 * where x_t is the input row of target token t (steps 1-4 above) and y_t the
 * target model's own cache row with the target RoPE undone (K; the rotation
 * is orthogonal, so the distance is the same before and after it) or as
 * stored (V).  Solved with a Cholesky factorisation X^T X + lambda I = L L^T
 * and two triangular solves per output column, all in double.
 *
 * tgt_k, tgt_v: [Lt] arrays of the target caches, each [B][Ht][t_max][dt].
 * w_k_out, w_v_out: [Lt][Ht][in][dt].  Returns nonzero if a system is not
 * positive definite or the geometry cannot be placed. */
KVXO_API int kvxo_fit(const kvxo_problem* p, const float* const* tgt_k, const float* const* tgt_v, double lambda,
                      double* w_k_out, double* w_v_out)
{
    int in = group_in(p), dt = p->dt, T = p->tgt_seq_off[p->batch];
    double* G = (double*)malloc(sizeof(double) * (size_t)in * in);
    double* Cm = (double*)malloc(sizeof(double) * (size_t)in * dt);
    double* x = (double*)malloc(sizeof(double) * (size_t)in);
    double* y = (double*)malloc(sizeof(double) * (size_t)dt);
    int rc = 0;
    for (int j = 0; j < p->Lt && !rc; ++j)
        for (int h = 0; h < p->Ht && !rc; ++h)
            for (int kv = 0; kv < 2 && !rc; ++kv) {
                memset(G, 0, sizeof(double) * (size_t)in * in);
                memset(Cm, 0, sizeof(double) * (size_t)in * dt);
                for (int tp = 0; tp < T; ++tp) {
                    if (kvxo_input_row(p, j, h, kv, tp, x)) { rc = 1; break; }
                    int b = 0;
                    while (b < p->batch - 1 && p->tgt_seq_off[b + 1] <= tp) ++b;
                    int t = tp - p->tgt_seq_off[b];
                    const float* row = (kv == 0 ? tgt_k[j] : tgt_v[j]) +
                                       (((size_t)b * p->Ht + h) * p->t_max + t) * dt;
                    for (int o = 0; o < dt; ++o) y[o] = (double)row[o];
                    if (kv == 0) {
                        double pt = p->tgt_pos ? (double)p->tgt_pos[tp] : (double)t;
                        kvxo_rope_sched_apply(y, dt, &p->rope_t, pt, -1);
                    }
                    for (int a = 0; a < in; ++a) {
                        for (int c = 0; c < in; ++c) G[(size_t)a * in + c] += x[a] * x[c];
                        for (int o = 0; o < dt; ++o) Cm[(size_t)a * dt + o] += x[a] * y[o];
                    }
                }
                if (rc) break;
                for (int a = 0; a < in; ++a) G[(size_t)a * in + a] += lambda;
                /* Cholesky: G = L L^T, L stored in the lower triangle of G */
                for (int c = 0; c < in && !rc; ++c) {
                    double d = G[(size_t)c * in + c];
                    for (int k = 0; k < c; ++k) d -= G[(size_t)c * in + k] * G[(size_t)c * in + k];
                    if (!(d > 0.0)) { rc = 2; break; }
                    d = sqrt(d);
                    G[(size_t)c * in + c] = d;
                    for (int r = c + 1; r < in; ++r) {
                        double v = G[(size_t)r * in + c];
                        for (int k = 0; k < c; ++k) v -= G[(size_t)r * in + k] * G[(size_t)c * in + k];
                        G[(size_t)r * in + c] = v / d;
                    }
                }
                if (rc) break;
                double* W = (kv == 0 ? w_k_out : w_v_out) + ((size_t)j * p->Ht + h) * (size_t)in * dt;
                for (int o = 0; o < dt; ++o) {
                    /* L z = c (forward), then L^T w = z (backward) */
                    for (int r = 0; r < in; ++r) {
                        double v = Cm[(size_t)r * dt + o];
                        for (int k = 0; k < r; ++k) v -= G[(size_t)r * in + k] * x[k];
                        x[r] = v / G[(size_t)r * in + r];
                    }
                    for (int r = in - 1; r >= 0; --r) {
                        double v = x[r];
                        for (int k = r + 1; k < in; ++k) v -= G[(size_t)k * in + r] * W[(size_t)k * dt + o];
                        W[(size_t)r * dt + o] = v / G[(size_t)r * in + r];
                    }
                }
            }
    free(G); free(Cm); free(x); free(y);
    return rc;
}
