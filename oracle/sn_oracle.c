/*
 * sn_oracle.c -- the CPU oracle for the SoftNeuro hot path (arXiv 2110.06037).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * load this file: only the test suite, the smoke check and the CPU-baseline
 * leg of the benchmark use it.  It shares no code, header or constant with
 * the CUDA library; the two meet only through arrays handed in by the tests.
 *
 * Everything here is a plain definition written out, in fp64 where the data
 * are floating point and in exact int64 where they are costs:
 *
 *   numerics (what every routine of a layer must compute, whatever its
 *   algorithm; routines differ only in speed, section III-C):
 *     - conv2: 2-D cross-correlation with zero padding, strides, dilations and
 *       channel groups; the layer parameters are those the paper lists for
 *       conv2 (section III-B) and the sum is the convolution written out in
 *       section II (no kernel flip).  Bias and ReLU/ReLU6 are folded into the
 *       layer as the importer's graph optimisation does (section III-A).
 *     - max pooling (-inf padding), global average pooling, elementwise add
 *       (+ optional ReLU), dense y = W x + b.
 *     - IEEE-754 round-to-nearest-even casts fp32 -> binary16 / bfloat16 and
 *       the exact widening back, written from the definition of the formats
 *       (value grid + ties-to-even), not from any vendor routine.
 *     - NCHW <-> NHWC permutation (an adapt layer's layout change, III-C).
 *
 *   path search (what DPRS must return, section IV):
 *     - F_i(lambda) = min over routines of schema lambda of T(r)      (Eq. 1)
 *     - T(S) = sum of the routine times in S plus one adapt time per edge
 *       whose endpoint schemas differ; a void adapt costs 0 (Def. 1, Def. 2,
 *       section IV-F)
 *     - S* = argmin over every schema assignment, by exhaustive enumeration
 *       (Def. 2, Eq. 2).  Ties go to the lexicographically smallest
 *       assignment, layer 0 most significant, lower schema index first.
 *
 * All layouts inside the oracle are NCHW, row-major, contiguous.
 * Costs: int64 nanoseconds, INT64_MAX = infeasible, saturating addition.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <fenv.h>

#define OR_INF INT64_MAX

enum { OR_ACT_NONE = 0, OR_ACT_RELU = 1, OR_ACT_RELU6 = 2, OR_ACT_HSWISH = 3, OR_ACT_HSIGMOID = 4 };

static double or_relu6(double v) { return v < 0.0 ? 0.0 : (v > 6.0 ? 6.0 : v); }

/* ReLU, ReLU6, and MobileNetV3's hard swish x * ReLU6(x + 3) / 6 and hard
 * sigmoid ReLU6(x + 3) / 6 */
static double or_act(double v, int act) {
    if (act == OR_ACT_RELU) return v > 0.0 ? v : 0.0;
    if (act == OR_ACT_RELU6) return or_relu6(v);
    if (act == OR_ACT_HSWISH) return v * or_relu6(v + 3.0) / 6.0;
    if (act == OR_ACT_HSIGMOID) return or_relu6(v + 3.0) / 6.0;
    return v;
}

/* ------------------------------------------------------------------------ */
/* conv2 (section II formula, section III-B parameters)                      */
/* ------------------------------------------------------------------------ */

/* Output extent along one axis: floor((H + 2p - d(k-1) - 1)/s) + 1. */
int64_t or_conv_out_dim(int64_t in, int64_t k, int64_t s, int64_t p, int64_t d) {
    int64_t span = d * (k - 1) + 1;
    if (in + 2 * p < span) return 0;
    return (in + 2 * p - span) / s + 1;
}

/*
 * y[n,k,p,q] = act( b[k] + sum_{c in group(k)} sum_{r,s}
 *                   x[n, c, p*sh - ph + r*dh, q*sw - pw + s*dw] * w[k, c - c0(k), r, s] )
 * with x = 0 outside the image.  w is [K, C/groups, R, S]; b may be NULL.
 * Returns 0, or -1 on inconsistent sizes.
 */
int or_conv2d(const double *x, int64_t N, int64_t C, int64_t H, int64_t W,
              const double *w, const double *b, int64_t K, int64_t R, int64_t S,
              int64_t sh, int64_t sw, int64_t ph, int64_t pw, int64_t dh, int64_t dw,
              int64_t groups, int act, double *y) {
    if (groups <= 0 || C % groups || K % groups || sh <= 0 || sw <= 0 || dh <= 0 || dw <= 0)
        return -1;
    const int64_t P = or_conv_out_dim(H, R, sh, ph, dh);
    const int64_t Q = or_conv_out_dim(W, S, sw, pw, dw);
    const int64_t Cg = C / groups, Kg = K / groups;
    int64_t nk;
#pragma omp parallel for schedule(static)
    for (nk = 0; nk < N * K; ++nk) {
        const int64_t n = nk / K, k = nk % K;
        const int64_t c0 = (k / Kg) * Cg;
        for (int64_t p = 0; p < P; ++p) {
            for (int64_t q = 0; q < Q; ++q) {
                double acc = 0.0;
                for (int64_t c = 0; c < Cg; ++c) {
                    for (int64_t r = 0; r < R; ++r) {
                        const int64_t h = p * sh - ph + r * dh;
                        if (h < 0 || h >= H) continue;
                        for (int64_t s = 0; s < S; ++s) {
                            const int64_t ww = q * sw - pw + s * dw;
                            if (ww < 0 || ww >= W) continue;
                            acc += x[((n * C + c0 + c) * H + h) * W + ww] *
                                   w[((k * Cg + c) * R + r) * S + s];
                        }
                    }
                }
                if (b) acc += b[k];
                y[((n * K + k) * P + p) * Q + q] = or_act(acc, act);
            }
        }
    }
    return 0;
}

/* Max pooling with -inf padding (a window entirely in the padding gives -inf). */
int or_maxpool2d(const double *x, int64_t N, int64_t C, int64_t H, int64_t W,
                 int64_t kh, int64_t kw, int64_t sh, int64_t sw, int64_t ph, int64_t pw,
                 double *y) {
    if (sh <= 0 || sw <= 0) return -1;
    const int64_t P = or_conv_out_dim(H, kh, sh, ph, 1);
    const int64_t Q = or_conv_out_dim(W, kw, sw, pw, 1);
    int64_t nc;
#pragma omp parallel for schedule(static)
    for (nc = 0; nc < N * C; ++nc) {
        for (int64_t p = 0; p < P; ++p)
            for (int64_t q = 0; q < Q; ++q) {
                double m = -INFINITY;
                for (int64_t r = 0; r < kh; ++r) {
                    const int64_t h = p * sh - ph + r;
                    if (h < 0 || h >= H) continue;
                    for (int64_t s = 0; s < kw; ++s) {
                        const int64_t ww = q * sw - pw + s;
                        if (ww < 0 || ww >= W) continue;
                        const double v = x[(nc * H + h) * W + ww];
                        if (v > m) m = v;
                    }
                }
                y[(nc * P + p) * Q + q] = m;
            }
    }
    return 0;
}

/* Global average pooling: y[n,c] = (1/(H W)) sum_{h,w} x[n,c,h,w]. */
void or_gap(const double *x, int64_t N, int64_t C, int64_t H, int64_t W, double *y) {
    for (int64_t nc = 0; nc < N * C; ++nc) {
        double acc = 0.0;
        for (int64_t i = 0; i < H * W; ++i) acc += x[nc * H * W + i];
        y[nc] = acc / (double)(H * W);
    }
}

/* Elementwise y = act(a + b). */
void or_add(const double *a, const double *b, int64_t n, int act, double *y) {
    for (int64_t i = 0; i < n; ++i) y[i] = or_act(a[i] + b[i], act);
}

/* Per-channel scale (squeeze-and-excite): y[n,c,h,w] = act(x[n,c,h,w] * s[n,c]), NCHW. */
void or_mul(const double *x, const double *s, int64_t N, int64_t C, int64_t HW, int act, double *y) {
    for (int64_t nc = 0; nc < N * C; ++nc)
        for (int64_t i = 0; i < HW; ++i) y[nc * HW + i] = or_act(x[nc * HW + i] * s[nc], act);
}

/* Dense: y[n,o] = act(b[o] + sum_i W[o,i] x[n,i]); W is [out, in]. */
void or_dense(const double *x, const double *w, const double *b, int64_t N, int64_t in,
              int64_t out, int act, double *y) {
    int64_t no;
#pragma omp parallel for schedule(static)
    for (no = 0; no < N * out; ++no) {
        const int64_t n = no / out, o = no % out;
        double acc = 0.0;
        for (int64_t i = 0; i < in; ++i) acc += w[o * in + i] * x[n * in + i];
        if (b) acc += b[o];
        y[no] = or_act(acc, act);
    }
}

/* ------------------------------------------------------------------------ */
/* IEEE-754 casts, from the definition of the formats                         */
/* ------------------------------------------------------------------------ */

/*
 * Round the real value |v| (finite, exactly representable in double) to the
 * grid of a binary format with `mant_bits` stored fraction bits and minimum
 * normal exponent emin, ties to even.  Returns the rounded magnitude.  The
 * grid spacing in the binade [2^e, 2^(e+1)) is 2^(e - mant_bits); below 2^emin
 * it is 2^(emin - mant_bits) (subnormals).  v / spacing is exact in double
 * for every fp32 input, and nearbyint() under FE_TONEAREST rounds half to even.
 */
static double or_round_to_grid(double a, int mant_bits, int emin) {
    if (a == 0.0) return 0.0;
    int e = ilogb(a);
    if (e < emin) e = emin;
    const double quantum = ldexp(1.0, e - mant_bits);
    return nearbyint(a / quantum) * quantum;
}

/* Encode a magnitude already on the grid into sign | exponent | fraction bits. */
static uint32_t or_encode(double a, int mant_bits, int emin, int bias) {
    if (a == 0.0) return 0;
    int e = ilogb(a);
    if (e < emin) { /* subnormal: fraction = a / 2^(emin - mant_bits), exponent field 0 */
        return (uint32_t)ldexp(a, mant_bits - emin);
    }
    const uint32_t frac = (uint32_t)(ldexp(a, mant_bits - e) - ldexp(1.0, mant_bits));
    return ((uint32_t)(e + bias) << mant_bits) | frac;
}

static float or_bits_to_f32(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }
static uint32_t or_f32_to_bits(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }

/*
 * Generic fp32 -> {binary16, bfloat16} RNE.  `max_finite` is the largest
 * finite magnitude; magnitudes at or above the midpoint between it and the
 * next power of two (where RNE rounds away from the last finite value)
 * become infinity.  NaN keeps its sign and becomes the quiet NaN with the
 * top fraction bits of the input (always non-zero).
 */
static uint16_t or_f32_to_small(float f, int mant_bits, int emin, int bias, int exp_bits) {
    fesetround(FE_TONEAREST);
    const uint32_t u = or_f32_to_bits(f);
    const uint16_t sign = (uint16_t)((u >> 31) << 15);
    const uint16_t exp_all_ones = (uint16_t)(((1u << exp_bits) - 1u) << mant_bits);
    if (isnan(f)) {
        const uint32_t payload = (u & 0x7fffffu) >> (23 - mant_bits);
        return (uint16_t)(sign | exp_all_ones | (1u << (mant_bits - 1)) | payload);
    }
    if (isinf(f)) return (uint16_t)(sign | exp_all_ones);
    const double a = fabs((double)f);
    const int emax = (1 << (exp_bits - 1)) - 1;
    /* midpoint between the largest finite value (2 - 2^-m) 2^emax and 2^(emax+1) */
    const double overflow_mid = ldexp(2.0 - ldexp(1.0, -mant_bits - 1), emax);
    if (a >= overflow_mid) return (uint16_t)(sign | exp_all_ones);
    const double r = or_round_to_grid(a, mant_bits, emin);
    return (uint16_t)(sign | or_encode(r, mant_bits, emin, bias));
}

static float or_small_to_f32(uint16_t h, int mant_bits, int emin, int bias, int exp_bits) {
    const uint32_t sign = (uint32_t)(h >> 15);
    const uint32_t e = (h >> mant_bits) & ((1u << exp_bits) - 1u);
    const uint32_t frac = h & ((1u << mant_bits) - 1u);
    if (e == (1u << exp_bits) - 1u) {
        if (frac == 0) return or_bits_to_f32((sign << 31) | 0x7f800000u);
        return or_bits_to_f32((sign << 31) | 0x7f800000u | (frac << (23 - mant_bits)));
    }
    double v;
    if (e == 0) v = ldexp((double)frac, emin - mant_bits);
    else v = ldexp((double)((1u << mant_bits) | frac), (int)e - bias - mant_bits);
    return (float)(sign ? -v : v); /* exact: every small-format value is an fp32 value */
}

/* binary16: 10 fraction bits, 5 exponent bits, bias 15, emin -14. */
uint16_t or_f32_to_f16(float f) { return or_f32_to_small(f, 10, -14, 15, 5); }
float or_f16_to_f32(uint16_t h) { return or_small_to_f32(h, 10, -14, 15, 5); }
/* bfloat16: 7 fraction bits, 8 exponent bits, bias 127, emin -126. */
uint16_t or_f32_to_bf16(float f) { return or_f32_to_small(f, 7, -126, 127, 8); }
float or_bf16_to_f32(uint16_t h) { return or_small_to_f32(h, 7, -126, 127, 8); }

void or_cast_f32_to_f16(const float *x, uint16_t *y, int64_t n) {
    for (int64_t i = 0; i < n; ++i) y[i] = or_f32_to_f16(x[i]);
}
void or_cast_f32_to_bf16(const float *x, uint16_t *y, int64_t n) {
    for (int64_t i = 0; i < n; ++i) y[i] = or_f32_to_bf16(x[i]);
}
void or_cast_f16_to_f32(const uint16_t *x, float *y, int64_t n) {
    for (int64_t i = 0; i < n; ++i) y[i] = or_f16_to_f32(x[i]);
}
void or_cast_bf16_to_f32(const uint16_t *x, float *y, int64_t n) {
    for (int64_t i = 0; i < n; ++i) y[i] = or_bf16_to_f32(x[i]);
}

/* ------------------------------------------------------------------------ */
/* Layout permutation (adapt layer, layout change)                           */
/* ------------------------------------------------------------------------ */

/* y[n,h,w,c] = x[n,c,h,w]; elements of `esize` bytes, copied bit for bit. */
void or_nchw_to_nhwc(const void *x, void *y, int64_t N, int64_t C, int64_t H, int64_t W,
                     int64_t esize) {
    const unsigned char *src = (const unsigned char *)x;
    unsigned char *dst = (unsigned char *)y;
    for (int64_t n = 0; n < N; ++n)
        for (int64_t c = 0; c < C; ++c)
            for (int64_t h = 0; h < H; ++h)
                for (int64_t w = 0; w < W; ++w)
                    memcpy(dst + (((n * H + h) * W + w) * C + c) * esize,
                           src + (((n * C + c) * H + h) * W + w) * esize, (size_t)esize);
}

/* y[n,c,h,w] = x[n,h,w,c]. */
void or_nhwc_to_nchw(const void *x, void *y, int64_t N, int64_t C, int64_t H, int64_t W,
                     int64_t esize) {
    const unsigned char *src = (const unsigned char *)x;
    unsigned char *dst = (unsigned char *)y;
    for (int64_t n = 0; n < N; ++n)
        for (int64_t c = 0; c < C; ++c)
            for (int64_t h = 0; h < H; ++h)
                for (int64_t w = 0; w < W; ++w)
                    memcpy(dst + (((n * C + c) * H + h) * W + w) * esize,
                           src + (((n * H + h) * W + w) * C + c) * esize, (size_t)esize);
}

/* ------------------------------------------------------------------------ */
/* Optimal routine path by exhaustive enumeration (Def. 1, Def. 2, Eq. 2)     */
/* ------------------------------------------------------------------------ */

static int64_t or_sat_add(int64_t a, int64_t b) {
    if (a == OR_INF || b == OR_INF) return OR_INF;
    return a + b; /* callers keep finite costs far below INT64_MAX/ (layers+edges) */
}

/*
 * F_i(lambda) = min over the routines r of layer i with schema lambda of T(r)
 * (Eq. 1).  cand_schema[j], cand_cost[j] for j in [0, n_cand) describe layer
 * i's routines; out[lambda] receives F_i(lambda) (INT64_MAX if none).
 */
void or_fastest_per_schema(int32_t n_cand, const int32_t *cand_schema, const int64_t *cand_cost,
                           int32_t n_schemas, int64_t *out) {
    for (int32_t l = 0; l < n_schemas; ++l) out[l] = OR_INF;
    for (int32_t j = 0; j < n_cand; ++j) {
        const int32_t l = cand_schema[j];
        if (l < 0 || l >= n_schemas) continue;
        if (cand_cost[j] < out[l]) out[l] = cand_cost[j];
    }
}

/*
 * T(S) for the schema assignment `assign` (one schema per layer):
 *   sum_i F_i(assign[i])  +  sum_{edges (j,i)} F^a_{j,i}(assign[j] -> assign[i]),
 * with F^a = 0 when the two schemas are equal (void adapt).
 * layer_cost: [n_layers][n_schemas]; edges: [n_edges][2] = (src, dst);
 * adapt_cost: [n_edges][n_schemas(from)][n_schemas(to)].
 */
int64_t or_path_cost(int32_t n_layers, int32_t n_schemas, const int64_t *layer_cost,
                     int32_t n_edges, const int32_t *edges, const int64_t *adapt_cost,
                     const int32_t *assign) {
    int64_t t = 0;
    for (int32_t i = 0; i < n_layers; ++i)
        t = or_sat_add(t, layer_cost[(int64_t)i * n_schemas + assign[i]]);
    for (int32_t e = 0; e < n_edges; ++e) {
        const int32_t a = assign[edges[2 * e]], b = assign[edges[2 * e + 1]];
        if (a == b) continue; /* void adapt routine, T = 0 */
        t = or_sat_add(t, adapt_cost[((int64_t)e * n_schemas + a) * n_schemas + b]);
    }
    return t;
}

/*
 * Exhaustive search of S* over every assignment in Lambda^n (Def. 2).
 * Writes the minimising assignment (ties: lexicographically smallest) into
 * best_assign and the number of minimising assignments into *n_min.
 * Returns T(S*), or INT64_MAX when every assignment is infeasible.
 * Enumeration is an n-digit base-|Lambda| counter, layer 0 most significant.
 */
int64_t or_brute_force(int32_t n_layers, int32_t n_schemas, const int64_t *layer_cost,
                       int32_t n_edges, const int32_t *edges, const int64_t *adapt_cost,
                       int32_t *best_assign, int64_t *n_min) {
    int32_t *a = (int32_t *)calloc((size_t)n_layers + 1, sizeof(int32_t));
    int64_t best = OR_INF, count = 0;
    for (int32_t i = 0; i < n_layers; ++i) best_assign[i] = 0;
    for (;;) {
        const int64_t t = or_path_cost(n_layers, n_schemas, layer_cost, n_edges, edges,
                                       adapt_cost, a);
        if (t != OR_INF) {
            if (t < best) {
                best = t;
                count = 1;
                memcpy(best_assign, a, sizeof(int32_t) * (size_t)n_layers);
            } else if (t == best) {
                ++count;
            }
        }
        int32_t i = n_layers - 1; /* next assignment in lexicographic order */
        while (i >= 0 && a[i] == n_schemas - 1) a[i--] = 0;
        if (i < 0) break;
        a[i]++;
    }
    free(a);
    *n_min = count;
    return best;
}
