/*
 * iq_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, CPU definition of what the integer quantized convolution
 * layer of "Training and Inference for Integer-Based Semantic Segmentation
 * Network" (Yang, Deng, Yang, Xie, Li; arXiv 2011.14504) computes, forward
 * and backward.  It exists so that the CUDA library can be checked against
 * it element by element.  Only the test suite, the smoke check and the CPU
 * baseline leg of the benchmark may load it; the product path never does.
 * It shares no code, header or constant table with the CUDA sources.
 *
 * Representation: a quantized tensor is (integer codes q, real scale s) and
 * stands for the real values q*s.  Integer work is exact (int64 / int128);
 * real-valued scale metadata is IEEE fp64 evaluated in the fixed operation
 * order written below (build with -ffp-contract=off so no FMA is formed).
 *
 * Every function names the passage of the paper it follows:
 *   Sec. 3.1.1 Eq. (del), Eq. (UQ)    quantization step and uniform quantizer
 *   Sec. 3.1.1 (constant x2 / x1/2)   for mu, sigma, gamma, beta
 *   Sec. 3.1.2 Eq. (ScaleFactor),(ScaleQ)   scale quantization
 *   Sec. 3.1.3 Eq. (SQ),(SR)          stochastic rounding quantizer RQ
 *   Sec. 3.2.1 Eq. (WQ0),(WQ1)        master / forward weights
 *   Sec. 3.2.2 Eq. (BN2),(BN4),(BN5) and the quantized-BN equation block
 *   Sec. 3.2.3 Eq. (AQ1)              activation quantization
 *   Sec. 3.3.1 Eq. (EQ)               error quantization
 *   Sec. 3.3.2 Eq. (GQ1),(GQ2)        gradient quantization
 *   Sec. 3.3.3 Eq. (UQ2)              update quantization
 * Where the paper is silent the reading taken is stated at the function.
 */
#include <stdint.h>
#include <stddef.h>
#include <math.h>
#include <string.h>
#include <stdlib.h>

typedef __int128 i128;
typedef unsigned __int128 u128;

/* ------------------------------------------------------------------ */
/* scalar helpers                                                      */
/* ------------------------------------------------------------------ */

static int64_t clamp64(int64_t v, int64_t lo, int64_t hi) {
    return v < lo ? lo : (v > hi ? hi : v);
}

/* floor(a / b) for b > 0 */
static i128 floordiv128(i128 a, i128 b) {
    i128 q = a / b;
    if ((a % b) != 0 && a < 0) q -= 1;
    return q;
}

/* Eq. (UQ) rounds with floor(y + 1/2): round half up, ties toward +inf.
 * On an fp64 y this is floor(y) + [y - floor(y) >= 1/2]; y - floor(y) is
 * exact, so no rounding of y + 1/2 can move the result across an integer. */
static double rhu(double y) {
    double f = floor(y);
    return f + ((y - f) >= 0.5 ? 1.0 : 0.0);
}

/* largest code of a k-bit grid: the clip of Eq. (UQ) at 1 - Delta(k) */
static int64_t qmax(int k) { return ((int64_t)1 << (k - 1)) - 1; }

/* rhu of an fp64 value, clipped to a k-bit symmetric grid */
static int64_t code_of(double y, int k) {
    if (y != y) return 0;                               /* NaN -> 0 */
    double lim = (double)qmax(k);
    double r = rhu(y);
    if (r > lim) r = lim;
    if (r < -lim) r = -lim;
    return (int64_t)r;
}

/* ------------------------------------------------------------------ */
/* Sec. 3.1.1: uniform quantizer on real (fp32) inputs                 */
/* ------------------------------------------------------------------ */

/* UQ(x,k) = Clip(Delta*floor(x/Delta + 1/2), -1+Delta, 1-Delta), Eq. (UQ),
 * Delta = 2^(1-k), Eq. (del).  Output: codes c with UQ(x,k) = c * 2^(1-k).
 * x/Delta = x * 2^(k-1) is exact in fp64 for every fp32 x. */
void or_uq_f32(const float* x, int64_t n, int k, int32_t* code) {
    for (int64_t i = 0; i < n; i++)
        code[i] = (int32_t)code_of(ldexp((double)x[i], k - 1), k);
}

/* 2*UQ(x/2, k): the constant x2 / x1/2 scaling used for mu, sigma, gamma,
 * beta (Sec. 3.1.1 and the quantized-BN equation block).  Codes c with
 * value c * 2^(2-k). */
void or_uq2_f32(const float* x, int64_t n, int k, int32_t* code) {
    for (int64_t i = 0; i < n; i++)
        code[i] = (int32_t)code_of(ldexp((double)x[i], k - 2), k);
}

/* SQ(x,k) = Scale(x) * UQ(x / Scale(x), k), Scale(x) = max|x|
 * (Eqs. (ScaleFactor),(ScaleQ)); Scale is taken over the whole tensor.
 * The quotient x/S of two fp32 numbers is formed in fp64; the result of
 * rhu on it equals rhu of the exact real quotient (see DESIGN notes).
 * Returns the output scale S * 2^(1-k); S == 0 gives all-zero codes and
 * scale 2^(1-k). */
double or_sq_f32(const float* x, int64_t n, int k, int32_t* code) {
    float S = 0.0f;
    for (int64_t i = 0; i < n; i++) {
        float a = fabsf(x[i]);
        if (a > S) S = a;
    }
    if (S == 0.0f) {
        for (int64_t i = 0; i < n; i++) code[i] = 0;
        return ldexp(1.0, 1 - k);
    }
    for (int64_t i = 0; i < n; i++) {
        double t = (double)x[i] / (double)S;
        code[i] = (int32_t)code_of(ldexp(t, k - 1), k);
    }
    return ldexp((double)S, 1 - k);
}

/* ------------------------------------------------------------------ */
/* Sec. 3.1.2: scale quantization of an integer-coded tensor            */
/* ------------------------------------------------------------------ */

/* SQ_k of a tensor given as integer codes q with real scale s.
 * With M = max|q|:  x / Scale(x) = q / M, so
 *   code = Clip(floor(q * 2^(k-1) / M + 1/2)) = Clip(floor((2^k q + M) / (2M)))
 * in exact integer arithmetic, and the output scale is
 *   Scale(x) * Delta = (s * M) * 2^(1-k).
 * relu != 0 applies ReLU first (q -> max(q, 0)), i.e. SQ(ReLU(x)).
 * M == 0 gives all-zero codes and scale s * 2^(1-k). */
double or_sq_int64(const int64_t* q, int64_t n, double s, int k, int relu,
                   int32_t* code) {
    int64_t M = 0;
    for (int64_t i = 0; i < n; i++) {
        int64_t v = q[i];
        if (relu && v < 0) v = 0;
        int64_t a = v < 0 ? -v : v;
        if (a > M) M = a;
    }
    if (M == 0) {
        for (int64_t i = 0; i < n; i++) code[i] = 0;
        return ldexp(s, 1 - k);
    }
    for (int64_t i = 0; i < n; i++) {
        int64_t v = q[i];
        if (relu && v < 0) v = 0;
        i128 num = ((i128)v << k) + M;
        i128 c = floordiv128(num, (i128)2 * M);
        code[i] = (int32_t)clamp64((int64_t)c, -qmax(k), qmax(k));
    }
    return ldexp(s * (double)M, 1 - k);
}

double or_sq_int32(const int32_t* q, int64_t n, double s, int k, int relu,
                   int32_t* code) {
    int64_t* t = (int64_t*)malloc(sizeof(int64_t) * (size_t)(n > 0 ? n : 1));
    for (int64_t i = 0; i < n; i++) t[i] = q[i];
    double r = or_sq_int64(t, n, s, k, relu, code);
    free(t);
    return r;
}

/* Eqs. (ScaleFactor),(ScaleQ) with Scale(x) taken per channel (the per-channel reading of
 * Scale): element (o, c, i) of q sits at (o C + c) inner + i; M_c = max over o and i of |q|
 * (of ReLU(q) when relu); code = clip(floor((2^k q + M_c) / (2 M_c))) = floor(2^(k-1) q / M_c
 * + 1/2) clipped to +-(2^(k-1) - 1); scale_c = s M_c 2^(1-k) (s 2^(1-k) when M_c = 0, codes 0). */
void or_sq_per_channel(const int64_t* q, int64_t outer, int64_t C, int64_t inner, double s,
                       int k, int relu, int32_t* code, double* scale) {
    for (int64_t c = 0; c < C; c++) {
        int64_t M = 0;
        for (int64_t o = 0; o < outer; o++)
            for (int64_t i = 0; i < inner; i++) {
                int64_t v = q[(o * C + c) * inner + i];
                if (relu && v < 0) v = 0;
                int64_t a = v < 0 ? -v : v;
                if (a > M) M = a;
            }
        scale[c] = M ? ldexp(s * (double)M, 1 - k) : ldexp(s, 1 - k);
        for (int64_t o = 0; o < outer; o++)
            for (int64_t i = 0; i < inner; i++) {
                const int64_t at = (o * C + c) * inner + i;
                int64_t v = q[at];
                if (relu && v < 0) v = 0;
                if (!M) {
                    code[at] = 0;
                    continue;
                }
                i128 num = ((i128)v << k) + M;
                code[at] = (int32_t)clamp64((int64_t)floordiv128(num, (i128)2 * M), -qmax(k),
                                            qmax(k));
            }
    }
}

/* ------------------------------------------------------------------ */
/* Sec. 3.1.3: stochastic rounding with a counter-based generator       */
/* ------------------------------------------------------------------ */

/* Philox4x64 with 10 rounds (Salmon, Moraes, Dror, Shaw, "Parallel random
 * numbers: as easy as 1, 2, 3", SC'11).  One round maps (x0,x1,x2,x3) with
 * key (k0,k1) to (hi(M1*x2)^x1^k0, lo(M1*x2), hi(M0*x0)^x3^k1, lo(M0*x0));
 * the key is advanced by the Weyl constants between rounds. */
void or_philox4x64_10(const uint64_t ctr[4], const uint64_t key[2],
                      uint64_t out[4]) {
    const uint64_t M0 = 0xD2E7470EE14C6C93ULL, M1 = 0xCA5A826395121157ULL;
    const uint64_t W0 = 0x9E3779B97F4A7C15ULL, W1 = 0xBB67AE8584CAA73BULL;
    uint64_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
    uint64_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; r++) {
        u128 p0 = (u128)M0 * x0;
        u128 p1 = (u128)M1 * x2;
        uint64_t y0 = (uint64_t)(p1 >> 64) ^ x1 ^ k0;
        uint64_t y1 = (uint64_t)p1;
        uint64_t y2 = (uint64_t)(p0 >> 64) ^ x3 ^ k1;
        uint64_t y3 = (uint64_t)p0;
        x0 = y0; x1 = y1; x2 = y2; x3 = y3;
        k0 += W0; k1 += W1;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* The 32-bit uniform word used for element i of a stochastically rounded
 * tensor: Philox4x64-10 with key (seed, layer) and counter (i/8, step, tag, 0);
 * element i takes 32-bit half (i mod 2) of 64-bit word ((i/2) mod 4). */
uint32_t or_rq_uniform(uint64_t seed, uint64_t layer, uint64_t step,
                       uint64_t tag, uint64_t i) {
    uint64_t ctr[4] = { i >> 3, step, tag, 0 };
    uint64_t key[2] = { seed, layer };
    uint64_t o[4];
    or_philox4x64_10(ctr, key, o);
    uint64_t w = o[(i >> 1) & 3];
    return (uint32_t)((i & 1) ? (w >> 32) : (w & 0xffffffffULL));
}

/* RQ(x,k) = Clip(Delta*Round(x/Delta)), Round stochastic with
 * P(up) = x - floor(x) (Eqs. (SQ),(SR)), applied to x = G / Scale(G)
 * as in Eqs. (GQ1),(GQ2).  With M = max|q|, y = q * 2^(k-1) / M:
 *   f = floor(y), rem = q*2^(k-1) - f*M in [0, M),
 *   round up iff u * M < rem * 2^32   (u the element's 32-bit uniform),
 * so P(up) = ceil(rem*2^32/M) / 2^32 = rem/M to within 2^-32.
 * gq_mode 1 = Eq. (GQ1) (magnitude kept): scale (s*M)*2^(1-k);
 * gq_mode 2 = Eq. (GQ2) (magnitude dropped): scale 2^(1-k).
 * M == 0 gives zero codes. */
double or_rq_int64(const int64_t* q, int64_t n, double s, int k, int gq_mode,
                   uint64_t seed, uint64_t layer, uint64_t step, uint64_t tag,
                   int32_t* code) {
    int64_t M = 0;
    for (int64_t i = 0; i < n; i++) {
        int64_t a = q[i] < 0 ? -q[i] : q[i];
        if (a > M) M = a;
    }
    if (M == 0) {
        for (int64_t i = 0; i < n; i++) code[i] = 0;
        return gq_mode == 1 ? ldexp(s, 1 - k) : ldexp(1.0, 1 - k);
    }
    for (int64_t i = 0; i < n; i++) {
        i128 num = (i128)q[i] << (k - 1);
        i128 f = floordiv128(num, (i128)M);
        i128 rem = num - f * M;
        uint32_t u = or_rq_uniform(seed, layer, step, tag, (uint64_t)i);
        int up = ((u128)u * (u128)M) < ((u128)rem << 32);
        code[i] = (int32_t)clamp64((int64_t)(f + up), -qmax(k), qmax(k));
    }
    return gq_mode == 1 ? ldexp(s * (double)M, 1 - k) : ldexp(1.0, 1 - k);
}

/* Eq. (ScaleQ) and Eqs. (SQ),(SR) for selected elements of a tensor whose
 * max |q| (after ReLU for SQ of ReLU) is M: the codes that or_sq_int64 and
 * or_rq_int64 give at those elements, and the output scale.  idx[j] is the
 * flat index of element q[j] in its tensor (the stochastic rounding's
 * counter).  For checking a large tensor at sampled positions. */
double or_sq_at(const int64_t* q, int64_t m, int64_t M, double s, int k, int relu,
                int32_t* code) {
    if (M == 0) {
        for (int64_t j = 0; j < m; j++) code[j] = 0;
        return ldexp(s, 1 - k);
    }
    for (int64_t j = 0; j < m; j++) {
        int64_t v = q[j];
        if (relu && v < 0) v = 0;
        i128 c = floordiv128(((i128)v << k) + M, (i128)2 * M);
        code[j] = (int32_t)clamp64((int64_t)c, -qmax(k), qmax(k));
    }
    return ldexp(s * (double)M, 1 - k);
}

double or_rq_at(const int64_t* q, const int64_t* idx, int64_t m, int64_t M, double s,
                int k, int gq_mode, uint64_t seed, uint64_t layer, uint64_t step,
                uint64_t tag, int32_t* code) {
    if (M == 0) {
        for (int64_t j = 0; j < m; j++) code[j] = 0;
        return gq_mode == 1 ? ldexp(s, 1 - k) : ldexp(1.0, 1 - k);
    }
    for (int64_t j = 0; j < m; j++) {
        i128 num = (i128)q[j] << (k - 1);
        i128 f = floordiv128(num, (i128)M);
        i128 rem = num - f * M;
        uint32_t u = or_rq_uniform(seed, layer, step, tag, (uint64_t)idx[j]);
        int up = ((u128)u * (u128)M) < ((u128)rem << 32);
        code[j] = (int32_t)clamp64((int64_t)(f + up), -qmax(k), qmax(k));
    }
    return gq_mode == 1 ? ldexp(s * (double)M, 1 - k) : ldexp(1.0, 1 - k);
}

/* ------------------------------------------------------------------ */
/* Sec. 3.2.1: weights                                                 */
/* ------------------------------------------------------------------ */

/* W_q = UQ(W_m, k_W), Eq. (WQ1), where the master weights W_m sit on the
 * k_U grid (Eq. (WQ0)) as codes m (value m * 2^(1-k_U)).  Then
 * W_m / Delta(k_W) = m / 2^(k_U - k_W) and floor(that + 1/2) is an exact
 * arithmetic shift.  The same map serves the x2-scaled gamma/beta masters
 * (both grids carry the same factor 2). */
void or_requant_master(const int32_t* m, int64_t n, int k_u, int k_w,
                       int32_t* wq) {
    int sh = k_u - k_w;
    for (int64_t i = 0; i < n; i++) {
        i128 v = (i128)m[i] + ((i128)1 << (sh - 1));
        i128 c = floordiv128(v, (i128)1 << sh);
        wq[i] = (int32_t)clamp64((int64_t)c, -qmax(k_w), qmax(k_w));
    }
}

/* ------------------------------------------------------------------ */
/* Convolution: the MAC of Sec. 3.2.3 on 8-bit W and A (Fig. 4)         */
/* ------------------------------------------------------------------ */

/* Geometry.  x: NHWC [n][h][w][c]; weights KRSC [k][r][s][c/groups];
 * output NPQK [n][p][q][k].  Output pixel (p,q) with tap (r,s) reads input
 * row p*stride_h + r*dil_h - pad_h, column q*stride_w + s*dil_w - pad_w;
 * outside the image the input is zero.  Group g owns input channels
 * [g*C/G, (g+1)*C/G) and output channels [g*K/G, (g+1)*K/G). */
typedef struct {
    int32_t n, h, w, c, k, r, s;
    int32_t stride_h, stride_w, pad_h, pad_w, dil_h, dil_w, groups;
    int32_t p, q;
} or_conv;

void or_conv_out_size(or_conv* d) {
    d->p = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    d->q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
}

#define X_AT(n_, h_, w_, c_) x[(((int64_t)(n_) * d->h + (h_)) * d->w + (w_)) * d->c + (c_)]
#define W_AT(k_, r_, s_, c_) wt[(((int64_t)(k_) * d->r + (r_)) * d->s + (s_)) * cg + (c_)]
#define Y_AT(n_, p_, q_, k_) ((((int64_t)(n_) * d->p + (p_)) * d->q + (q_)) * d->k + (k_))

/* forward: acc[n,p,q,k] = sum_{r,s,c in group} x[...] * w[k,r,s,c] */
void or_conv_fwd(const or_conv* d, const int8_t* x, const int8_t* wt,
                 int32_t* acc) {
    const int cg = d->c / d->groups, kg = d->k / d->groups;
    #pragma omp parallel for collapse(2) schedule(static)
    for (int n = 0; n < d->n; n++)
        for (int p = 0; p < d->p; p++)
            for (int q = 0; q < d->q; q++)
                for (int k = 0; k < d->k; k++) {
                    int g = k / kg;
                    int64_t sum = 0;
                    for (int r = 0; r < d->r; r++) {
                        int hh = p * d->stride_h + r * d->dil_h - d->pad_h;
                        if (hh < 0 || hh >= d->h) continue;
                        for (int s = 0; s < d->s; s++) {
                            int ww = q * d->stride_w + s * d->dil_w - d->pad_w;
                            if (ww < 0 || ww >= d->w) continue;
                            for (int c = 0; c < cg; c++)
                                sum += (int64_t)X_AT(n, hh, ww, g * cg + c) *
                                       (int64_t)W_AT(k, r, s, c);
                        }
                    }
                    acc[Y_AT(n, p, q, k)] = (int32_t)sum;
                }
}

/* data gradient: the adjoint of the forward map,
 * dx[n,h,w,c] = sum over (p,q,k,r,s) with h = p*sh + r*dh - ph,
 * w = q*sw + s*dw - pw of e[n,p,q,k] * w[k,r,s,c].  Scattered image by
 * image (integer sums, so the order is immaterial); int64 result, since the
 * reduction over k, r, s can exceed 2^31 (fc6: 4096 * 49 products). */
void or_conv_dgrad(const or_conv* d, const int8_t* e, const int8_t* wt,
                   int64_t* dx) {
    const int cg = d->c / d->groups, kg = d->k / d->groups;
    const int64_t img = (int64_t)d->h * d->w * d->c;
    #pragma omp parallel for schedule(static)
    for (int n = 0; n < d->n; n++) {
        int64_t* t = (int64_t*)calloc((size_t)img, sizeof(int64_t));
        for (int p = 0; p < d->p; p++)
            for (int q = 0; q < d->q; q++)
                for (int k = 0; k < d->k; k++) {
                    int64_t ev = e[Y_AT(n, p, q, k)];
                    if (ev == 0) continue;
                    int g = k / kg;
                    for (int r = 0; r < d->r; r++) {
                        int hh = p * d->stride_h + r * d->dil_h - d->pad_h;
                        if (hh < 0 || hh >= d->h) continue;
                        for (int s = 0; s < d->s; s++) {
                            int ww = q * d->stride_w + s * d->dil_w - d->pad_w;
                            if (ww < 0 || ww >= d->w) continue;
                            for (int c = 0; c < cg; c++)
                                t[((int64_t)hh * d->w + ww) * d->c + g * cg + c] +=
                                    ev * (int64_t)W_AT(k, r, s, c);
                        }
                    }
                }
        for (int64_t i = 0; i < img; i++) dx[n * img + i] = t[i];
        free(t);
    }
}

/* weight gradient: g[k,r,s,c] = sum_{n,p,q} e[n,p,q,k] * x[n, h, w, c_g]
 * with h, w as in the forward map; int64 accumulation (the sum runs over
 * N*P*Q products and exceeds 2^31 at segmentation sizes). */
void or_conv_wgrad(const or_conv* d, const int8_t* e, const int8_t* x,
                   int64_t* gw) {
    const int cg = d->c / d->groups, kg = d->k / d->groups;
    #pragma omp parallel for schedule(static)
    for (int k = 0; k < d->k; k++) {
        int g = k / kg;
        for (int r = 0; r < d->r; r++)
            for (int s = 0; s < d->s; s++)
                for (int c = 0; c < cg; c++) {
                    int64_t sum = 0;
                    for (int n = 0; n < d->n; n++)
                        for (int p = 0; p < d->p; p++) {
                            int hh = p * d->stride_h + r * d->dil_h - d->pad_h;
                            if (hh < 0 || hh >= d->h) continue;
                            for (int q = 0; q < d->q; q++) {
                                int ww = q * d->stride_w + s * d->dil_w - d->pad_w;
                                if (ww < 0 || ww >= d->w) continue;
                                sum += (int64_t)e[Y_AT(n, p, q, k)] *
                                       (int64_t)X_AT(n, hh, ww, g * cg + c);
                            }
                        }
                    gw[(((int64_t)k * d->r + r) * d->s + s) * cg + c] = sum;
                }
    }
}

/* Selected outputs of the three convolutions, one at a time: out[j] is the
 * sum that or_conv_fwd / or_conv_dgrad / or_conv_wgrad would store at the
 * flat output index idx[j] (NPQK, NHWC and KRSC order respectively), written
 * out from the same definitions.  They let a tensor too large for the full
 * loops be checked at sampled positions. */
void or_conv_fwd_at(const or_conv* d, const int8_t* x, const int8_t* wt,
                    const int64_t* idx, int64_t m, int64_t* out) {
    const int cg = d->c / d->groups, kg = d->k / d->groups;
    #pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < m; j++) {
        int64_t t = idx[j];
        int k = (int)(t % d->k); t /= d->k;
        int q = (int)(t % d->q); t /= d->q;
        int p = (int)(t % d->p);
        int n = (int)(t / d->p);
        int g = k / kg;
        int64_t sum = 0;
        for (int r = 0; r < d->r; r++) {
            int hh = p * d->stride_h + r * d->dil_h - d->pad_h;
            if (hh < 0 || hh >= d->h) continue;
            for (int s = 0; s < d->s; s++) {
                int ww = q * d->stride_w + s * d->dil_w - d->pad_w;
                if (ww < 0 || ww >= d->w) continue;
                for (int c = 0; c < cg; c++)
                    sum += (int64_t)X_AT(n, hh, ww, g * cg + c) * (int64_t)W_AT(k, r, s, c);
            }
        }
        out[j] = sum;
    }
}

/* dx[n,h,w,c]: every (p, r) with p*sh + r*dh - ph = h and every (q, s) alike,
 * over the output channels k of c's group. */
void or_conv_dgrad_at(const or_conv* d, const int8_t* e, const int8_t* wt,
                      const int64_t* idx, int64_t m, int64_t* out) {
    const int cg = d->c / d->groups, kg = d->k / d->groups;
    #pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < m; j++) {
        int64_t t = idx[j];
        int c = (int)(t % d->c); t /= d->c;
        int w = (int)(t % d->w); t /= d->w;
        int h = (int)(t % d->h);
        int n = (int)(t / d->h);
        int g = c / cg;
        int64_t sum = 0;
        for (int r = 0; r < d->r; r++) {
            int num_p = h + d->pad_h - r * d->dil_h;
            if (num_p < 0 || num_p % d->stride_h) continue;
            int p = num_p / d->stride_h;
            if (p >= d->p) continue;
            for (int s = 0; s < d->s; s++) {
                int num_q = w + d->pad_w - s * d->dil_w;
                if (num_q < 0 || num_q % d->stride_w) continue;
                int q = num_q / d->stride_w;
                if (q >= d->q) continue;
                for (int k = g * kg; k < (g + 1) * kg; k++)
                    sum += (int64_t)e[Y_AT(n, p, q, k)] * (int64_t)W_AT(k, r, s, c - g * cg);
            }
        }
        out[j] = sum;
    }
}

void or_conv_wgrad_at(const or_conv* d, const int8_t* e, const int8_t* x,
                      const int64_t* idx, int64_t m, int64_t* out) {
    const int cg = d->c / d->groups, kg = d->k / d->groups;
    #pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < m; j++) {
        int64_t t = idx[j];
        int c = (int)(t % cg); t /= cg;
        int s = (int)(t % d->s); t /= d->s;
        int r = (int)(t % d->r);
        int k = (int)(t / d->r);
        int g = k / kg;
        int64_t sum = 0;
        for (int n = 0; n < d->n; n++)
            for (int p = 0; p < d->p; p++) {
                int hh = p * d->stride_h + r * d->dil_h - d->pad_h;
                if (hh < 0 || hh >= d->h) continue;
                for (int q = 0; q < d->q; q++) {
                    int ww = q * d->stride_w + s * d->dil_w - d->pad_w;
                    if (ww < 0 || ww >= d->w) continue;
                    sum += (int64_t)e[Y_AT(n, p, q, k)] * (int64_t)X_AT(n, hh, ww, g * cg + c);
                }
            }
        out[j] = sum;
    }
}

/* ------------------------------------------------------------------ */
/* Sec. 3.2.2: quantized L1 batch normalization, forward                */
/* ------------------------------------------------------------------ */

typedef struct {
    int32_t k_mu, k_sigma, k_xhat, k_gamma, k_beta, k_a;
} or_bn_bits;

/* Per-tensor and per-channel values the forward pass produces; the
 * backward pass consumes c_sigma and s_xhat, the rest is for inspection. */
typedef struct {
    double s_xhat;     /* scale of the X codes: M_xhat * 2^(1-k_xhat)      */
    double s_a;        /* scale of the A codes: M_y * 2^(1-k_a)            */
    double m_xhat;     /* max |xhat| over the tensor                        */
    double m_y;        /* max ReLU(y) over the tensor                       */
    int32_t p_x, p_a;  /* fixed-point shifts of the two per-element maps    */
} or_bn_out;

static int frexp_exp(double v) { int e; frexp(v, &e); return e; }

/* One L1BN layer in training (batch statistics) or inference (the same
 * batch statistics; the paper defines no running estimate).  Input: conv
 * accumulators acc[m][C] with real scale s_acc.  Steps, in the paper's order:
 *
 *  Eq. (BN2)  mu_B = (1/m) sum_i x_i,  x_i = acc_i * s_acc
 *  Eq. (BN5)  sigma_B = (1/m) sum_i |x_i - mu_B|        (no square, no root)
 *             evaluated exactly as T = sum_i |m*acc_i - S1| (S1 = sum acc),
 *             sigma_B = T * s_acc / m^2 in fp64.
 *  QBN block  mu_q = 2*UQ(mu_B/2, k_mu), sigma_q = 2*UQ(sigma_B/2, k_sigma)
 *  Eq. (BN4)  xhat_i = (x_i - mu_q) / (sigma_q + eps),  eps = 2^(2-k_sigma),
 *             one step of the sigma_q grid (the paper gives no value).
 *  QBN block  X = SQ(xhat, k_xhat) with Scale = M_xhat = max|xhat|.
 *             Per channel xhat is increasing in acc, so M_xhat is reached at
 *             the channel's largest or smallest accumulator.
 *  QBN block  gamma_q = 2*UQ(gamma/2, k_gamma), beta_q likewise (codes given)
 *             y_i = gamma_q * xhat_q,i + beta_q
 *  Eq. (AQ1)  A = SQ(ReLU(y), k_a) with Scale = M_y = max ReLU(y).
 *
 * Element-wise the two quantizers are evaluated in fixed point, as an
 * integer-only device would: per channel the code of X is
 * rhu(a_c*acc + b_c) for real a_c, b_c, computed as
 *   X = floor((F_c*acc + B_c) / 2^P),  F_c = rhu(a_c 2^P),
 *   B_c = rhu(b_c 2^P) + 2^(P-1),
 * with one shift P per tensor chosen as large as int64 allows; A from X
 * likewise.  All fp64 steps are written out in evaluation order. */
int or_bn_fwd(int64_t m, int32_t C, const int32_t* acc, double s_acc,
              const int32_t* gam, const int32_t* bet, const or_bn_bits* b,
              int16_t* X, int8_t* A, int32_t* c_mu, int32_t* c_sigma,
              int64_t* F, int64_t* Bc, int64_t* G, int64_t* H,
              or_bn_out* out) {
    if (m <= 0 || C <= 0) return -1;
    int64_t* S1 = (int64_t*)calloc((size_t)C, sizeof(int64_t));
    int64_t* hi = (int64_t*)malloc(sizeof(int64_t) * (size_t)C);
    int64_t* lo = (int64_t*)malloc(sizeof(int64_t) * (size_t)C);
    u128* T = (u128*)calloc((size_t)C, sizeof(u128));
    for (int c = 0; c < C; c++) { hi[c] = INT64_MIN; lo[c] = INT64_MAX; }
    /* Eq. (BN2): channel sums and extremes */
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            int64_t v = acc[i * C + c];
            S1[c] += v;
            if (v > hi[c]) hi[c] = v;
            if (v < lo[c]) lo[c] = v;
        }
    /* Eq. (BN5): T = sum |m*acc - S1| exactly */
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            i128 dv = (i128)m * acc[i * C + c] - S1[c];
            T[c] += (u128)(dv < 0 ? -dv : dv);
        }
    const double mu_step = ldexp(1.0, 2 - b->k_mu);       /* grid of mu_q */
    const double sg_step = ldexp(1.0, 2 - b->k_sigma);    /* grid of sigma_q = eps */
    double* den = (double*)malloc(sizeof(double) * (size_t)C);
    double* muq = (double*)malloc(sizeof(double) * (size_t)C);
    const double md = (double)m;
    for (int c = 0; c < C; c++) {
        double mu_b = ((double)S1[c] * s_acc) / md;
        double sg_b = ((double)T[c] * s_acc) / (md * md);
        int64_t cm = code_of(ldexp(mu_b, b->k_mu - 2), b->k_mu);
        int64_t cs = code_of(ldexp(sg_b, b->k_sigma - 2), b->k_sigma);
        c_mu[c] = (int32_t)cm;
        c_sigma[c] = (int32_t)cs;
        muq[c] = (double)cm * mu_step;
        den[c] = (double)(cs + 1) * sg_step;              /* sigma_q + eps */
    }
    /* M_xhat from the channel extremes */
    double mx = 0.0, vmax = 0.0;
    for (int c = 0; c < C; c++) {
        double xh = ((double)hi[c] * s_acc - muq[c]) / den[c];
        double xl = ((double)lo[c] * s_acc - muq[c]) / den[c];
        if (fabs(xh) > mx) mx = fabs(xh);
        if (fabs(xl) > mx) mx = fabs(xl);
        double av = fabs((double)hi[c]) > fabs((double)lo[c]) ? fabs((double)hi[c]) : fabs((double)lo[c]);
        if (av > vmax) vmax = av;
    }
    out->m_xhat = mx;
    out->s_xhat = mx > 0.0 ? ldexp(mx, 1 - b->k_xhat) : ldexp(1.0, 1 - b->k_xhat);
    const int64_t xq = qmax(b->k_xhat);
    /* fixed-point map acc -> X */
    int px = 0;
    if (mx > 0.0) {
        const double qx = ldexp(1.0, b->k_xhat - 1) / mx;
        double lmax = 0.0;
        for (int c = 0; c < C; c++) {
            double a = (s_acc / den[c]) * qx;
            double bb = (-muq[c] / den[c]) * qx;
            double l = fabs(a) * vmax + fabs(bb);
            if (l > lmax) lmax = l;
        }
        px = 62 - frexp_exp(lmax + 1.0);
        if (px > 62) px = 62;
        if (px < 1) { px = 1; }
        for (int c = 0; c < C; c++) {
            double a = (s_acc / den[c]) * qx;
            double bb = (-muq[c] / den[c]) * qx;
            F[c] = (int64_t)rhu(ldexp(a, px));
            Bc[c] = (int64_t)rhu(ldexp(bb, px)) + ((int64_t)1 << (px - 1));
        }
    } else {
        px = 1;
        for (int c = 0; c < C; c++) { F[c] = 0; Bc[c] = 0; }
    }
    out->p_x = px;
    /* X at the channel extremes (X is nondecreasing in acc: F_c >= 0) */
    const double gstep = ldexp(1.0, 2 - b->k_gamma), bstep = ldexp(1.0, 2 - b->k_beta);
    double my = 0.0;
    for (int c = 0; c < C; c++) {
        int64_t xs[2] = { hi[c], lo[c] };
        for (int j = 0; j < 2; j++) {
            i128 t = (i128)F[c] * xs[j] + Bc[c];
            int64_t xc = clamp64((int64_t)(t >> px), -xq, xq);
            double t1 = ((double)gam[c] * gstep) * out->s_xhat;
            double y = t1 * (double)xc + (double)bet[c] * bstep;
            if (y > my) my = y;
        }
    }
    out->m_y = my;
    out->s_a = my > 0.0 ? ldexp(my, 1 - b->k_a) : ldexp(1.0, 1 - b->k_a);
    const int64_t aq = qmax(b->k_a);
    int pa = 1;
    if (my > 0.0) {
        const double qa = ldexp(1.0, b->k_a - 1) / my;
        double lmax = 0.0;
        for (int c = 0; c < C; c++) {
            double t1 = ((double)gam[c] * gstep) * out->s_xhat;
            double l = fabs(t1 * qa) * (double)xq + fabs(((double)bet[c] * bstep) * qa);
            if (l > lmax) lmax = l;
        }
        pa = 62 - frexp_exp(lmax + 1.0);
        if (pa > 62) pa = 62;
        if (pa < 1) pa = 1;
        for (int c = 0; c < C; c++) {
            double t1 = ((double)gam[c] * gstep) * out->s_xhat;
            G[c] = (int64_t)rhu(ldexp(t1 * qa, pa));
            H[c] = (int64_t)rhu(ldexp(((double)bet[c] * bstep) * qa, pa)) + ((int64_t)1 << (pa - 1));
        }
    } else {
        for (int c = 0; c < C; c++) { G[c] = 0; H[c] = 0; }
    }
    out->p_a = pa;
    /* element-wise: X = Q_xhat(xhat), A = Q_A(ReLU(gamma_q xhat_q + beta_q)) */
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            i128 t = (i128)F[c] * acc[i * C + c] + Bc[c];
            int64_t xc = clamp64((int64_t)(t >> px), -xq, xq);
            if (X) X[i * C + c] = (int16_t)xc;
            i128 u = (i128)G[c] * xc + H[c];
            A[i * C + c] = (int8_t)clamp64((int64_t)(u >> pa), 0, aq);
        }
    free(S1); free(hi); free(lo); free(T); free(den); free(muq);
    return 0;
}

/* The element maps of the L1BN forward with constants fixed by an earlier
 * call (F, B, G, H per channel and the shifts px, pa that or_bn_fwd returns
 * for a calibration batch): the inference mode with frozen statistics, a
 * reading of the paper's L1BN at inference (it defines no running estimate).
 * X = clip(floor((F acc + B) / 2^px)), A = clip(floor((G X + H) / 2^pa), 0,
 * 2^(k_a-1)-1), the products in 128 bits (an accumulator beyond the
 * calibration range cannot overflow them). */
void or_bn_apply_fixed(int64_t m, int32_t C, const int32_t* acc, const int64_t* F,
                       const int64_t* B, const int64_t* G, const int64_t* H, int px,
                       int pa, int k_xhat, int k_a, int16_t* X, int8_t* A) {
    const int64_t xq = qmax(k_xhat), aq = qmax(k_a);
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            i128 t = (i128)F[c] * acc[i * C + c] + B[c];
            i128 xs = t >> px;
            int64_t xc = xs < -xq ? -xq : (xs > xq ? xq : (int64_t)xs);
            if (X) X[i * C + c] = (int16_t)xc;
            i128 u = (i128)G[c] * xc + H[c];
            i128 as = u >> pa;
            A[i * C + c] = (int8_t)(as < 0 ? 0 : (as > aq ? aq : (int64_t)as));
        }
}

/* ------------------------------------------------------------------ */
/* Sec. 3.3: backward through ReLU and quantized L1BN                   */
/* ------------------------------------------------------------------ */

/* Input: the error of this layer's activation e_A (codes, scale s_e; it is
 * E_1 of Eq. (EQ) coming from the next layer), the forward outputs A and X,
 * the gamma codes and the sigma_q codes.  Steps:
 *   ReLU:   e_y,i = e_A,i if A_i > 0 else 0 (the mask of the stored A).
 *   d beta_c = s_e * sum e_y;  d gamma_c = s_e * s_X * sum e_y * X
 *            (returned as the integer sums; their scales are s_e, s_e*s_X).
 *   E_2 = Q_E(gamma_q * e_y, k_E2), Eq. (EQ): SQ of z_i = e_y,i * g_c.
 *   L1BN backward (derived from Eqs. (BN4),(BN5); the paper prints none):
 *     d x_i = (1/(sigma_q+eps)) [ g_i - mean(g) - mean(g xhat) (sgn_i - mean(sgn)) ]
 *     with g = E_2 (real), xhat = X * s_X, sgn_i = sign(X_i); means over the
 *     channel's m elements, straight-through for the mu/sigma quantizers.
 *   E_conv = Q_E(d x, k_E) (SQ8), the error the conv's dgrad/wgrad consume.
 * Per element the last step is one fixed-point affine map of (E_2, sgn). */
int or_bn_bwd(int64_t m, int32_t C, const int8_t* eA, double s_e,
              const int8_t* A, const int16_t* X, double s_x,
              const int32_t* gam, const int32_t* c_sigma, int k_sigma,
              int k_gamma, int k_e2, int k_e, int8_t* E, double* s_out,
              int64_t* dgam, int64_t* dbet) {
    if (m <= 0 || C <= 0) return -1;
    /* ReLU mask and gamma/beta gradient sums */
    int64_t M2 = 0;
    for (int c = 0; c < C; c++) { dgam[c] = 0; dbet[c] = 0; }
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            int64_t ey = A[i * C + c] > 0 ? eA[i * C + c] : 0;
            dbet[c] += ey;
            dgam[c] += ey * (int64_t)X[i * C + c];
            int64_t z = ey * (int64_t)gam[c];
            if (z < 0) z = -z;
            if (z > M2) M2 = z;
        }
    /* E_2 = SQ_{k_e2}(gamma_q e_y) */
    const double s_z = s_e * ldexp(1.0, 2 - k_gamma);
    const double s_e2 = M2 > 0 ? ldexp(s_z * (double)M2, 1 - k_e2) : ldexp(s_z, 1 - k_e2);
    int32_t* E2 = (int32_t*)malloc(sizeof(int32_t) * (size_t)(m * C));
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            int64_t ey = A[i * C + c] > 0 ? eA[i * C + c] : 0;
            int64_t z = ey * (int64_t)gam[c];
            if (M2 == 0) { E2[i * C + c] = 0; continue; }
            i128 q = floordiv128(((i128)z << k_e2) + M2, (i128)2 * M2);
            E2[i * C + c] = (int32_t)clamp64((int64_t)q, -qmax(k_e2), qmax(k_e2));
        }
    /* channel means of E_2, E_2*X and sign(X) as exact integer sums */
    int64_t* SE = (int64_t*)calloc((size_t)C, sizeof(int64_t));
    int64_t* SEX = (int64_t*)calloc((size_t)C, sizeof(int64_t));
    int64_t* SS = (int64_t*)calloc((size_t)C, sizeof(int64_t));
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            int64_t e2 = E2[i * C + c];
            int64_t xv = X[i * C + c];
            SE[c] += e2;
            SEX[c] += e2 * xv;
            SS[c] += (xv > 0) - (xv < 0);
        }
    /* per channel: d x_i = w_c * (E2_i + kap_c * sgn_i + lam_c) */
    double* w = (double*)malloc(sizeof(double) * (size_t)C);
    double* kap = (double*)malloc(sizeof(double) * (size_t)C);
    double* lam = (double*)malloc(sizeof(double) * (size_t)C);
    const double md = (double)m;
    const double sg_step = ldexp(1.0, 2 - k_sigma);
    for (int c = 0; c < C; c++) {
        double gx = ((double)SEX[c] * s_x) / md;           /* mean(g xhat) / s_e2 */
        kap[c] = -gx;
        lam[c] = gx * ((double)SS[c] / md) - (double)SE[c] / md;
        w[c] = s_e2 / ((double)(c_sigma[c] + 1) * sg_step);
    }
    /* Scale of d x: the largest |d x_i| over the tensor */
    double M = 0.0;
    for (int64_t i = 0; i < m; i++)
        for (int c = 0; c < C; c++) {
            int64_t xv = X[i * C + c];
            double sg = (double)((xv > 0) - (xv < 0));
            double dx = w[c] * (((double)E2[i * C + c] + kap[c] * sg) + lam[c]);
            if (fabs(dx) > M) M = fabs(dx);
        }
    const int64_t eq = qmax(k_e);
    if (M == 0.0) {
        for (int64_t i = 0; i < m * C; i++) E[i] = 0;
        *s_out = ldexp(1.0, 1 - k_e);
    } else {
        const double qe = ldexp(1.0, k_e - 1) / M;
        const double emax = (double)qmax(k_e2);
        double lmax = 0.0;
        for (int c = 0; c < C; c++) {
            double om = w[c] * qe;
            double l = fabs(om) * emax + fabs(om * kap[c]) + fabs(om * lam[c]);
            if (l > lmax) lmax = l;
        }
        int pe = 62 - frexp_exp(lmax + 1.0);
        if (pe > 62) pe = 62;
        if (pe < 1) pe = 1;
        for (int c = 0; c < C; c++) {
            double om = w[c] * qe;
            int64_t fw = (int64_t)rhu(ldexp(om, pe));
            int64_t fk = (int64_t)rhu(ldexp(om * kap[c], pe));
            int64_t fl = (int64_t)rhu(ldexp(om * lam[c], pe)) + ((int64_t)1 << (pe - 1));
            for (int64_t i = 0; i < m; i++) {
                int64_t xv = X[i * C + c];
                int64_t sg = (xv > 0) - (xv < 0);
                i128 t = (i128)fw * E2[i * C + c] + (i128)fk * sg + fl;
                E[i * C + c] = (int8_t)clamp64((int64_t)(t >> pe), -eq, eq);
            }
        }
        *s_out = ldexp(M, 1 - k_e);
    }
    free(E2); free(SE); free(SEX); free(SS); free(w); free(kap); free(lam);
    return 0;
}

/* ReLU backward for layers without BN: e_acc = e_A where A > 0 (same
 * codes, same scale). */
void or_relu_bwd(int64_t n, const int8_t* eA, const int8_t* A, int8_t* e) {
    for (int64_t i = 0; i < n; i++) e[i] = A[i] > 0 ? eA[i] : 0;
}

/* ------------------------------------------------------------------ */
/* Sec. 3.3.3: update                                                  */
/* ------------------------------------------------------------------ */

/* Delta W = Q_U(G_q, k_U) = UQ(G_q * lr, k_U), Eq. (UQ2), with G_q given as
 * codes c and scale s_g, lr = 2^(-lr_log2) (a power of two, halved
 * discretely as the paper's schedule does).  The master codes m live on the
 * k_U grid (value m * 2^(1-k_U), or m * 2^(2-k_U) for the x2-scaled
 * gamma/beta masters, x2 != 0).  Plain SGD: m <- Clip(m - dW).
 * Then the forward copy is regenerated: w_q = UQ(W_m, k_W), Eq. (WQ1). */
void or_update(int64_t n, int32_t* master, int32_t* wq, const int32_t* gc,
               double s_g, int lr_log2, int k_u, int k_w, int x2) {
    const int sh = (x2 ? k_u - 2 : k_u - 1) - lr_log2;
    for (int64_t i = 0; i < n; i++) {
        double t = (double)gc[i] * s_g;
        int64_t du = code_of(ldexp(t, sh), k_u);
        int64_t nm = clamp64((int64_t)master[i] - du, -qmax(k_u), qmax(k_u));
        master[i] = (int32_t)nm;
    }
    or_requant_master(master, n, k_u, k_w, wq);
}

/* L2 weight decay (Sec. 5.1 states its coefficient, not its quantized form), read as a
 * decoupled shrink of the k_u-grid master codes after each update: with the decay step
 * lambda lr = 2^-shift, m <- m - floor(m / 2^shift + 1/2) (round half up, on the master
 * grid), then W_q = UQ(W_m, k_w) regenerated (Eq. (WQ1)).  shift >= 1. */
void or_weight_decay(int64_t n, int32_t* master, int32_t* wq, int shift, int k_u, int k_w) {
    for (int64_t i = 0; i < n; i++) {
        const int64_t m = master[i];
        const int64_t d = (int64_t)floordiv128((i128)m + ((i128)1 << (shift - 1)),
                                               (i128)1 << shift);
        master[i] = (int32_t)(m - d);
    }
    or_requant_master(master, n, k_u, k_w, wq);
}

/* Correctly rounded conversion of a 128-bit unsigned integer to fp64 (the
 * conversion the sigma_B step applies to T); exposed for its test. */
double or_u128_to_double(uint64_t hi, uint64_t lo) {
    u128 v = ((u128)hi << 64) | lo;
    return (double)v;
}

/* Network input (Sec. 5 feeds images to the first conv; Eq. (AQ1)): the real
 * pixel value p/255 quantized with SQ(., 8).  Scale = P/255 with P the largest
 * pixel, so x/Scale = p/P and code = floor((256 p + P) / (2P)), clipped at 127;
 * output scale (P/255) * 2^-7.  Input uint8 NHWC with c channels, output int8
 * NHWC with c_out >= c channels (the extra channels zero). */
double or_quantize_image_u8(const uint8_t* img, int64_t npix, int c, int c_out,
                            int8_t* out) {
    int64_t P = 0;
    for (int64_t i = 0; i < npix * c; i++) if (img[i] > P) P = img[i];
    for (int64_t p = 0; p < npix; p++)
        for (int j = 0; j < c_out; j++) {
            int64_t v = 0;
            if (j < c && P > 0) {
                v = (256 * (int64_t)img[p * c + j] + P) / (2 * P);
                if (v > 127) v = 127;
            }
            out[p * c_out + j] = (int8_t)v;
        }
    return P > 0 ? ldexp((double)P / 255.0, -7) : ldexp(1.0, -7);
}

/* ------------------------------------------------------------------ */
/* Network glue of the FCN-VGG16 path (Sec. 2.1, Sec. 5)                */
/* ------------------------------------------------------------------ */

/* Max pooling on codes (the scale is positive, so the max of the codes is the
 * code of the max).  Window k x k, stride s, zero-size padding p counted as
 * -infinity.  The position of the first maximum in (r, s) scan order is kept
 * for the backward pass (tap index r*k + s; 255 when the window is empty). */
void or_maxpool_fwd(const int8_t* x, int n, int h, int w, int c, int k, int s, int p,
                    int8_t* y, uint8_t* arg, int* ph, int* pw) {
    int P = (h + 2 * p - k) / s + 1, Q = (w + 2 * p - k) / s + 1;
    *ph = P; *pw = Q;
    for (int b = 0; b < n; b++)
        for (int i = 0; i < P; i++)
            for (int j = 0; j < Q; j++)
                for (int ch = 0; ch < c; ch++) {
                    int best = -1000, bi = 255;
                    for (int r = 0; r < k; r++)
                        for (int t = 0; t < k; t++) {
                            int hh = i * s + r - p, ww = j * s + t - p;
                            if (hh < 0 || hh >= h || ww < 0 || ww >= w) continue;
                            int v = x[(((int64_t)b * h + hh) * w + ww) * c + ch];
                            if (v > best) { best = v; bi = r * k + t; }
                        }
                    int64_t o = (((int64_t)b * P + i) * Q + j) * c + ch;
                    y[o] = (int8_t)(bi == 255 ? 0 : best);
                    arg[o] = (uint8_t)bi;
                }
}

/* Backward of max pooling: each output error goes to its window's first
 * maximum; overlapping windows add.  Returns the int32 sums. */
void or_maxpool_bwd(const int8_t* e, const uint8_t* arg, int n, int h, int w, int c, int k,
                    int s, int p, int32_t* ex) {
    int P = (h + 2 * p - k) / s + 1, Q = (w + 2 * p - k) / s + 1;
    memset(ex, 0, sizeof(int32_t) * (size_t)n * h * w * c);
    for (int b = 0; b < n; b++)
        for (int i = 0; i < P; i++)
            for (int j = 0; j < Q; j++)
                for (int ch = 0; ch < c; ch++) {
                    int64_t o = (((int64_t)b * P + i) * Q + j) * c + ch;
                    if (arg[o] == 255) continue;
                    int r = arg[o] / k, t = arg[o] % k;
                    int hh = i * s + r - p, ww = j * s + t - p;
                    ex[(((int64_t)b * h + hh) * w + ww) * c + ch] += e[o];
                }
}

/* Gradient of the MSE loss on quantized logits (Sec. 5, FCN: MSE loss), up to
 * its constant factor: E = z s_z - onehot(label) per element, then Q_E = SQ(E, k)
 * (Eq. (EQ)).  With M = max |E| (fp64, over all elements), the code is
 * Clip(rhu(E 2^(k-1) / M)) evaluated, like the BN maps, as the fixed-point map
 * floor((F z + B_t) / 2^P) with F = rhu(s_z q 2^P), B_t = rhu(-t q 2^P) + 2^(P-1),
 * q = 2^(k-1)/M, t in {0,1}.  Labels >= c (e.g. 255) have no target. */
double or_mse_grad(const int8_t* z, int64_t npix, int c, double s_z, const uint8_t* lab, int k,
                   int8_t* E) {
    double M = 0.0;
    for (int64_t i = 0; i < npix; i++)
        for (int ch = 0; ch < c; ch++) {
            double t = lab[i] == ch ? 1.0 : 0.0;
            double v = (double)z[i * c + ch] * s_z - t;
            if (fabs(v) > M) M = fabs(v);
        }
    const int64_t lim = qmax(k);
    if (M == 0.0) {
        memset(E, 0, (size_t)(npix * c));
        return ldexp(1.0, 1 - k);
    }
    const double q = ldexp(1.0, k - 1) / M;
    double lmax = fabs(s_z * q) * 127.0 + fabs(q);
    int P = 62 - frexp_exp(lmax + 1.0);
    if (P > 62) P = 62;
    if (P < 1) P = 1;
    int64_t F = (int64_t)rhu(ldexp(s_z * q, P));
    int64_t B0 = ((int64_t)1 << (P - 1));
    int64_t B1 = (int64_t)rhu(ldexp(-q, P)) + ((int64_t)1 << (P - 1));
    for (int64_t i = 0; i < npix; i++)
        for (int ch = 0; ch < c; ch++) {
            int64_t b = lab[i] == ch ? B1 : B0;
            i128 t = (i128)F * z[i * c + ch] + b;
            E[i * c + ch] = (int8_t)clamp64((int64_t)(t >> P), -lim, lim);
        }
    return ldexp(M, 1 - k);
}

/* ------------------------------------------------------------------ */
/* Network glue of the DeepLabv3-ResNet50 path                          */
/* ------------------------------------------------------------------ */

/* One operand of a combination: integer codes v (int8 or int16, [npix][c] or, when
 * bcast != 0, [n][c] broadcast over the hw pixels of each image), real value
 * a_c v + b_c with a_c = scale (or (gamma_c 2^(2-k_gamma)) * scale for a BN affine term)
 * and b_c = 0 (or beta_c 2^(2-k_beta)). */
typedef struct {
    const void* codes;
    int32_t is16, c, c_offset, bcast;
    double scale;
    const int32_t* gamma;
    const int32_t* beta;
    int32_t k_gamma, k_beta;
} or_term;

static double term_a(const or_term* t, int c) {
    return t->gamma ? ((double)t->gamma[c] * ldexp(1.0, 2 - t->k_gamma)) * t->scale : t->scale;
}
static double term_b(const or_term* t, int c) {
    return t->beta ? (double)t->beta[c] * ldexp(1.0, 2 - t->k_beta) : 0.0;
}
static int64_t term_v(const or_term* t, int64_t img, int64_t pix, int64_t hw, int c) {
    int64_t idx = t->bcast ? img * t->c + c : (img * hw + pix) * t->c + c;
    return t->is16 ? (int64_t)((const int16_t*)t->codes)[idx] : (int64_t)((const int8_t*)t->codes)[idx];
}

/* Sums (concat == 0: every term covers all c_out channels) or channel concatenations
 * (concat != 0: term t fills channels [c_offset, c_offset + c)) of quantized tensors --
 * the residual add of a bottleneck, the sum of the errors reaching one tensor, the ASPP
 * concatenation -- followed by Q_A / Q_E = SQ(act(.), 8) (Eqs. (AQ1),(EQ)).  The real sum
 * is carried in fixed point: z = sum_t (F_t,c v + B_t,c) with F = rhu(a 2^P),
 * B = rhu(b 2^P) and P = 50 - exponent of sum_t max_c(|a| vmax + |b|), so |z| < 2^51;
 * then SQ on the integer z (value z 2^-P) is exact: code = floor((256 z + M) / (2M)).
 * Returns the output scale (M 2^-P) 2^-7. */
double or_combine(const or_term* terms, int nt, int concat, int64_t n, int64_t hw, int c_out,
                  int relu, int8_t* out) {
    double bound = 0.0;
    for (int t = 0; t < nt; t++) {
        double vmax = terms[t].is16 ? 32767.0 : 127.0, lt = 0.0;
        for (int c = 0; c < terms[t].c; c++) {
            double l = fabs(term_a(&terms[t], c)) * vmax + fabs(term_b(&terms[t], c));
            if (l > lt) lt = l;
        }
        bound = bound + lt;
    }
    int P = 50 - frexp_exp(bound + 1.0);
    if (P > 62) P = 62;
    int64_t* z = (int64_t*)malloc(sizeof(int64_t) * (size_t)(n * hw * c_out));
    int64_t M = 0;
    for (int64_t img = 0; img < n; img++)
        for (int64_t pix = 0; pix < hw; pix++)
            for (int co = 0; co < c_out; co++) {
                i128 acc = 0;
                for (int t = 0; t < nt; t++) {
                    int c = co;
                    if (concat) {
                        c = co - terms[t].c_offset;
                        if (c < 0 || c >= terms[t].c) continue;
                    }
                    int64_t F = (int64_t)rhu(ldexp(term_a(&terms[t], c), P));
                    int64_t B = (int64_t)rhu(ldexp(term_b(&terms[t], c), P));
                    acc += (i128)F * term_v(&terms[t], img, pix, hw, c) + B;
                }
                int64_t v = (int64_t)acc;
                if (relu && v < 0) v = 0;
                z[(img * hw + pix) * c_out + co] = v;
                int64_t av = v < 0 ? -v : v;
                if (av > M) M = av;
            }
    for (int64_t i = 0; i < n * hw * c_out; i++) {
        if (M == 0) { out[i] = 0; continue; }
        i128 q = floordiv128(((i128)z[i] << 8) + M, (i128)2 * M);
        out[i] = (int8_t)clamp64((int64_t)q, -127, 127);
    }
    free(z);
    return M ? ldexp((double)M, -P - 7) : ldexp(1.0, -P - 7);
}

/* Per image, the sum over its hw pixels of channels [c_off, c_off + c) of a tensor with
 * c_total channels, then SQ8.  mean != 0: global average pooling (the ASPP image-pooling
 * branch), real value s sum / hw; the 1/hw cancels in x / Scale(x), so the codes are SQ8
 * of the integer sums and the scale is ((s M) / hw) 2^-7.  mean == 0: the backward of a
 * broadcast over the pixels (the error of the pooled branch), scale (s M) 2^-7. */
double or_spatial_sum(const int8_t* x, int64_t n, int64_t hw, int c_total, int c_off, int c,
                      double s, int mean, int8_t* out) {
    int64_t* sums = (int64_t*)malloc(sizeof(int64_t) * (size_t)(n * c + 1));
    int64_t M = 0;
    for (int64_t img = 0; img < n; img++)
        for (int ch = 0; ch < c; ch++) {
            int64_t acc = 0;
            for (int64_t p = 0; p < hw; p++) acc += x[(img * hw + p) * c_total + c_off + ch];
            sums[img * c + ch] = acc;
            if ((acc < 0 ? -acc : acc) > M) M = acc < 0 ? -acc : acc;
        }
    for (int64_t i = 0; i < n * c; i++) {
        if (M == 0) { out[i] = 0; continue; }
        i128 q = floordiv128(((i128)sums[i] << 8) + M, (i128)2 * M);
        out[i] = (int8_t)clamp64((int64_t)q, -127, 127);
    }
    free(sums);
    double sm = M ? s * (double)M : s;
    return ldexp(mean ? sm / (double)hw : sm, -7);
}

/* Bilinear upsampling by an integer factor f with aligned corners (output size
 * (h-1) f + 1, the DeepLab logits 65 -> 513 for f = 8): output (f i + r, f j + t) is
 * ((f-r)(f-t) x[i,j] + r(f-t) x[i+1,j] + (f-r) t x[i,j+1] + r t x[i+1,j+1]) / f^2, exact
 * in integers; SQ8 of the integer numerators (the 1/f^2 cancels), scale ((s M)/f^2) 2^-7. */
double or_bilinear_up(const int8_t* x, int n, int h, int w, int c, int f, double s,
                      int32_t* acc_out, int8_t* out) {
    int H = (h - 1) * f + 1, W = (w - 1) * f + 1;
    int64_t total = (int64_t)n * H * W * c;
    int32_t* a = acc_out ? acc_out : (int32_t*)malloc(sizeof(int32_t) * (size_t)total);
    int64_t M = 0;
    for (int b = 0; b < n; b++)
        for (int I = 0; I < H; I++)
            for (int J = 0; J < W; J++)
                for (int ch = 0; ch < c; ch++) {
                    int i = I / f, r = I % f, j = J / f, t = J % f;
                    int i1 = i + 1 < h ? i + 1 : i, j1 = j + 1 < w ? j + 1 : j;
#define XV(ii, jj) ((int64_t)x[(((int64_t)b * h + (ii)) * w + (jj)) * c + ch])
                    int64_t v = (int64_t)(f - r) * (f - t) * XV(i, j) + (int64_t)r * (f - t) * XV(i1, j) +
                                (int64_t)(f - r) * t * XV(i, j1) + (int64_t)r * t * XV(i1, j1);
#undef XV
                    a[(((int64_t)b * H + I) * W + J) * c + ch] = (int32_t)v;
                    if ((v < 0 ? -v : v) > M) M = v < 0 ? -v : v;
                }
    for (int64_t i = 0; i < total; i++) {
        if (M == 0) { out[i] = 0; continue; }
        i128 q = floordiv128(((i128)a[i] << 8) + M, (i128)2 * M);
        out[i] = (int8_t)clamp64((int64_t)q, -127, 127);
    }
    if (!acc_out) free(a);
    return M ? ldexp((s * (double)M) / (double)(f * f), -7) : ldexp(s / (double)(f * f), -7);
}

/* Adjoint of or_bilinear_up: the error at low-resolution pixel (i, j) collects
 * w_r w_t e[f i' + r, f j' + t] over every output that interpolates from it, with the same
 * integer weights (f-r or r, f-t or t); SQ8 of the integer sums, scale ((s M)/f^2) 2^-7.
 * Output row f i + r (0 < r < f) takes weight (f - r) from row i and r from row i + 1;
 * the last row (h - 1) f takes weight f from row h - 1. */
double or_bilinear_up_bwd(const int8_t* e, int n, int h, int w, int c, int f, double s,
                          int64_t* acc_out, int8_t* out) {
    int H = (h - 1) * f + 1, W = (w - 1) * f + 1;
    int64_t total = (int64_t)n * h * w * c;
    int64_t* a = (int64_t*)calloc((size_t)total, sizeof(int64_t));
    for (int b = 0; b < n; b++)
        for (int I = 0; I < H; I++)
            for (int J = 0; J < W; J++)
                for (int ch = 0; ch < c; ch++) {
                    int i = I / f, r = I % f, j = J / f, t = J % f;
                    int64_t ev = e[(((int64_t)b * H + I) * W + J) * c + ch];
#define AX(ii, jj) a[(((int64_t)b * h + (ii)) * w + (jj)) * c + ch]
                    AX(i, j) += (int64_t)(f - r) * (f - t) * ev;
                    if (r) AX(i + 1, j) += (int64_t)r * (f - t) * ev;
                    if (t) AX(i, j + 1) += (int64_t)(f - r) * t * ev;
                    if (r && t) AX(i + 1, j + 1) += (int64_t)r * t * ev;
#undef AX
                }
    int64_t M = 0;
    for (int64_t i = 0; i < total; i++) {
        int64_t v = a[i] < 0 ? -a[i] : a[i];
        if (v > M) M = v;
    }
    for (int64_t i = 0; i < total; i++) {
        if (M == 0) { out[i] = 0; continue; }
        i128 q = floordiv128(((i128)a[i] << 8) + M, (i128)2 * M);
        out[i] = (int8_t)clamp64((int64_t)q, -127, 127);
    }
    if (acc_out) memcpy(acc_out, a, sizeof(int64_t) * (size_t)total);
    free(a);
    return M ? ldexp((s * (double)M) / (double)(f * f), -7) : ldexp(s / (double)(f * f), -7);
}

/* fp32 exponential for t <= 0, written out so that any IEEE single-precision machine
 * computes the same bits (no fused multiply-add).  Cody-Waite range reduction: k =
 * rhu(t log2 e), r = (t - k c1) - k c2 with c1 + c2 = ln 2 and c1 carrying 15 significant
 * bits, so k c1 is exact for |k| < 2^9; e^r from its Taylor series to degree 7 in Horner
 * form (|r| <= ln2/2 + tiny, truncation below 8e-9 relative); times 2^k by building the
 * exponent field.  t < -87 (and any k < -126) gives 0. */
float or_exp_f32(float t) {
    if (!(t >= -87.0f)) return 0.0f;
    if (t > 0.0f) t = 0.0f;
    const float log2e = 0x1.715476p+0f;   /* fp32 nearest to log2(e) */
    const float c1 = 0x1.62e4p-1f;        /* ln 2 to 15 significant bits */
    const float c2 = 0x1.7f7d1cp-20f;     /* ln 2 - c1, rounded to fp32 */
    float kf = floorf(t * log2e + 0.5f);
    float r = (t - kf * c1) - kf * c2;
    /* Taylor coefficients 1/n!, each the nearest fp32 */
    float p = 0x1.a01a02p-13f;            /* 1/5040 */
    p = p * r + 0x1.6c16c2p-10f;          /* 1/720 */
    p = p * r + 0x1.111112p-7f;           /* 1/120 */
    p = p * r + 0x1.555556p-5f;           /* 1/24 */
    p = p * r + 0x1.555556p-3f;           /* 1/6 */
    p = p * r + 0.5f;
    p = p * r + 1.0f;
    p = p * r + 1.0f;
    int k = (int)kf;
    if (k < -126) return 0.0f;
    union { uint32_t u; float f; } sc;
    sc.u = (uint32_t)(k + 127) << 23;
    return p * sc.f;
}

/* Softmax cross-entropy gradient on quantized logits (the DeepLab head; sum over
 * classes, mean over labelled pixels): per pixel t_c = (z_c - max z) * (float)s_z,
 * e_c = or_exp_f32(t_c), S = e_0 + e_1 + ... (class order), p_c = e_c / S,
 * g_c = p_c - [c == label]; pixels labelled `ignore` give 0.  E = SQ8 of g as a float
 * tensor (Scale = max|g|, Eq. (ScaleQ) on floats, code = rhu(fl(g / Scale) 128) clipped),
 * and its scale is (Scale 2^-7) / n_valid, the 1/n_valid of the mean loss.  All-zero g:
 * codes 0 and scale 2^-7 / max(n_valid, 1).  Returns the scale; *n_valid_out gets the
 * count of labelled pixels. */
double or_ce_grad(const int8_t* z, double s_z, const uint8_t* labels, int64_t npix, int c,
                  int ignore, int8_t* E, int64_t* n_valid_out) {
    float* g = (float*)malloc(sizeof(float) * (size_t)(npix * c + 1));
    float* ex = (float*)malloc(sizeof(float) * (size_t)c);
    const float sf = (float)s_z;
    int64_t nv = 0;
    float gmax = 0.0f;
    for (int64_t p = 0; p < npix; p++) {
        const int8_t* zp = z + p * c;
        int lab = labels[p];
        if (lab == ignore) {
            for (int ch = 0; ch < c; ch++) g[p * c + ch] = 0.0f;
            continue;
        }
        nv++;
        int zm = -128;
        for (int ch = 0; ch < c; ch++) if (zp[ch] > zm) zm = zp[ch];
        float S = 0.0f;
        for (int ch = 0; ch < c; ch++) {
            float t = (float)(zp[ch] - zm) * sf;
            ex[ch] = or_exp_f32(t);
            S = S + ex[ch];
        }
        for (int ch = 0; ch < c; ch++) {
            float pc = ex[ch] / S;
            float gv = ch == lab ? pc - 1.0f : pc;
            g[p * c + ch] = gv;
            if (fabsf(gv) > gmax) gmax = fabsf(gv);
        }
    }
    double scale;
    if (gmax == 0.0f) {
        for (int64_t i = 0; i < npix * c; i++) E[i] = 0;
        scale = ldexp(1.0, -7) / (double)(nv > 0 ? nv : 1);
    } else {
        for (int64_t i = 0; i < npix * c; i++) {
            float t = g[i] / gmax;
            float y = t * 128.0f;
            float f = floorf(y);
            int64_t q = (int64_t)f + ((y - f) >= 0.5f ? 1 : 0);
            E[i] = (int8_t)clamp64(q, -127, 127);
        }
        scale = ldexp((double)gmax, -7) / (double)nv;
    }
    if (n_valid_out) *n_valid_out = nv;
    free(g); free(ex);
    return scale;
}

/* or_exp_f32 over an array (for its tests). */
void or_exp_f32_n(const float* t, int64_t n, float* out) {
    for (int64_t i = 0; i < n; i++) out[i] = or_exp_f32(t[i]);
}
