// iq_glue.cu -- the network glue of the FCN-VGG16 path: max pooling on codes, the
// depthwise (per-class) transposed-convolution upsampling of the decoder (Sec. 2.1,
// Sec. 3.2.1: bilinear-initialised, trainable) with its data and weight gradients, and
// the quantized gradient of the MSE loss on quantized logits (Sec. 5).
// All of these are bandwidth-bound element-wise or windowed kernels on NHWC codes.
#include "iq_internal.cuh"

#include <climits>

namespace iq {

// ------------------------------------------------------------------ max pooling

__global__ void k_maxpool_fwd(const int8_t* __restrict__ x, int n, int h, int w, int c, int k,
                              int s, int p, int P, int Q, int8_t* __restrict__ y,
                              uint8_t* __restrict__ arg) {
    const int64_t total = (int64_t)n * P * Q * c;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < total;
         o += (int64_t)gridDim.x * blockDim.x) {
        int ch = (int)(o % c);
        int64_t t = o / c;
        int j = (int)(t % Q); t /= Q;
        int i = (int)(t % P);
        int b = (int)(t / P);
        int best = -1000, bi = 255;
        for (int r = 0; r < k; r++) {
            int hh = i * s + r - p;
            if (hh < 0 || hh >= h) continue;
            for (int q = 0; q < k; q++) {
                int ww = j * s + q - p;
                if (ww < 0 || ww >= w) continue;
                int v = x[(((int64_t)b * h + hh) * w + ww) * c + ch];
                if (v > best) { best = v; bi = r * k + q; }
            }
        }
        y[o] = (int8_t)(bi == 255 ? 0 : best);
        arg[o] = (uint8_t)bi;
    }
}

// gather form of the backward: input position (hh, ww) sums the errors of the
// windows whose first maximum it is (no atomics, deterministic)
__global__ void k_maxpool_bwd(const int8_t* __restrict__ e, const uint8_t* __restrict__ arg,
                              int n, int h, int w, int c, int k, int s, int p, int P, int Q,
                              int32_t* __restrict__ out32, int8_t* __restrict__ out8,
                              unsigned long long* __restrict__ amax) {
    const int64_t total = (int64_t)n * h * w * c;
    uint64_t mx = 0;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < total;
         o += (int64_t)gridDim.x * blockDim.x) {
        int ch = (int)(o % c);
        int64_t t = o / c;
        int ww = (int)(t % w); t /= w;
        int hh = (int)(t % h);
        int b = (int)(t / h);
        int sum = 0;
        // windows (i, j) with i*s - p <= hh < i*s - p + k
        int i_lo = (hh + p - k + s) / s; if (hh + p - k + 1 < 0) i_lo = 0;
        int i_hi = (hh + p) / s;
        int j_lo = (ww + p - k + s) / s; if (ww + p - k + 1 < 0) j_lo = 0;
        int j_hi = (ww + p) / s;
        if (i_lo < 0) i_lo = 0;
        if (j_lo < 0) j_lo = 0;
        if (i_hi > P - 1) i_hi = P - 1;
        if (j_hi > Q - 1) j_hi = Q - 1;
        for (int i = i_lo; i <= i_hi; i++)
            for (int j = j_lo; j <= j_hi; j++) {
                int r = hh - (i * s - p), q = ww - (j * s - p);
                if (r < 0 || r >= k || q < 0 || q >= k) continue;
                int64_t oo = (((int64_t)b * P + i) * Q + j) * c + ch;
                if (arg[oo] == r * k + q) sum += e[oo];
            }
        if (out8) out8[o] = (int8_t)sum;
        if (out32) out32[o] = sum;
        uint64_t a = (uint64_t)(sum < 0 ? -sum : sum);
        mx = a > mx ? a : mx;
    }
    if (amax) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(amax, (unsigned long long)mx);
    }
}

// windows that do not overlap (k == s, no padding): each window scatters its error to
// its first maximum; every input receives at most one error.  4 channels per thread.
__global__ void k_maxpool_bwd_tiled(const int8_t* __restrict__ e, const uint8_t* __restrict__ arg,
                                    int n, int h, int w, int c4, int k, int P, int Q,
                                    int8_t* __restrict__ ex) {
    const int64_t total = (int64_t)n * P * Q * c4;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < total;
         o += (int64_t)gridDim.x * blockDim.x) {
        const int cg = (int)(o % c4);
        int64_t t = o / c4;
        const int j = (int)(t % Q); t /= Q;
        const int i = (int)(t % P);
        const int b = (int)(t / P);
        const uint32_t ev = reinterpret_cast<const uint32_t*>(e)[o];
        const uint32_t av = reinterpret_cast<const uint32_t*>(arg)[o];
        for (int r = 0; r < k; r++) {
            const int hh = i * k + r;
            if (hh >= h) break;
            for (int q = 0; q < k; q++) {
                const int ww = j * k + q;
                if (ww >= w) break;
                const uint32_t tap = (uint32_t)(r * k + q);
                uint32_t v = 0;
#pragma unroll
                for (int l = 0; l < 4; l++)
                    if (((av >> (8 * l)) & 0xffu) == tap) v |= ev & (0xffu << (8 * l));
                reinterpret_cast<uint32_t*>(ex)[(((int64_t)b * h + hh) * w + ww) * c4 + cg] = v;
            }
        }
    }
}

__global__ void k_copy_scale(const double* __restrict__ a, double* __restrict__ b) { *b = *a; }
__global__ void k_scale_pow2(const double* __restrict__ a, int e, double* __restrict__ out) {
    *out = ldexp(*a, e);
}
__global__ void k_scale_product(const double* __restrict__ a, const double* __restrict__ b,
                                double* __restrict__ out) {
    *out = __dmul_rn(*a, *b);
}

// ------------------------------------------------------------------ depthwise transposed conv
// out[n, H, W, c] = sum over (i, j) with r = H + pad - i*st in [0,R), t = W + pad - j*st in [0,R)
// of x[n, i, j, c] * w[c][r][t].  x: [n][h][w][c], w: [c][R][R].

struct UpP {
    int n, h, w, c, R, st, pad, H, W;
};

// One block per (n, output row, 32 output columns); one thread per channel.  The input
// rows / columns reaching an output pixel are i = (Ho + pad - r) / st for the taps r of the
// kernel with the right residue: at most ceil(R / st) of them per dimension.
template <bool CODES>
__global__ void k_up_fwd(UpP u, const int8_t* __restrict__ x, const int8_t* __restrict__ wT,
                         unsigned long long* __restrict__ amax, const RqDiv* __restrict__ dv,
                         int k, int8_t* __restrict__ out, int32_t* __restrict__ acc_out) {
    const int Ho = blockIdx.y % u.H;
    const int b = blockIdx.y / u.H;
    const int Wo0 = blockIdx.x * 32;
    const int ch = threadIdx.x;
    RqDiv d;
    if (CODES) d = *dv;
    const int64_t lim = qmax(k);
    uint64_t mx = 0;
    // input rows of this output row
    int rows_i[4], rows_r[4], nr = 0;
    for (int i = (Ho + u.pad) / u.st; i >= 0 && nr < 4; i--) {
        int r = Ho + u.pad - i * u.st;
        if (r >= u.R) break;
        if (i < u.h) { rows_i[nr] = i; rows_r[nr] = r; nr++; }
    }
    if (ch < u.c) {
        for (int wo = 0; wo < 32; wo++) {
            const int Wo = Wo0 + wo;
            if (Wo >= u.W) break;
            int sum = 0;
            for (int j = (Wo + u.pad) / u.st; j >= 0; j--) {
                int t = Wo + u.pad - j * u.st;
                if (t >= u.R) break;
                if (j >= u.w) continue;
                for (int a = 0; a < nr; a++)
                    sum += (int)x[(((int64_t)b * u.h + rows_i[a]) * u.w + j) * u.c + ch] *
                           (int)wT[((int64_t)rows_r[a] * u.R + t) * u.c + ch];
            }
            const int64_t o = (((int64_t)b * u.H + Ho) * u.W + Wo) * u.c + ch;
            if (CODES) {
                if (acc_out) acc_out[o] = sum;
                int64_t c = 0;
                if (d.M) {
                    uint64_t num = ((uint64_t)((int64_t)sum + (int64_t)d.M) << k) + d.M;
                    c = clamp64((int64_t)udiv(num, d.div) - (int64_t(1) << (k - 1)), -lim, lim);
                }
                out[o] = (int8_t)c;
            } else {
                uint64_t a = (uint64_t)(sum < 0 ? -sum : sum);
                mx = a > mx ? a : mx;
            }
        }
    }
    if (!CODES) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(amax, (unsigned long long)mx);
    }
}

__global__ void k_sq_prepare(const unsigned long long* __restrict__ cell,
                             const double* __restrict__ s_in, int k, RqDiv* __restrict__ dv,
                             double* __restrict__ s_out) {
    uint64_t M = *cell;
    RqDiv d;
    d.M = M;
    d.div = make_udiv(M ? 2 * M : 1);
    *dv = d;
    *s_out = M ? ldexp(__dmul_rn(*s_in, (double)M), 1 - k) : ldexp(*s_in, 1 - k);
}

// weights [c][R][R] -> [R][R][c] so that a warp over channels reads them coalesced
__global__ void k_up_wT(const int8_t* __restrict__ w, int8_t* __restrict__ wT, int c, int R) {
    const int64_t total = (int64_t)c * R * R;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        int ch = (int)(i / ((int64_t)R * R));
        int rt = (int)(i % ((int64_t)R * R));
        wT[(int64_t)rt * c + ch] = w[i];
    }
}

// data gradient: ex[n, i, j, c] = sum_{r,t} E[n, i*st + r - pad, j*st + t - pad, c] w[c][r][t]
// one block per input pixel (n, i, j); threads over channels
__global__ void k_up_bwd(UpP u, const int8_t* __restrict__ E, const int8_t* __restrict__ wT,
                         int32_t* __restrict__ ex, unsigned long long* __restrict__ amax) {
    const int pix = blockIdx.x;
    const int b = pix / (u.h * u.w);
    const int i = (pix / u.w) % u.h;
    const int j = pix % u.w;
    uint64_t mx = 0;
    for (int ch = threadIdx.x; ch < u.c; ch += blockDim.x) {
        int sum = 0;
        for (int r = 0; r < u.R; r++) {
            int Ho = i * u.st + r - u.pad;
            if (Ho < 0 || Ho >= u.H) continue;
            for (int t = 0; t < u.R; t++) {
                int Wo = j * u.st + t - u.pad;
                if (Wo < 0 || Wo >= u.W) continue;
                sum += (int)E[(((int64_t)b * u.H + Ho) * u.W + Wo) * u.c + ch] *
                       (int)wT[((int64_t)r * u.R + t) * u.c + ch];
            }
        }
        ex[(int64_t)pix * u.c + ch] = sum;
        uint64_t a = (uint64_t)(sum < 0 ? -sum : sum);
        mx = a > mx ? a : mx;
    }
    mx = warp_max_u64(mx);
    if ((threadIdx.x & 31) == 0 && mx) atomicMax(amax, (unsigned long long)mx);
}

// weight gradient: g[c][r][t] = sum_{n,i,j} x[n,i,j,c] E[n, i*st + r - pad, j*st + t - pad, c]
// one block per tap (r, t); threads over channels; int32 partial sums (n h w 127^2 < 2^31)
__global__ void k_up_wgrad(UpP u, const int8_t* __restrict__ x, const int8_t* __restrict__ E,
                           long long* __restrict__ g) {
    const int r = blockIdx.x / u.R, t = blockIdx.x % u.R;
    for (int ch = threadIdx.x; ch < u.c; ch += blockDim.x) {
        int sum = 0;
        for (int b = 0; b < u.n; b++)
            for (int i = 0; i < u.h; i++) {
                int Ho = i * u.st + r - u.pad;
                if (Ho < 0 || Ho >= u.H) continue;
                for (int j = 0; j < u.w; j++) {
                    int Wo = j * u.st + t - u.pad;
                    if (Wo < 0 || Wo >= u.W) continue;
                    sum += (int)x[(((int64_t)b * u.h + i) * u.w + j) * u.c + ch] *
                           (int)E[(((int64_t)b * u.H + Ho) * u.W + Wo) * u.c + ch];
                }
            }
        g[((int64_t)ch * u.R + r) * u.R + t] = sum;
    }
}

// ------------------------------------------------------------------ MSE loss gradient

struct MseP {
    long long F, B0, B1;
    int P;
    double s_out;
};

// extremes of z for target (t=1) and non-target (t=0) elements: [max0, min0, max1, min1]
__global__ void k_mse_stats(const int8_t* __restrict__ z, const uint8_t* __restrict__ lab,
                            int64_t npix, int c, int* __restrict__ ext) {
    int mx0 = INT_MIN, mn0 = INT_MAX, mx1 = INT_MAX, mn1 = INT_MAX;
    mx1 = INT_MIN;
    const UDiv dc = make_udiv((uint64_t)c);
    const int64_t total = npix * c;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < total;
         o += (int64_t)gridDim.x * blockDim.x) {
        int v = z[o];
        const int64_t px = (int64_t)udiv((uint64_t)o, dc);
        bool tgt = lab[px] == (uint8_t)(o - px * c);
        if (tgt) { mx1 = max(mx1, v); mn1 = min(mn1, v); }
        else { mx0 = max(mx0, v); mn0 = min(mn0, v); }
    }
    for (int off = 16; off > 0; off >>= 1) {
        mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
        mn0 = min(mn0, __shfl_xor_sync(0xffffffffu, mn0, off));
        mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
        mn1 = min(mn1, __shfl_xor_sync(0xffffffffu, mn1, off));
    }
    if ((threadIdx.x & 31) == 0) {
        atomicMax(&ext[0], mx0); atomicMin(&ext[1], mn0);
        atomicMax(&ext[2], mx1); atomicMin(&ext[3], mn1);
    }
}

__global__ void k_mse_init(int* ext) {
    ext[0] = INT_MIN; ext[1] = INT_MAX; ext[2] = INT_MIN; ext[3] = INT_MAX;
}

__device__ __forceinline__ int frexp_e(double v) {
    int e;
    frexp(v, &e);
    return e;
}

// M = max |z s_z - t| from the extremes (|fl(z s_z) - t| is monotone in z per t)
__global__ void k_mse_fin(const int* __restrict__ ext, const double* __restrict__ s_zp, int k,
                          MseP* __restrict__ prm, double* __restrict__ s_out) {
    const double s_z = *s_zp;
    double M = 0.0;
    for (int t = 0; t < 2; t++) {
        int hi = ext[2 * t], lo = ext[2 * t + 1];
        if (lo > hi) continue;
        double tv = (double)t;
        M = fmax(M, fabs(__dsub_rn(__dmul_rn((double)hi, s_z), tv)));
        M = fmax(M, fabs(__dsub_rn(__dmul_rn((double)lo, s_z), tv)));
    }
    MseP p;
    if (M == 0.0) {
        p.F = 0; p.B0 = 0; p.B1 = 0; p.P = 1; p.s_out = ldexp(1.0, 1 - k);
    } else {
        const double q = __ddiv_rn(ldexp(1.0, k - 1), M);
        double lmax = __dadd_rn(__dmul_rn(fabs(__dmul_rn(s_z, q)), 127.0), fabs(q));
        int P = 62 - frexp_e(__dadd_rn(lmax, 1.0));
        P = P > 62 ? 62 : (P < 1 ? 1 : P);
        p.P = P;
        p.F = (long long)rhu(ldexp(__dmul_rn(s_z, q), P));
        p.B0 = 1LL << (P - 1);
        p.B1 = (long long)rhu(ldexp(-q, P)) + (1LL << (P - 1));
        p.s_out = ldexp(M, 1 - k);
    }
    *prm = p;
    *s_out = p.s_out;
}

__global__ void k_mse_codes(const int8_t* __restrict__ z, const uint8_t* __restrict__ lab,
                            int64_t npix, int c, int k, const MseP* __restrict__ prm,
                            int8_t* __restrict__ E) {
    const MseP p = *prm;
    const int64_t lim = qmax(k);
    const UDiv dc = make_udiv((uint64_t)c);
    const int64_t total = npix * c;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < total;
         o += (int64_t)gridDim.x * blockDim.x) {
        const int64_t px = (int64_t)udiv((uint64_t)o, dc);
        bool tgt = lab[px] == (uint8_t)(o - px * c);
        long long t = p.F * (long long)z[o] + (tgt ? p.B1 : p.B0);
        E[o] = (int8_t)clamp64(t >> p.P, -lim, lim);
    }
}

}  // namespace iq

using namespace iq;

// ==================================================================== C ABI

extern "C" iq_status iq_maxpool_fwd(const int8_t* x, int32_t n, int32_t h, int32_t w, int32_t c,
                                    int32_t k, int32_t s, int32_t p, int8_t* y, uint8_t* arg,
                                    iq_stream stream) {
    if (!x || !y || !arg || n <= 0 || h <= 0 || w <= 0 || c <= 0 || k <= 0 || s <= 0 || p < 0 ||
        k > 15 || 2 * p >= k + 1 || h + 2 * p < k || w + 2 * p < k)
        return IQ_ERR_INVALID_ARG;
    int P = (h + 2 * p - k) / s + 1, Q = (w + 2 * p - k) / s + 1;
    int64_t total = (int64_t)n * P * Q * c;
    k_maxpool_fwd<<<grid_for(total), kThreads, 0, (cudaStream_t)stream>>>(x, n, h, w, c, k, s, p,
                                                                          P, Q, y, arg);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_maxpool_bwd(const int8_t* e, const double* s_e, const uint8_t* arg,
                                    int32_t n, int32_t h, int32_t w, int32_t c, int32_t k,
                                    int32_t s, int32_t p, int8_t* ex, double* s_ex, void* ws,
                                    size_t ws_bytes, iq_stream stream) {
    if (!e || !s_e || !arg || !ex || !s_ex || n <= 0 || h <= 0 || w <= 0 || c <= 0 || k <= 0 ||
        s <= 0 || p < 0 || k > 15 || 2 * p >= k + 1 || h + 2 * p < k || w + 2 * p < k)
        return IQ_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    int P = (h + 2 * p - k) / s + 1, Q = (w + 2 * p - k) / s + 1;
    int64_t total = (int64_t)n * h * w * c;
    if (k <= s) {
        // windows do not overlap: every input receives at most one error, same scale
        const bool tiled = k == s && p == 0 && c % 4 == 0 && h % k == 0 && w % k == 0 &&
                           ((((uintptr_t)e) | (uintptr_t)arg | (uintptr_t)ex) & 3) == 0;
        if (tiled) {
            k_maxpool_bwd_tiled<<<grid_for((int64_t)n * P * Q * (c / 4)), kThreads, 0, st>>>(
                e, arg, n, h, w, c / 4, k, P, Q, ex);
        } else {
            k_maxpool_bwd<<<grid_for(total), kThreads, 0, st>>>(e, arg, n, h, w, c, k, s, p, P,
                                                                Q, nullptr, ex, nullptr);
        }
        IQ_LAUNCH_CHECK();
        k_copy_scale<<<1, 1, 0, st>>>(s_e, s_ex);
        IQ_LAUNCH_CHECK();
        return IQ_OK;
    }
    size_t need = (size_t)total * 4 + requant_ws_bytes() + 512;
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    WsCursor cur(ws, ws_bytes);
    int32_t* sums = cur.take<int32_t>((size_t)total);
    void* rq = cur.take<char>(requant_ws_bytes());
    unsigned long long* cell = (unsigned long long*)rq;
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, 8, st));
    k_maxpool_bwd<<<grid_for(total), kThreads, 0, st>>>(e, arg, n, h, w, c, k, s, p, P, Q, sums,
                                                        nullptr, cell);
    IQ_LAUNCH_CHECK();
    // overlapping windows add errors: Q_E = SQ(., 8) of the sums, same element scale s_e
    return requant_apply(sums, IQ_I32, total, s_e, 8, IQ_MODE_SQ, 0, 0, 0, 0, ex, IQ_I8, s_ex, rq,
                         st);
}

static bool up_dims(int32_t n, int32_t h, int32_t w, int32_t c, int32_t R, int32_t st, int32_t pad,
                    UpP* u) {
    if (n <= 0 || h <= 0 || w <= 0 || c <= 0 || R <= 0 || st <= 0 || pad < 0) return false;
    u->n = n; u->h = h; u->w = w; u->c = c; u->R = R; u->st = st; u->pad = pad;
    u->H = (h - 1) * st - 2 * pad + R;
    u->W = (w - 1) * st - 2 * pad + R;
    return u->H > 0 && u->W > 0;
}

extern "C" iq_status iq_upsample_workspace_size(int32_t n, int32_t h, int32_t w, int32_t c,
                                                int32_t R, size_t* bytes) {
    if (!bytes || n <= 0 || h <= 0 || w <= 0 || c <= 0 || R <= 0) return IQ_ERR_INVALID_ARG;
    *bytes = (size_t)c * R * R * 8 + (size_t)n * h * w * c * 4 + requant_ws_bytes() + 2048;
    return IQ_OK;
}

extern "C" iq_status iq_upsample_fwd(const int8_t* x, const double* s_x, const int8_t* w,
                                     int32_t n, int32_t h, int32_t wd, int32_t c, int32_t R,
                                     int32_t stride, int32_t pad, int8_t* out, double* s_out,
                                     int32_t* acc_out, void* ws, size_t ws_bytes,
                                     iq_stream stream) {
    UpP u;
    if (!x || !s_x || !w || !out || !s_out || !up_dims(n, h, wd, c, R, stride, pad, &u))
        return IQ_ERR_INVALID_ARG;
    if (c > 1024 || (R + stride - 1) / stride > 4) return IQ_ERR_UNSUPPORTED;
    size_t need = 0;
    iq_upsample_workspace_size(n, h, wd, c, R, &need);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    WsCursor cur(ws, ws_bytes);
    unsigned long long* cell = cur.take<unsigned long long>(1);
    RqDiv* dv = cur.take<RqDiv>(1);
    double* s_acc = cur.take<double>(1);
    int8_t* wT = cur.take<int8_t>((size_t)c * R * R);
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, 8, st));
    k_up_wT<<<grid_for((int64_t)c * R * R), kThreads, 0, st>>>(w, wT, c, R);
    IQ_LAUNCH_CHECK();
    dim3 grid((unsigned)((u.W + 31) / 32), (unsigned)(n * u.H));
    const int thr = (c + 31) / 32 * 32;
    k_up_fwd<false><<<grid, thr, 0, st>>>(u, x, wT, cell, nullptr, 8, nullptr, nullptr);
    IQ_LAUNCH_CHECK();
    k_scale_pow2<<<1, 1, 0, st>>>(s_x, -7, s_acc);   // weights on the 8-bit grid
    IQ_LAUNCH_CHECK();
    k_sq_prepare<<<1, 1, 0, st>>>(cell, s_acc, 8, dv, s_out);
    IQ_LAUNCH_CHECK();
    k_up_fwd<true><<<grid, thr, 0, st>>>(u, x, wT, nullptr, dv, 8, out, acc_out);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_upsample_bwd(const int8_t* E, const double* s_e, const int8_t* w,
                                     int32_t n, int32_t h, int32_t wd, int32_t c, int32_t R,
                                     int32_t stride, int32_t pad, int8_t* ex, double* s_ex,
                                     int32_t* acc_out, void* ws, size_t ws_bytes,
                                     iq_stream stream) {
    UpP u;
    if (!E || !s_e || !w || !ex || !s_ex || !up_dims(n, h, wd, c, R, stride, pad, &u))
        return IQ_ERR_INVALID_ARG;
    if ((int64_t)R * R * 16129 >= (int64_t(1) << 31)) return IQ_ERR_OVERFLOW_RISK;
    size_t need = 0;
    iq_upsample_workspace_size(n, h, wd, c, R, &need);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    WsCursor cur(ws, ws_bytes);
    int8_t* wT = cur.take<int8_t>((size_t)c * R * R);
    int32_t* sums = cur.take<int32_t>((size_t)n * h * wd * c);
    void* rq = cur.take<char>(requant_ws_bytes());
    double* s_in = cur.take<double>(1);
    int32_t* acc = acc_out ? acc_out : sums;
    k_up_wT<<<grid_for((int64_t)c * R * R), kThreads, 0, st>>>(w, wT, c, R);
    IQ_LAUNCH_CHECK();
    unsigned long long* cell = (unsigned long long*)rq;
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, 8, st));
    int thr = c >= 256 ? 256 : ((c + 31) / 32) * 32;
    k_up_bwd<<<n * h * wd, thr, 0, st>>>(u, E, wT, acc, cell);
    IQ_LAUNCH_CHECK();
    k_scale_pow2<<<1, 1, 0, st>>>(s_e, -7, s_in);
    IQ_LAUNCH_CHECK();
    return requant_apply(acc, IQ_I32, (int64_t)n * h * wd * c, s_in, 8, IQ_MODE_SQ, 0, 0, 0, 0, ex,
                         IQ_I8, s_ex, rq, st);
}

extern "C" iq_status iq_upsample_wgrad(const int8_t* x, const double* s_x, const int8_t* E,
                                       const double* s_e, int32_t n, int32_t h, int32_t wd,
                                       int32_t c, int32_t R, int32_t stride, int32_t pad,
                                       int gq_mode, uint64_t seed, uint64_t layer, uint64_t step,
                                       int8_t* g, double* s_g, int64_t* g_acc_out, void* ws,
                                       size_t ws_bytes, iq_stream stream) {
    UpP u;
    if (!x || !s_x || !E || !s_e || !g || !s_g || !up_dims(n, h, wd, c, R, stride, pad, &u))
        return IQ_ERR_INVALID_ARG;
    if (gq_mode != 1 && gq_mode != 2) return IQ_ERR_INVALID_ARG;
    if ((int64_t)n * h * wd * 16129 >= (int64_t(1) << 31)) return IQ_ERR_OVERFLOW_RISK;
    size_t need = 0;
    iq_upsample_workspace_size(n, h, wd, c, R, &need);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    WsCursor cur(ws, ws_bytes);
    int64_t* gw = cur.take<int64_t>((size_t)c * R * R);
    void* rq = cur.take<char>(requant_ws_bytes());
    double* s_in = cur.take<double>(1);
    int64_t* G = g_acc_out ? g_acc_out : gw;
    int thr = c >= 256 ? 256 : ((c + 31) / 32) * 32;
    k_up_wgrad<<<R * R, thr, 0, st>>>(u, x, E, (long long*)G);
    IQ_LAUNCH_CHECK();
    k_scale_product<<<1, 1, 0, st>>>(s_x, s_e, s_in);
    IQ_LAUNCH_CHECK();
    return requant_int(G, IQ_I64, (int64_t)c * R * R, s_in, 8,
                       gq_mode == 1 ? IQ_MODE_RQ_GQ1 : IQ_MODE_RQ_GQ2, seed, layer, step, 0, g,
                       IQ_I8, s_g, rq, st);
}

extern "C" iq_status iq_mse_grad(const int8_t* z, const double* s_z, const uint8_t* labels,
                                 int64_t npix, int32_t c, int8_t* E, double* s_e, void* ws,
                                 size_t ws_bytes, iq_stream stream) {
    if (!z || !s_z || !labels || !E || !s_e || npix <= 0 || c <= 0 || c > 255)
        return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < 1024) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    WsCursor cur(ws, ws_bytes);
    int* ext = cur.take<int>(4);
    MseP* prm = cur.take<MseP>(1);
    k_mse_init<<<1, 1, 0, st>>>(ext);
    IQ_LAUNCH_CHECK();
    int64_t total = npix * c;
    k_mse_stats<<<grid_for(total), kThreads, 0, st>>>(z, labels, npix, c, ext);
    IQ_LAUNCH_CHECK();
    k_mse_fin<<<1, 1, 0, st>>>(ext, s_z, 8, prm, s_e);
    IQ_LAUNCH_CHECK();
    k_mse_codes<<<grid_for(total), kThreads, 0, st>>>(z, labels, npix, c, 8, prm, E);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}
