// iq_glue.cu -- the network glue of the FCN-VGG16 path: max pooling on codes, the
// depthwise (per-class) transposed-convolution upsampling of the decoder (Sec. 2.1,
// Sec. 3.2.1: bilinear-initialised, trainable) with its data and weight gradients, and
// the quantized gradient of the MSE loss on quantized logits (Sec. 5).
// All of these are bandwidth-bound element-wise or windowed kernels on NHWC codes.
#include "iq_internal.cuh"
#include "iq_tc_ptx.cuh"

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

// four channels per thread (c % 4 == 0): block (image b, output row i, a slice of the
// row's Q x c/4 channel groups); 4-byte loads and stores, no 64-bit divisions
__global__ void k_maxpool_fwd4(const int8_t* __restrict__ x, int h, int w, int c, int k, int s,
                               int p, int P, int Q, int8_t* __restrict__ y,
                               uint8_t* __restrict__ arg, uint2* __restrict__ y16) {
    const int c4 = c >> 2;
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= Q * c4) return;
    const int i = blockIdx.y, b = blockIdx.z;
    const int j = idx / c4, cg = idx - j * c4;
    int best[4] = {-1000, -1000, -1000, -1000}, bi[4] = {255, 255, 255, 255};
    for (int r = 0; r < k; r++) {
        const int hh = i * s + r - p;
        if (hh < 0 || hh >= h) continue;
        const int8_t* row = x + (((int64_t)b * h + hh) * w) * c + 4 * cg;
        for (int q = 0; q < k; q++) {
            const int ww = j * s + q - p;
            if (ww < 0 || ww >= w) continue;
            const int v = __ldg(reinterpret_cast<const int*>(row + (int64_t)ww * c));
#pragma unroll
            for (int t = 0; t < 4; t++) {
                const int vt = (int)(int8_t)((v >> (8 * t)) & 0xff);
                if (vt > best[t]) { best[t] = vt; bi[t] = r * k + q; }
            }
        }
    }
    uint32_t yo = 0, ao = 0;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        yo |= ((uint32_t)(bi[t] == 255 ? 0 : best[t]) & 0xffu) << (8 * t);
        ao |= ((uint32_t)bi[t] & 0xffu) << (8 * t);
    }
    const int64_t o = (((int64_t)b * P + i) * Q + j) * c + 4 * cg;
    *reinterpret_cast<uint32_t*>(y + o) = yo;
    *reinterpret_cast<uint32_t*>(arg + o) = ao;
    if (y16) {                        // the fp16 copy of the 4 output codes
        uint2 hv;
        tc::i8x4_to_f16x4(yo, hv.x, hv.y);
        y16[o >> 2] = hv;
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

// Overlapping windows: one thread per 4 channels of an input pixel, for kPoolRows rows (grid:
// pixel-channel groups of a row, row groups, images; 32-bit index arithmetic).  Each input
// sums the errors of the windows whose first maximum it is; the block's largest |sum| goes to
// *amax with one atomic (a single address takes every block's atomic).
constexpr int kPoolRows = 4;

__global__ void __launch_bounds__(kThreads) k_maxpool_bwd4(
    const uint32_t* __restrict__ e4, const uint32_t* __restrict__ arg4, int h, int w, int c4,
    int k, int s, int p, int P, int Q, int4* __restrict__ sums4,
    unsigned long long* __restrict__ amax) {
    __shared__ unsigned long long wmax[kThreads / 32];
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    const int b = blockIdx.z;
    uint64_t mx = 0;
    if (idx < w * c4) {
        const int ww = idx / c4, cg = idx - ww * c4;
        // windows j with j s - p <= ww <= j s - p + k - 1 (likewise i for hh)
        const int j_lo = ww + p - k + 1 > 0 ? (ww + p - k + s) / s : 0;
        const int j_hi = min((ww + p) / s, Q - 1);
        const int h_end = min(h, (int)(blockIdx.y + 1) * kPoolRows);
        for (int hh = blockIdx.y * kPoolRows; hh < h_end; hh++) {
            int sum[4] = {0, 0, 0, 0};
            const int i_lo = hh + p - k + 1 > 0 ? (hh + p - k + s) / s : 0;
            const int i_hi = min((hh + p) / s, P - 1);
            for (int i = i_lo; i <= i_hi; i++) {
                const int r = hh - (i * s - p);
                for (int j = j_lo; j <= j_hi; j++) {
                    const uint32_t tap = (uint32_t)(r * k + ww - (j * s - p));
                    const int64_t oo = (((int64_t)b * P + i) * Q + j) * c4 + cg;
                    const uint32_t av = __ldg(arg4 + oo), ev = __ldg(e4 + oo);
#pragma unroll
                    for (int l = 0; l < 4; l++)
                        if (((av >> (8 * l)) & 0xffu) == tap)
                            sum[l] += (int)(int8_t)(ev >> (8 * l));
                }
            }
            sums4[(((int64_t)b * h + hh) * w + ww) * c4 + cg] =
                make_int4(sum[0], sum[1], sum[2], sum[3]);
#pragma unroll
            for (int l = 0; l < 4; l++) {
                const uint64_t a = (uint64_t)(sum[l] < 0 ? -sum[l] : sum[l]);
                mx = a > mx ? a : mx;
            }
        }
    }
    mx = warp_max_u64(mx);
    if ((threadIdx.x & 31) == 0) wmax[threadIdx.x >> 5] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int i = 1; i < kThreads / 32; i++) mx = wmax[i] > mx ? wmax[i] : mx;
        if (mx) atomicMax(amax, (unsigned long long)mx);
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

// 32-bit invariant division (Granlund & Montgomery, Sec. 4, N = 32) for SQ numerators that
// fit 32 bits: q = floor(n / d) for n < 2^32, 1 <= d < 2^31.
struct Div32 {
    uint32_t mp;
    int sh1, sh2;
};
__device__ __forceinline__ Div32 make_div32(uint32_t d) {
    int l = 0;
    while ((1u << l) < d && l < 31) l++;
    if ((1u << l) < d) l = 32;
    Div32 r;
    r.mp = (uint32_t)(((((uint64_t)1 << l) - d) << 32) / d + 1);
    r.sh1 = l < 1 ? l : 1;
    r.sh2 = l - 1 > 0 ? l - 1 : 0;
    return r;
}
__device__ __forceinline__ uint32_t div32(uint32_t n, const Div32& d) {
    const uint32_t t = __umulhi(d.mp, n);
    return (t + ((n - t) >> d.sh1)) >> d.sh2;
}

// The FCN decoder's shape -- kernel 64, stride 32, padding 16 -- as its own kernel.  Block
// (q, r1, b) covers the output columns J = 32 q - 16 + t (t < 32) of the output rows
// I = 32 p - 16 + r1: every such output reads the inputs (row p-1 or p, column q-1 or q)
// through the taps (r1 + 32 or r1, t + 32 or t).  A thread (one channel) keeps the 4 taps
// of every t packed in one word, so an output is one dp4a of those with the 4 inputs.
template <bool CODES>
__global__ void __launch_bounds__(256) k_up32_fwd(UpP u, const int8_t* __restrict__ x,
                                                  const int8_t* __restrict__ w,
                                                  unsigned long long* __restrict__ amax,
                                                  const RqDiv* __restrict__ dv,
                                                  int8_t* __restrict__ out,
                                                  int32_t* __restrict__ acc_out) {
    const int q = blockIdx.x, r1 = blockIdx.y, b = blockIdx.z, ch = threadIdx.x;
    const bool act = ch < u.c;
    uint32_t wt[32];
    {
        uint32_t w0[16], w1[16];     // tap rows r1 + 32 (input row p-1) and r1 (input row p)
#pragma unroll
        for (int k = 0; k < 4; k++) {
            int4 a = make_int4(0, 0, 0, 0), c = make_int4(0, 0, 0, 0);
            if (act) {
                a = __ldg(reinterpret_cast<const int4*>(w + ((int64_t)ch * 64 + r1 + 32) * 64) + k);
                c = __ldg(reinterpret_cast<const int4*>(w + ((int64_t)ch * 64 + r1) * 64) + k);
            }
            w0[4 * k] = a.x; w0[4 * k + 1] = a.y; w0[4 * k + 2] = a.z; w0[4 * k + 3] = a.w;
            w1[4 * k] = c.x; w1[4 * k + 1] = c.y; w1[4 * k + 2] = c.z; w1[4 * k + 3] = c.w;
        }
        // wt[t] bytes: (w0[t+32], w0[t], w1[t+32], w1[t]) for inputs (p-1,q-1), (p-1,q),
        // (p,q-1), (p,q)
#pragma unroll
        for (int t = 0; t < 32; t++) {
            const uint32_t sh_hi = 8 * ((t + 32) & 3), sh_lo = 8 * (t & 3);
            const uint32_t a0 = (w0[(t + 32) >> 2] >> sh_hi) & 0xffu;
            const uint32_t a1 = (w0[t >> 2] >> sh_lo) & 0xffu;
            const uint32_t a2 = (w1[(t + 32) >> 2] >> sh_hi) & 0xffu;
            const uint32_t a3 = (w1[t >> 2] >> sh_lo) & 0xffu;
            wt[t] = a0 | (a1 << 8) | (a2 << 16) | (a3 << 24);
        }
    }
    uint32_t M = 0;
    Div32 d32;
    if (CODES) {
        M = (uint32_t)dv->M;
        d32 = make_div32(M ? 2 * M : 1);
    }
    uint32_t mx = 0;
    const int Jb = 32 * q - 16;
    const int t_lo = Jb < 0 ? -Jb : 0;
    const int t_hi = Jb + 32 > u.W ? u.W - Jb : 32;
    for (int p = 0; p <= u.h; p++) {
        const int I = 32 * p - 16 + r1;
        if (I < 0 || I >= u.H || !act) continue;
        const bool rp = p >= 1, rc = p < u.h, cp = q >= 1, cc = q < u.w;
        auto xin = [&](int i, int j) -> uint32_t {
            return (uint8_t)x[(((int64_t)b * u.h + i) * u.w + j) * u.c + ch];
        };
        const uint32_t x00 = (rp && cp) ? xin(p - 1, q - 1) : 0u;
        const uint32_t x01 = (rp && cc) ? xin(p - 1, q) : 0u;
        const uint32_t x10 = (rc && cp) ? xin(p, q - 1) : 0u;
        const uint32_t x11 = (rc && cc) ? xin(p, q) : 0u;
        const int xv = (int)(x00 | (x01 << 8) | (x10 << 16) | (x11 << 24));
        const int64_t row0 = ((int64_t)b * u.H + I) * u.W;
        if (CODES && t_lo == 0 && t_hi == 32 && !acc_out) {
            // a whole 32-column segment: the codes of column t at ob[t c]
            int8_t* ob = out + (row0 + Jb) * u.c + ch;
#pragma unroll
            for (int t = 0; t < 32; t++) {
                const int sum = __dp4a(xv, (int)wt[t], 0);
                int c = 0;
                if (M) {
                    const uint32_t num = ((uint32_t)(sum + (int)M) << 8) + M;
                    c = (int)div32(num, d32) - 128;
                    c = c > 127 ? 127 : (c < -127 ? -127 : c);
                }
                ob[t * u.c] = (int8_t)c;
            }
            continue;
        }
#pragma unroll
        for (int t = 0; t < 32; t++) {
            if (t < t_lo || t >= t_hi) continue;
            const int64_t o = (row0 + Jb + t) * u.c + ch;
            const int sum = __dp4a(xv, (int)wt[t], 0);
            if (CODES) {
                int c = 0;
                if (M) {
                    const uint32_t num = ((uint32_t)(sum + (int)M) << 8) + M;
                    c = (int)div32(num, d32) - 128;
                    c = c > 127 ? 127 : (c < -127 ? -127 : c);
                }
                out[o] = (int8_t)c;
                if (acc_out) acc_out[o] = sum;
            } else {
                const uint32_t a = (uint32_t)(sum < 0 ? -sum : sum);
                mx = a > mx ? a : mx;
            }
        }
    }
    if (!CODES) {
        mx = warp_max_u32(mx);
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

// ---- the decoder's backward at kernel 64, stride 32, padding 16, on channel-major errors

// NHWC -> NCHW bytes: block (n, row Ho, 128 columns): the 128 x c bytes of the row segment
// come in as 16-byte loads, each channel's 128 bytes go out as 16-byte stores
__global__ void k_up_tr(const int8_t* __restrict__ E, int8_t* __restrict__ Et, int H, int W,
                        int c) {
    extern __shared__ __align__(16) uint8_t tile[];
    const int w0 = blockIdx.x * 128, Ho = blockIdx.y, b = blockIdx.z;
    const int64_t src0 = (((int64_t)b * H + Ho) * W + w0) * c;
    const int nbytes = 128 * c;
    for (int i = threadIdx.x; i < nbytes / 16; i += blockDim.x)
        reinterpret_cast<uint4*>(tile)[i] = __ldg(reinterpret_cast<const uint4*>(E + src0) + i);
    __syncthreads();
    for (int i = threadIdx.x; i < c * 8; i += blockDim.x) {
        const int ch = i >> 3, seg = i & 7;
        uint32_t w[4];
#pragma unroll
        for (int k = 0; k < 4; k++) {
            uint32_t v = 0;
#pragma unroll
            for (int bb = 0; bb < 4; bb++)
                v |= (uint32_t)tile[(seg * 16 + 4 * k + bb) * c + ch] << (8 * bb);
            w[k] = v;
        }
        int8_t* dst = Et + (((int64_t)b * c + ch) * H + Ho) * W + w0 + seg * 16;
        *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// data gradient: thread per (n, c, i, j) with j fastest; each tap row r contributes the dot
// product of 64 error bytes (4 x 16-byte loads of the channel-major row) with the weight row
__global__ void __launch_bounds__(256) k_up32_bwd(UpP u, const int8_t* __restrict__ Et,
                                                  const int8_t* __restrict__ w,
                                                  int32_t* __restrict__ ex,
                                                  unsigned long long* __restrict__ amax) {
    const int64_t total = (int64_t)u.n * u.c * u.h * u.w;
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    uint32_t mx = 0;
    if (idx < total) {
        const int j = (int)(idx % u.w);
        const int i = (int)((idx / u.w) % u.h);
        const int ch = (int)((idx / ((int64_t)u.w * u.h)) % u.c);
        const int b = (int)(idx / ((int64_t)u.w * u.h * u.c));
        const int8_t* plane = Et + ((int64_t)b * u.c + ch) * u.H * u.W;
        const int8_t* wr = w + (int64_t)ch * 64 * 64;
        const int col0 = 32 * j - 16;
        int sum = 0;
        for (int r = 0; r < 64; r++) {
            const int Ho = 32 * i + r - 16;
            if (Ho < 0 || Ho >= u.H) continue;
            const int8_t* row = plane + (int64_t)Ho * u.W;
#pragma unroll
            for (int q = 0; q < 4; q++) {
                const int col = col0 + 16 * q;
                if (col < 0 || col >= u.W) continue;
                const int4 e = __ldg(reinterpret_cast<const int4*>(row + col));
                const int4 f = __ldg(reinterpret_cast<const int4*>(wr + r * 64 + 16 * q));
                sum = __dp4a(e.x, f.x, sum);
                sum = __dp4a(e.y, f.y, sum);
                sum = __dp4a(e.z, f.z, sum);
                sum = __dp4a(e.w, f.w, sum);
            }
        }
        ex[(((int64_t)b * u.h + i) * u.w + j) * u.c + ch] = sum;
        mx = (uint32_t)(sum < 0 ? -sum : sum);
    }
    mx = warp_max_u32(mx);
    if ((threadIdx.x & 31) == 0 && mx) atomicMax(amax, (unsigned long long)mx);
}

// weight gradient: block (c, 4 tap rows), 64 threads = 4 rows x 16 groups of 4 tap columns;
// the channel's input codes sit in shared memory, each term is one 4-byte error load and
// 4 products
__global__ void __launch_bounds__(64) k_up32_wgrad(UpP u, const int8_t* __restrict__ x,
                                                   const int8_t* __restrict__ Et,
                                                   long long* __restrict__ g) {
    extern __shared__ int8_t xs[];
    const int ch = blockIdx.x, r = blockIdx.y * 4 + (threadIdx.x >> 4), q = threadIdx.x & 15;
    const int nx = u.n * u.h * u.w;
    for (int k = threadIdx.x; k < nx; k += blockDim.x) xs[k] = x[(int64_t)k * u.c + ch];
    __syncthreads();
    int s0 = 0, s1 = 0, s2 = 0, s3 = 0;
    for (int b = 0; b < u.n; b++) {
        const int8_t* plane = Et + ((int64_t)b * u.c + ch) * u.H * u.W;
        for (int i = 0; i < u.h; i++) {
            const int Ho = 32 * i + r - 16;
            if (Ho < 0 || Ho >= u.H) continue;
            const int8_t* row = plane + (int64_t)Ho * u.W;
            const int8_t* xr = xs + (b * u.h + i) * u.w;
            for (int j = 0; j < u.w; j++) {
                const int col = 32 * j - 16 + 4 * q;
                if (col < 0 || col >= u.W) continue;
                const int xv = xr[j];
                const int e = __ldg(reinterpret_cast<const int*>(row + col));
                s0 += xv * (int)(int8_t)(e & 0xff);
                s1 += xv * (int)(int8_t)((e >> 8) & 0xff);
                s2 += xv * (int)(int8_t)((e >> 16) & 0xff);
                s3 += xv * (int)(int8_t)(e >> 24);
            }
        }
    }
    long long* dst = g + ((int64_t)ch * 64 + r) * 64 + 4 * q;
    dst[0] = s0; dst[1] = s1; dst[2] = s2; dst[3] = s3;
}

// ------------------------------------------------------------------ MSE loss gradient

struct MseP {
    long long F, B0, B1;
    int P;
    double s_out;
};

__device__ __forceinline__ uint32_t word_of(const uint32_t (&w)[4], int t) {
    return t < 8 ? (t < 4 ? w[0] : w[1]) : (t < 12 ? w[2] : w[3]);
}
__device__ __forceinline__ int sbyte_of(const uint32_t (&w)[4], int t) {
    return (int)(int8_t)(word_of(w, t) >> (8 * (t & 3)));
}
__device__ __forceinline__ void set_byte(uint32_t (&w)[4], int t, uint32_t v) {
    const uint32_t sh = 8 * (t & 3), m = ~(0xffu << sh);
#pragma unroll
    for (int k = 0; k < 4; k++)
        if ((t >> 2) == k) w[k] = (w[k] & m) | ((v & 0xffu) << sh);
}

// extremes of z for target (t=1) and non-target (t=0) elements: [max0, min0, max1, min1].
// 16 elements per thread and step (one 16-byte load).  With c >= 16 a step holds at most two
// target elements (one per pixel it touches): they are taken out one by one, replaced by a
// non-target byte of the same step, and the 16 bytes go through packed __vmaxs4 / __vmins4.
__global__ void k_mse_stats(const int8_t* __restrict__ z, const uint8_t* __restrict__ lab,
                            int64_t npix, int c, int* __restrict__ ext, UDiv dc, bool vec) {
    int mx0 = INT_MIN, mn0 = INT_MAX, mx1 = INT_MIN, mn1 = INT_MAX;
    uint32_t pmx = 0x80808080u, pmn = 0x7f7f7f7fu;     // packed running extremes (non-target)
    const int64_t total = npix * c;
    const int64_t n16 = vec ? total / 16 : 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n16; u += stride) {
        const int4 v = __ldg(reinterpret_cast<const int4*>(z) + u);
        uint32_t w[4] = {(uint32_t)v.x, (uint32_t)v.y, (uint32_t)v.z, (uint32_t)v.w};
        int64_t px = (int64_t)udiv((uint64_t)(u * 16), dc);
        const int ch0 = (int)(u * 16 - px * c);
        if (c >= 16) {
            const int n0 = c - ch0 < 16 ? c - ch0 : 16;    // bytes of pixel px
            const int t1 = (int)lab[px] - ch0;
            const bool v1 = t1 >= 0 && t1 < n0;
            int t2 = 16;
            if (n0 < 16) {
                const int l2 = lab[px + 1];
                if (l2 < 16 - n0) t2 = n0 + l2;
            }
            const bool v2 = t2 < 16;
            if (v1) { const int x = sbyte_of(w, t1); mx1 = max(mx1, x); mn1 = min(mn1, x); }
            if (v2) { const int x = sbyte_of(w, t2); mx1 = max(mx1, x); mn1 = min(mn1, x); }
            if (v1 || v2) {
                int r = 0;
                if ((v1 && t1 == r) || (v2 && t2 == r)) r = 1;
                if ((v1 && t1 == r) || (v2 && t2 == r)) r = 2;
                const uint32_t rb = (uint32_t)sbyte_of(w, r) & 0xffu;
                if (v1) set_byte(w, t1, rb);
                if (v2) set_byte(w, t2, rb);
            }
            pmx = __vmaxs4(pmx, __vmaxs4(__vmaxs4(w[0], w[1]), __vmaxs4(w[2], w[3])));
            pmn = __vmins4(pmn, __vmins4(__vmins4(w[0], w[1]), __vmins4(w[2], w[3])));
        } else {
            int ch = ch0;
            int lb = lab[px];
#pragma unroll
            for (int j = 0; j < 16; j++) {
                const int zv = (int)(int8_t)(w[j >> 2] >> (8 * (j & 3)));
                if (lb == ch) { mx1 = max(mx1, zv); mn1 = min(mn1, zv); }
                else { mx0 = max(mx0, zv); mn0 = min(mn0, zv); }
                if (++ch == c && j < 15) { ch = 0; px++; lb = lab[px]; }
            }
        }
    }
    if (n16 > 0 && c >= 16 && (int64_t)blockIdx.x * blockDim.x + threadIdx.x < n16) {
#pragma unroll
        for (int j = 0; j < 4; j++) {
            mx0 = max(mx0, (int)(int8_t)(pmx >> (8 * j)));
            mn0 = min(mn0, (int)(int8_t)(pmn >> (8 * j)));
        }
    }
    for (int64_t o = n16 * 16 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < total;
         o += stride) {
        const int zv = z[o];
        const int64_t px = (int64_t)udiv((uint64_t)o, dc);
        if (lab[px] == (int)(o - px * c)) { mx1 = max(mx1, zv); mn1 = min(mn1, zv); }
        else { mx0 = max(mx0, zv); mn0 = min(mn0, zv); }
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

__device__ __forceinline__ int mse_code(int zv, bool tgt, const MseP& p, int64_t lim) {
    long long t = p.F * (long long)zv + (tgt ? p.B1 : p.B0);
    return (int)clamp64(t >> p.P, -lim, lim);
}

__global__ void k_mse_codes(const int8_t* __restrict__ z, const uint8_t* __restrict__ lab,
                            int64_t npix, int c, int k, const MseP* __restrict__ prm,
                            int8_t* __restrict__ E, UDiv dc, bool vec) {
    // the code of every (z, target) pair, from the fixed-point map: one table per block
    __shared__ int8_t tab[512];
    {
        const MseP p = *prm;
        const int64_t lim = qmax(k);
        for (int i = threadIdx.x; i < 512; i += blockDim.x)
            tab[i] = (int8_t)mse_code((int)(int8_t)(i & 0xff), i >= 256, p, lim);
    }
    __syncthreads();
    const int64_t total = npix * c;
    const int64_t n16 = vec ? total / 16 : 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n16; u += stride) {
        const int4 v = __ldg(reinterpret_cast<const int4*>(z) + u);
        const uint32_t wv[4] = {(uint32_t)v.x, (uint32_t)v.y, (uint32_t)v.z, (uint32_t)v.w};
        int64_t px = (int64_t)udiv((uint64_t)(u * 16), dc);
        int ch = (int)(u * 16 - px * c);
        int lb = lab[px];
        uint32_t o[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int j = 0; j < 16; j++) {
            const uint32_t zb = (wv[j >> 2] >> (8 * (j & 3))) & 0xffu;
            const uint32_t e = (uint8_t)tab[zb | (lb == ch ? 256u : 0u)];
            o[j >> 2] |= e << (8 * (j & 3));
            if (++ch == c && j < 15) { ch = 0; px++; lb = lab[px]; }
        }
        reinterpret_cast<int4*>(E)[u] = make_int4((int)o[0], (int)o[1], (int)o[2], (int)o[3]);
    }
    for (int64_t i = n16 * 16 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += stride) {
        const int64_t px = (int64_t)udiv((uint64_t)i, dc);
        const uint32_t zb = (uint8_t)z[i];
        E[i] = tab[zb | (lab[px] == (int)(i - px * c) ? 256u : 0u)];
    }
}

}  // namespace iq

using namespace iq;

// ==================================================================== C ABI

extern "C" iq_status iq_maxpool_fwd(const int8_t* x, int32_t n, int32_t h, int32_t w, int32_t c,
                                    int32_t k, int32_t s, int32_t p, int8_t* y, uint8_t* arg,
                                    void* y_f16, iq_stream stream) {
    if (!x || !y || !arg || n <= 0 || h <= 0 || w <= 0 || c <= 0 || k <= 0 || s <= 0 || p < 0 ||
        k > 15 || 2 * p >= k + 1 || h + 2 * p < k || w + 2 * p < k)
        return IQ_ERR_INVALID_ARG;
    int P = (h + 2 * p - k) / s + 1, Q = (w + 2 * p - k) / s + 1;
    int64_t total = (int64_t)n * P * Q * c;
    if (y_f16 && !f16_copy_ok(y, y_f16, total)) return IQ_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    if (c % 4 == 0 && (((uintptr_t)x | (uintptr_t)y | (uintptr_t)arg) & 3) == 0 && n <= 65535 &&
        P <= 65535) {
        dim3 grid((unsigned)((Q * (c / 4) + kThreads - 1) / kThreads), (unsigned)P, (unsigned)n);
        k_maxpool_fwd4<<<grid, kThreads, 0, st>>>(x, h, w, c, k, s, p, P, Q, y, arg,
                                                   (uint2*)y_f16);
        IQ_LAUNCH_CHECK();
        return IQ_OK;
    }
    k_maxpool_fwd<<<grid_for(total), kThreads, 0, st>>>(x, n, h, w, c, k, s, p, P, Q, y, arg);
    IQ_LAUNCH_CHECK();
    if (y_f16) return codes_to_f16(y, (__half*)y_f16, total, st);
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
    // 4 channels a thread over kPoolRows rows, a block row of (pixel, channel group)s
    const bool vec4 = c % 4 == 0 && n <= 65535 && (h + kPoolRows - 1) / kPoolRows <= 65535 &&
                      (int64_t)w * (c / 4) < (1 << 30) &&
                      ((((uintptr_t)e) | (uintptr_t)arg) & 3) == 0;
    if (vec4)
        k_maxpool_bwd4<<<dim3((unsigned)((w * (c / 4) + kThreads - 1) / kThreads),
                              (unsigned)((h + kPoolRows - 1) / kPoolRows), (unsigned)n),
                         kThreads, 0, st>>>((const uint32_t*)e, (const uint32_t*)arg, h, w, c / 4,
                                            k, s, p, P, Q, (int4*)sums, cell);
    else
        k_maxpool_bwd<<<grid_for(total), kThreads, 0, st>>>(e, arg, n, h, w, c, k, s, p, P, Q,
                                                            sums, nullptr, cell);
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
    // + the channel-major copy of the errors used at kernel R, stride R/2 (H = h R/2)
    *bytes = (size_t)c * R * R * 8 + (size_t)n * h * w * c * 4 + requant_ws_bytes() + 2048 +
             (size_t)n * h * w * c * ((size_t)R / 2) * ((size_t)R / 2) + 256;
    return IQ_OK;
}

// whether the decoder backward can take the channel-major path: kernel 64, stride 32,
// padding 16, output width a multiple of 128, aligned buffers, room in the workspace
static bool up32_ok(const UpP& u, const void* E, const void* w, size_t ws_bytes, size_t used) {
    return u.R == 64 && u.st == 32 && u.pad == 16 && u.W % 128 == 0 &&
           (128 * (int64_t)u.c) % 16 == 0 && (((uintptr_t)E | (uintptr_t)w) & 15) == 0 &&
           128 * u.c <= 48 * 1024 && u.n <= 65535 && u.H <= 65535 &&
           (int64_t)u.n * u.h * u.w <= 48 * 1024 &&
           ws_bytes >= used + (size_t)u.n * u.H * u.W * u.c + 256;
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
    if (R == 64 && stride == 32 && pad == 16 && c <= 256 && ((uintptr_t)w & 15) == 0 &&
        n <= 65535) {
        // the FCN decoder shape: |sum| <= 4 * 127^2, so the SQ numerators fit 32 bits
        dim3 g32((unsigned)(wd + 1), 32u, (unsigned)n);
        const int thr = (c + 31) / 32 * 32;
        k_up32_fwd<false><<<g32, thr, 0, st>>>(u, x, w, cell, nullptr, nullptr, nullptr);
        IQ_LAUNCH_CHECK();
        k_scale_pow2<<<1, 1, 0, st>>>(s_x, -7, s_acc);
        IQ_LAUNCH_CHECK();
        k_sq_prepare<<<1, 1, 0, st>>>(cell, s_acc, 8, dv, s_out);
        IQ_LAUNCH_CHECK();
        k_up32_fwd<true><<<g32, thr, 0, st>>>(u, x, w, nullptr, dv, out, acc_out);
        IQ_LAUNCH_CHECK();
        return IQ_OK;
    }
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
    unsigned long long* cell = (unsigned long long*)rq;
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, 8, st));
    if (up32_ok(u, E, w, ws_bytes, cur.off)) {
        int8_t* Et = cur.take<int8_t>((size_t)n * u.H * u.W * c);
        dim3 gt((unsigned)(u.W / 128), (unsigned)u.H, (unsigned)n);
        k_up_tr<<<gt, 256, 128 * c, st>>>(E, Et, u.H, u.W, c);
        IQ_LAUNCH_CHECK();
        const int64_t total = (int64_t)n * c * h * wd;
        k_up32_bwd<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(u, Et, w, acc, cell);
        IQ_LAUNCH_CHECK();
    } else {
        k_up_wT<<<grid_for((int64_t)c * R * R), kThreads, 0, st>>>(w, wT, c, R);
        IQ_LAUNCH_CHECK();
        int thr = c >= 256 ? 256 : ((c + 31) / 32) * 32;
        k_up_bwd<<<n * h * wd, thr, 0, st>>>(u, E, wT, acc, cell);
        IQ_LAUNCH_CHECK();
    }
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
    if (up32_ok(u, E, x, ws_bytes, cur.off)) {
        int8_t* Et = cur.take<int8_t>((size_t)n * u.H * u.W * c);
        dim3 gt((unsigned)(u.W / 128), (unsigned)u.H, (unsigned)n);
        k_up_tr<<<gt, 256, 128 * c, st>>>(E, Et, u.H, u.W, c);
        IQ_LAUNCH_CHECK();
        k_up32_wgrad<<<dim3((unsigned)c, 16u), 64, (size_t)n * h * wd, st>>>(u, x, Et,
                                                                          (long long*)G);
        IQ_LAUNCH_CHECK();
    } else {
        int thr = c >= 256 ? 256 : ((c + 31) / 32) * 32;
        k_up_wgrad<<<R * R, thr, 0, st>>>(u, x, E, (long long*)G);
        IQ_LAUNCH_CHECK();
    }
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
    const UDiv dc = make_udiv((uint64_t)c);
    const bool vec = (((uintptr_t)z | (uintptr_t)E) & 15) == 0;
    const int g = grid_for(vec ? total / 16 + 1 : total);
    k_mse_stats<<<g, kThreads, 0, st>>>(z, labels, npix, c, ext, dc, vec);
    IQ_LAUNCH_CHECK();
    k_mse_fin<<<1, 1, 0, st>>>(ext, s_z, 8, prm, s_e);
    IQ_LAUNCH_CHECK();
    k_mse_codes<<<g, kThreads, 0, st>>>(z, labels, npix, c, 8, prm, E, dc, vec);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}
