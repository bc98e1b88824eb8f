// iq_head.cu -- the DeepLab segmentation head after the classifier: bilinear
// upsampling by an integer factor with aligned corners (x8, 65 -> 513), its adjoint on
// errors, and the softmax cross-entropy gradient on quantized logits (Sec. 5).
#include "iq_internal.cuh"

namespace iq {

namespace {

// Max |v| of a pass and the SQ(., 8) parameters derived from it.
struct SqHdr {
    unsigned long long maxv;
    uint64_t M;
    UDiv div;
    unsigned int gmax_bits;     // softmax head: max |g| as fp32 bits
    unsigned int pad;
    unsigned long long nvalid;  // softmax head: labelled pixels
};

__device__ __forceinline__ int8_t sq8_code(int64_t v, uint64_t M, const UDiv& d) {
    if (!M) return 0;
    uint64_t num = ((uint64_t)(v + (int64_t)M) << 8) + M;
    return (int8_t)clamp64((int64_t)udiv(num, d) - 128, -127, 127);
}

// s_out = ((s M) / den) 2^-7, M = 0: (s / den) 2^-7 (the oracle's operation order)
__global__ void k_sq8_params(SqHdr* hdr, const double* __restrict__ s_in, double den,
                             double* __restrict__ s_out) {
    const uint64_t M = hdr->maxv;
    hdr->M = M;
    hdr->div = make_udiv(M ? 2 * M : 1);
    const double s = *s_in;
    const double sm = M ? __dmul_rn(s, (double)M) : s;
    *s_out = ldexp(__ddiv_rn(sm, den), -7);
}

// ---------------------------------------------------------------- bilinear

// One block per output row (image b, row I); threads over the row's W*c elements.
template <int PASS>
__global__ void __launch_bounds__(kThreads) k_bil_fwd(const int8_t* __restrict__ x, int h, int w,
                                                      int c, int f, SqHdr* hdr,
                                                      int8_t* __restrict__ out) {
    const int H = (h - 1) * f + 1, W = (w - 1) * f + 1;
    const int row = blockIdx.x;
    const int b = row / H, I = row - b * H;
    const int i = I / f, r = I - i * f;
    const int i1 = i + 1 < h ? i + 1 : i;
    const int8_t* x0 = x + ((int64_t)b * h + i) * w * c;
    const int8_t* x1 = x + ((int64_t)b * h + i1) * w * c;
    int8_t* o = out + (int64_t)row * W * c;
    uint64_t M = 0;
    UDiv d;
    if (PASS == 1) {
        M = hdr->M;
        d = hdr->div;
    }
    uint32_t mx = 0;
    const int n_el = W * c;
    for (int e = threadIdx.x; e < n_el; e += blockDim.x) {
        const int J = e / c, ch = e - J * c;
        const int j = J / f, t = J - j * f;
        const int j1 = j + 1 < w ? j + 1 : j;
        const int v = (f - r) * (f - t) * (int)x0[j * c + ch] + r * (f - t) * (int)x1[j * c + ch] +
                      (f - r) * t * (int)x0[j1 * c + ch] + r * t * (int)x1[j1 * c + ch];
        if (PASS == 0) {
            uint32_t a = (uint32_t)(v < 0 ? -v : v);
            mx = a > mx ? a : mx;
        } else {
            o[e] = sq8_code(v, M, d);
        }
    }
    if (PASS == 0) {
        mx = warp_max_u32(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxv, (unsigned long long)mx);
    }
}

// Adjoint: one thread per input element; rows I in (f(i-1), f(i+1)) with weight
// f - |I - f i|, columns likewise.
__global__ void __launch_bounds__(kThreads) k_bil_bwd(const int8_t* __restrict__ e, int n, int h,
                                                      int w, int c, int f, SqHdr* hdr,
                                                      int32_t* __restrict__ acc) {
    const int H = (h - 1) * f + 1, W = (w - 1) * f + 1;
    const int64_t total = (int64_t)n * h * w * c;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    uint32_t mx = 0;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total; idx += stride) {
        const int ch = (int)(idx % c);
        const int64_t p = idx / c;
        const int j = (int)(p % w);
        const int64_t q = p / w;
        const int i = (int)(q % h);
        const int b = (int)(q / h);
        const int I0 = max(0, f * (i - 1) + 1), I1 = min(H - 1, f * (i + 1) - 1);
        const int J0 = max(0, f * (j - 1) + 1), J1 = min(W - 1, f * (j + 1) - 1);
        int sum = 0;
        for (int I = I0; I <= I1; I++) {
            const int wr = f - abs(I - f * i);
            const int8_t* er = e + (((int64_t)b * H + I) * W) * c + ch;
            int rs = 0;
            for (int J = J0; J <= J1; J++) rs += (f - abs(J - f * j)) * (int)er[(int64_t)J * c];
            sum += wr * rs;
        }
        acc[idx] = sum;
        uint32_t a = (uint32_t)(sum < 0 ? -sum : sum);
        mx = a > mx ? a : mx;
    }
    mx = warp_max_u32(mx);
    if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxv, (unsigned long long)mx);
}

__global__ void k_sq8_i32(const int32_t* __restrict__ acc, int64_t n, const SqHdr* hdr,
                          int8_t* __restrict__ out) {
    const uint64_t M = hdr->M;
    const UDiv d = hdr->div;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        out[i] = sq8_code(acc[i], M, d);
}

// ---------------------------------------------------------------- softmax head

// exp(t) for t <= 0 as a fixed fp32 sequence: k = floor(t log2e + 1/2), r = (t - k c1) - k c2
// (Cody & Waite; c1 holds the leading 15 bits of ln 2 so k c1 is exact), e^r by its Taylor
// polynomial of degree 7 (Horner), times 2^k.  No fused multiply-add anywhere.
__device__ __forceinline__ float exp_f32(float t) {
    if (!(t >= -87.0f)) return 0.0f;
    if (t > 0.0f) t = 0.0f;
    const float kf = floorf(__fadd_rn(__fmul_rn(t, 0x1.715476p+0f), 0.5f));
    const float r = __fsub_rn(__fsub_rn(t, __fmul_rn(kf, 0x1.62e4p-1f)), __fmul_rn(kf, 0x1.7f7d1cp-20f));
    float p = 0x1.a01a02p-13f;
    p = __fadd_rn(__fmul_rn(p, r), 0x1.6c16c2p-10f);
    p = __fadd_rn(__fmul_rn(p, r), 0x1.111112p-7f);
    p = __fadd_rn(__fmul_rn(p, r), 0x1.555556p-5f);
    p = __fadd_rn(__fmul_rn(p, r), 0x1.555556p-3f);
    p = __fadd_rn(__fmul_rn(p, r), 0.5f);
    p = __fadd_rn(__fmul_rn(p, r), 1.0f);
    p = __fadd_rn(__fmul_rn(p, r), 1.0f);
    const int k = (int)kf;
    if (k < -126) return 0.0f;
    return __fmul_rn(p, __int_as_float((k + 127) << 23));
}

// g_c of one pixel, recomputing e_c = exp(t_c) where it is needed (no per-class storage).
struct Pixel {
    const int8_t* z;
    int c, zm;
    float sf, S;
    __device__ void init(const int8_t* zp, int nc, float s) {
        z = zp; c = nc; sf = s;
        int m = -128;
        for (int ch = 0; ch < c; ch++) m = max(m, (int)z[ch]);
        zm = m;
        float acc = 0.0f;
        for (int ch = 0; ch < c; ch++) acc = __fadd_rn(acc, ex(ch));
        S = acc;
    }
    __device__ float ex(int ch) const {
        return exp_f32(__fmul_rn(__int2float_rn((int)z[ch] - zm), sf));
    }
    __device__ float g(int ch, int lab) const {
        const float p = __fdiv_rn(ex(ch), S);
        return ch == lab ? __fsub_rn(p, 1.0f) : p;
    }
};

template <int PASS>
__global__ void __launch_bounds__(kThreads) k_ce(const int8_t* __restrict__ z,
                                                 const double* __restrict__ s_z,
                                                 const uint8_t* __restrict__ labels, int64_t npix,
                                                 int c, int ignore, SqHdr* hdr,
                                                 int8_t* __restrict__ E) {
    const float sf = __double2float_rn(*s_z);
    float gmax = 0.0f;
    if (PASS == 1) gmax = __uint_as_float(hdr->gmax_bits);
    unsigned int mxb = 0;
    unsigned long long nv = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < npix; p += stride) {
        const int lab = labels[p];
        int8_t* ep = E + p * c;
        if (lab == ignore) {
            if (PASS == 1)
                for (int ch = 0; ch < c; ch++) ep[ch] = 0;
            continue;
        }
        Pixel px;
        px.init(z + p * c, c, sf);
        if (PASS == 0) {
            nv++;
            for (int ch = 0; ch < c; ch++) mxb = max(mxb, __float_as_uint(fabsf(px.g(ch, lab))));
        } else {
            for (int ch = 0; ch < c; ch++) {
                int q = 0;
                if (gmax != 0.0f) {
                    const float y = __fmul_rn(__fdiv_rn(px.g(ch, lab), gmax), 128.0f);
                    const float fl = floorf(y);
                    q = (int)fl + (__fsub_rn(y, fl) >= 0.5f ? 1 : 0);
                    q = q > 127 ? 127 : (q < -127 ? -127 : q);
                }
                ep[ch] = (int8_t)q;
            }
        }
    }
    if (PASS == 0) {
        mxb = warp_max_u32(mxb);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) nv += __shfl_xor_sync(0xffffffffu, nv, o);
        if ((threadIdx.x & 31) == 0) {
            if (mxb) atomicMax(&hdr->gmax_bits, mxb);
            if (nv) atomicAdd(&hdr->nvalid, nv);
        }
    }
}

__global__ void k_ce_params(const SqHdr* hdr, double* __restrict__ s_e,
                            int64_t* __restrict__ n_valid) {
    const float gmax = __uint_as_float(hdr->gmax_bits);
    const unsigned long long nv = hdr->nvalid;
    if (gmax == 0.0f)
        *s_e = __ddiv_rn(ldexp(1.0, -7), (double)(nv > 0 ? nv : 1));
    else
        *s_e = __ddiv_rn(ldexp((double)gmax, -7), (double)nv);
    if (n_valid) *n_valid = (int64_t)nv;
}

}  // namespace

}  // namespace iq

using namespace iq;

extern "C" iq_status iq_bilinear_workspace_size(int32_t n, int32_t h, int32_t w, int32_t c,
                                                size_t* bytes) {
    if (!bytes || n < 1 || h < 1 || w < 1 || c < 1) return IQ_ERR_INVALID_ARG;
    *bytes = 256 + (((size_t)n * h * w * c * 4 + 255) & ~size_t(255));
    return IQ_OK;
}

extern "C" iq_status iq_bilinear_up_fwd(const int8_t* x, const double* s_x, int32_t n, int32_t h,
                                        int32_t w, int32_t c, int32_t f, int8_t* out,
                                        double* s_out, void* ws, size_t ws_bytes,
                                        iq_stream stream) {
    if (!x || !s_x || !out || !s_out || n < 1 || h < 1 || w < 1 || c < 1 || f < 1 || f > 64)
        return IQ_ERR_INVALID_ARG;
    const int64_t H = (int64_t)(h - 1) * f + 1, W = (int64_t)(w - 1) * f + 1;
    if (W * c > INT32_MAX || (int64_t)n * H > INT32_MAX) return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < 256) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    SqHdr* hdr = (SqHdr*)ws;
    IQ_CUDA_CHECK(cudaMemsetAsync(hdr, 0, sizeof(SqHdr), st));
    const unsigned rows = (unsigned)(n * H);
    k_bil_fwd<0><<<rows, kThreads, 0, st>>>(x, h, w, c, f, hdr, out);
    IQ_LAUNCH_CHECK();
    k_sq8_params<<<1, 1, 0, st>>>(hdr, s_x, (double)(f * f), s_out);
    IQ_LAUNCH_CHECK();
    k_bil_fwd<1><<<rows, kThreads, 0, st>>>(x, h, w, c, f, hdr, out);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_bilinear_up_bwd(const int8_t* e, const double* s_e, int32_t n, int32_t h,
                                        int32_t w, int32_t c, int32_t f, int8_t* ex,
                                        double* s_ex, void* ws, size_t ws_bytes,
                                        iq_stream stream) {
    if (!e || !s_e || !ex || !s_ex || n < 1 || h < 1 || w < 1 || c < 1 || f < 1 || f > 64)
        return IQ_ERR_INVALID_ARG;
    const int64_t H = (int64_t)(h - 1) * f + 1, W = (int64_t)(w - 1) * f + 1;
    if (W * c > INT32_MAX || (int64_t)n * H > INT32_MAX) return IQ_ERR_INVALID_ARG;
    const int64_t total = (int64_t)n * h * w * c;
    size_t need = 0;
    iq_bilinear_workspace_size(n, h, w, c, &need);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    SqHdr* hdr = (SqHdr*)ws;
    int32_t* acc = (int32_t*)((char*)ws + 256);
    IQ_CUDA_CHECK(cudaMemsetAsync(hdr, 0, sizeof(SqHdr), st));
    k_bil_bwd<<<grid_for(total), kThreads, 0, st>>>(e, n, h, w, c, f, hdr, acc);
    IQ_LAUNCH_CHECK();
    k_sq8_params<<<1, 1, 0, st>>>(hdr, s_e, (double)(f * f), s_ex);
    IQ_LAUNCH_CHECK();
    k_sq8_i32<<<grid_for(total), kThreads, 0, st>>>(acc, total, hdr, ex);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_ce_grad(const int8_t* z, const double* s_z, const uint8_t* labels,
                                int64_t npix, int32_t c, int32_t ignore, int8_t* E, double* s_e,
                                int64_t* n_valid, void* ws, size_t ws_bytes, iq_stream stream) {
    if (!z || !s_z || !labels || !E || !s_e || npix < 0 || c < 1 || c > 1024)
        return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < 256) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    SqHdr* hdr = (SqHdr*)ws;
    IQ_CUDA_CHECK(cudaMemsetAsync(hdr, 0, sizeof(SqHdr), st));
    const int g = grid_for(npix > 0 ? npix : 1);
    if (npix > 0) {
        k_ce<0><<<g, kThreads, 0, st>>>(z, s_z, labels, npix, c, ignore, hdr, E);
        IQ_LAUNCH_CHECK();
    }
    k_ce_params<<<1, 1, 0, st>>>(hdr, s_e, n_valid);
    IQ_LAUNCH_CHECK();
    if (npix > 0) {
        k_ce<1><<<g, kThreads, 0, st>>>(z, s_z, labels, npix, c, ignore, hdr, E);
        IQ_LAUNCH_CHECK();
    }
    return IQ_OK;
}
