// iq_quant.cu -- the quantizers of Sec. 3.1 and the update of Sec. 3.3.3.
//
// Bandwidth-bound element-wise kernels: 16-byte loads where the layout allows,
// grid-stride loops over a grid of a few blocks per SM, warp-shuffle + one
// atomic per warp for the tensor-wide max |x| that Scale(x) needs.
#include "iq_internal.cuh"
#include "iq_tc_ptx.cuh"

#include <atomic>
#include <mutex>
#include <climits>

namespace iq {

static std::atomic<unsigned long long> g_launches{0};
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// The fourth Philox counter word of every stochastic rounding: 0 unless advanced on the device
// (iq_rq_epoch_advance), so that a captured training step replayed as a graph draws new
// random numbers on each replay.
static __device__ unsigned long long g_rq_epoch;
static std::mutex g_epoch_mu;
static unsigned long long* g_epoch_ptr[256] = {};

unsigned long long* rq_epoch_ptr() {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return nullptr;
    std::lock_guard<std::mutex> lock(g_epoch_mu);
    if (!g_epoch_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_rq_epoch) != cudaSuccess || !p) return nullptr;
        g_epoch_ptr[dev] = static_cast<unsigned long long*>(p);
    }
    return g_epoch_ptr[dev];
}

__global__ void k_epoch_update(unsigned long long* e, unsigned long long v, int set) {
    *e = set ? v : *e + v;
}

// ------------------------------------------------------------------ absmax

// max |x| of fp32 data as the bit pattern of |x| (non-negative floats order as
// their unsigned bit patterns).
__global__ void k_absmax_f32(const float* __restrict__ x, int64_t n, int relu,
                             unsigned* __restrict__ cell) {
    uint32_t m = 0;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    int64_t n4 = (((uintptr_t)x & 15) == 0) ? n / 4 : 0;
    const float4* x4 = reinterpret_cast<const float4*>(x);
    for (int64_t v = i; v < n4; v += stride) {
        float4 f = x4[v];
        float a[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
        for (int j = 0; j < 4; j++) {
            float t = relu ? fmaxf(a[j], 0.0f) : fabsf(a[j]);
            m = max(m, __float_as_uint(t));
        }
    }
    for (int64_t v = n4 * 4 + i; v < n; v += stride) {
        float t = relu ? fmaxf(x[v], 0.0f) : fabsf(x[v]);
        m = max(m, __float_as_uint(t));
    }
    m = warp_max_u32(m);
    if ((threadIdx.x & 31) == 0 && m) atomicMax(cell, m);
}

template <typename T>
__global__ void k_absmax_int(const T* __restrict__ q, int64_t n, int relu,
                             unsigned long long* __restrict__ cell) {
    uint64_t m = 0;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        int64_t v = (int64_t)q[i];
        if (relu && v < 0) v = 0;
        uint64_t a = (uint64_t)(v < 0 ? -v : v);
        m = a > m ? a : m;
    }
    m = warp_max_u64(m);
    if ((threadIdx.x & 31) == 0 && m) atomicMax(cell, (unsigned long long)m);
}

// ------------------------------------------------------------------ stores

__device__ __forceinline__ void store_code(void* out, int dtype, int64_t i, int64_t c) {
    if (dtype == IQ_I8) ((int8_t*)out)[i] = (int8_t)c;
    else if (dtype == IQ_I16) ((int16_t*)out)[i] = (int16_t)c;
    else ((int32_t*)out)[i] = (int32_t)c;
}

// ------------------------------------------------------------------ UQ / UQ2 / SQ on fp32

// Eq. (UQ): code = clip(floor(x 2^sh + 1/2)), sh = k-1 (UQ) or k-2 (2*UQ(x/2)).
__global__ void k_uq_f32(const float* __restrict__ x, int64_t n, int k, int sh,
                         void* __restrict__ out, int dtype) {
    const double p2 = ldexp(1.0, sh);
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        store_code(out, dtype, i, code_of(__dmul_rn((double)x[i], p2), k));
}

// Eq. (ScaleQ) on fp32: S = max|x| (cell, as bits); code = clip(rhu(x/S 2^(k-1)))
// with x/S formed in fp64 (its rhu equals that of the exact quotient).
__global__ void k_sq_f32(const float* __restrict__ x, int64_t n, int k, int relu,
                         const unsigned* __restrict__ cell, void* __restrict__ out, int dtype) {
    const float S = __uint_as_float(*cell);
    const double Sd = (double)S, p2 = ldexp(1.0, k - 1);
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        float v = relu ? fmaxf(x[i], 0.0f) : x[i];
        int64_t c = 0;
        if (S != 0.0f) c = code_of(__dmul_rn(__ddiv_rn((double)v, Sd), p2), k);
        store_code(out, dtype, i, c);
    }
}

__global__ void k_set_double(double* p, double v) { *p = v; }

__global__ void k_sq_f32_scale(const unsigned* __restrict__ cell, int k, double* s_out) {
    float S = __uint_as_float(*cell);
    *s_out = S != 0.0f ? ldexp((double)S, 1 - k) : ldexp(1.0, 1 - k);
}

// ------------------------------------------------------------------ SQ / RQ on integer codes


size_t requant_ws_bytes() { return 512; }

__global__ void k_rq_finalize(const unsigned long long* __restrict__ cell,
                              const double* __restrict__ s_in, int k, int mode,
                              RqParams* __restrict__ prm, double* __restrict__ s_out) {
    const RqParams p = rq_params_make(*cell, s_in ? *s_in : 1.0, k, mode);
    *prm = p;
    if (s_out) *s_out = p.s_out;
}

// SQ: code = floor((2^k (q + M) + M) / (2M)) - 2^(k-1), the non-negative shift of
// floor((2^k q + M) / (2M)); the numerator is < 2^(k+1) M + M < 2^57.  q is first clipped to
// [-M, M], which changes no code (both ends already give +-(2^(k-1) - 1)) and keeps the
// numerator non-negative when M is a frozen maximum that this tensor exceeds.
template <bool CLIP>
__device__ __forceinline__ int64_t sq_code(int64_t v, const RqParams& p, int k, int relu,
                                           int64_t lim) {
    if (relu && v < 0) v = 0;
    if (!p.M) return 0;
    if (CLIP) v = clamp64(v, -(int64_t)p.M, (int64_t)p.M);   // M not this tensor's maximum
    uint64_t num = ((uint64_t)(v + (int64_t)p.M) << k) + p.M;
    return clamp64((int64_t)udiv(num, p.div) - (int64_t(1) << (k - 1)), -lim, lim);
}

// SQ with k = 8 for int32 codes and 128 < M <= 2^31, in 32-bit arithmetic: with u = v + M
// in [0, 2M] the code is q - 128 for q = floor((256 u + M) / (2M)) = floor(128 u / M + 1/2).
// t = floor(u R8 / 2^32), R8 = floor(2^39 / M), lies in [floor(128 u / M) - 1,
// floor(128 u / M)], so q = t + [(2t + 1) M <= 256 u] + [(2t + 3) M <= 256 u] exactly (both
// sides below 2^41).  Clipping to +-127 is q in [1, 255]; the code byte is q ^ 0x80.
template <bool CLIP>
__device__ __forceinline__ uint32_t sq8_byte(int v, uint32_t M, uint32_t R8, int relu) {
    if (relu && v < 0) v = 0;
    // with an M that is not this tensor's maximum (frozen statistics) v is clipped to [-M, M]
    // first: u stays in [0, 2M] (M = 2^31 bounds every int32)
    if (CLIP && M < 0x80000000u) v = min(max(v, -(int)M), (int)M);
    const uint32_t u = (uint32_t)v + M;
    const uint32_t t = __umulhi(u, R8);
    const uint64_t rhs = (uint64_t)u << 8;
    const uint64_t l1 = (uint64_t)(2 * t + 1) * M;
    uint32_t q = t + (l1 <= rhs ? 1u : 0u) + (l1 + 2 * (uint64_t)M <= rhs ? 1u : 0u);
    q = q < 1u ? 1u : (q > 255u ? 255u : q);
    return q ^ 0x80u;
}

// 4 codes of sq8_byte, each decided in fp32 where that provably gives q = floor(128 u / M + 1/2)
// (u = v + M in [0, 2M]; the integer pipe, which sq8_byte's 64-bit comparisons saturate, is
// left mostly idle): u = 2^16 uh + ul with both halves exact in fp32 (the low mantissa bits
// of 2^23, by a mask or a byte permute), y = fl(uh 2^16 kq + fl(ul kq + 1/2)) with
// kq = fl(128 / M).  Against Y* = 128 u / M + 1/2 (u K <= 256, K = 128 / M): the kq rounding
// adds at most 256 2^-24 and each of the two fma roundings at most 257 2^-24, so
// |y - Y*| < 2^-14.  y clamped to [3/2, 255 + 1/2] (the clamp of q to [1, 255] commutes with
// the floor there), q = floor(y) and f = y - q exactly through y + 1.5 2^23 rounded
// downward (its low byte is q); q is taken when 2^-13 <= f < 1 - 2^-13, so Y* has the same
// floor.  Otherwise (about one element in four thousand) sq8_byte decides, under one branch
// per word.  The code byte is q ^ 0x80.
template <bool CLIP>
__device__ __forceinline__ uint32_t sq8_word_f(const int4& v, uint32_t M, uint32_t R8, float kq,
                                               int relu) {
    constexpr float MAG = 12582912.0f;                  // 1.5 2^23
    const int vs[4] = {v.x, v.y, v.z, v.w};
    uint32_t tb[4];
    bool ok[4];
#pragma unroll
    for (int j = 0; j < 4; j++) {
        int vv = vs[j];
        if (relu && vv < 0) vv = 0;
        if (CLIP && M < 0x80000000u) vv = min(max(vv, -(int)M), (int)M);
        const uint32_t u = (uint32_t)vv + M;
        const float fl = __int_as_float((int)(0x4B000000u | (u & 0xffffu))) - 8388608.0f;
        const float fh = __int_as_float((int)__byte_perm(u, 0x4B000000u, 0x7432)) - 8388608.0f;
        const float y = fminf(fmaxf(fmaf(fh * 65536.0f, kq, fmaf(fl, kq, 0.5f)), 1.5f), 255.5f);
        const float t = __fadd_rd(y, MAG);
        const float f = y - (t - MAG);
        tb[j] = __float_as_uint(t);
        ok[j] = f >= 0x1p-13f && f < 1.0f - 0x1p-13f;
    }
    uint32_t w = __byte_perm(__byte_perm(tb[0], tb[1], 0x0040), __byte_perm(tb[2], tb[3], 0x0040),
                             0x5410) ^ 0x80808080u;
    if (!(ok[0] && ok[1] && ok[2] && ok[3])) {
#pragma unroll
        for (int j = 0; j < 4; j++)
            if (!ok[j])
                w = (w & ~(0xffu << (8 * j))) | (sq8_byte<CLIP>(vs[j], M, R8, relu) << (8 * j));
    }
    return w;
}

// bytes 0xff where the 4 int8 codes of a are > 0 (nonzero with a clear sign bit), through
// prmt's sign-replicating selectors
__device__ __forceinline__ uint32_t pos_bytes(uint32_t a) {
    const uint32_t nz = ((a & 0x7f7f7f7fu) + 0x7f7f7f7fu) | a;
    uint32_t pn, sg;
    asm("prmt.b32 %0, %1, 0, 0xBA98;" : "=r"(pn) : "r"(nz));
    asm("prmt.b32 %0, %1, 0, 0xBA98;" : "=r"(sg) : "r"(a));
    return pn & ~sg;
}

// the fp16 copy of 4 codes (one 8-byte store) when the caller asked for it
__device__ __forceinline__ void put_f16x4(uint2* __restrict__ out16, int64_t i, uint32_t w) {
    if (out16) {
        uint2 h;
        tc::i8x4_to_f16x4(w, h.x, h.y);
        out16[i] = h;
    }
}

// int32 accumulators -> int8 codes, 4 per thread (16-byte loads, 4-byte stores), and
// optionally their fp16 copies.  MASK: the codes are zeroed where mask4's codes are not
// positive (a compile-time switch, so that the unmasked form carries no mask loads)
template <bool CLIP, bool MASK>
__global__ void k_sq_i32_i8x4(const int4* __restrict__ q, int64_t n4, int k, int relu,
                              const RqParams* __restrict__ prm, uint32_t* __restrict__ out,
                              uint2* __restrict__ out16, const uint32_t* __restrict__ mask4) {
    const RqParams p = *prm;
    const int64_t lim = qmax(k);
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    if (p.R8) {
        // four 16-byte loads in flight per thread
        const uint32_t M = (uint32_t)p.M;
        const float kq = p.kq;
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
             i += 4 * stride) {
            int4 v[4];
            uint32_t mk[4];
            // the mask words are loaded beside the sums, so that both are in flight at once
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const bool in = i + j * stride < n4;
                v[j] = in ? __ldg(q + i + j * stride) : make_int4(0, 0, 0, 0);
                if (MASK) mk[j] = in ? __ldg(mask4 + i + j * stride) : 0u;
            }
#pragma unroll
            for (int j = 0; j < 4; j++)
                if (i + j * stride < n4) {
                    uint32_t w = sq8_word_f<CLIP>(v[j], M, p.R8, kq, relu);
                    if (MASK) w &= pos_bytes(mk[j]);
                    out[i + j * stride] = w;
                    put_f16x4(out16, i + j * stride, w);
                }
        }
        return;
    }
    // two 16-byte loads in flight per thread
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += 2 * stride) {
        const int64_t i2 = i + stride;
        const int4 v = __ldg(q + i);
        const int4 v2 = i2 < n4 ? __ldg(q + i2) : make_int4(0, 0, 0, 0);
        const uint32_t mk = MASK ? __ldg(mask4 + i) : 0u;
        const uint32_t mk2 = MASK && i2 < n4 ? __ldg(mask4 + i2) : 0u;
        uint32_t w = ((uint32_t)sq_code<CLIP>(v.x, p, k, relu, lim) & 0xffu) |
                     (((uint32_t)sq_code<CLIP>(v.y, p, k, relu, lim) & 0xffu) << 8) |
                     (((uint32_t)sq_code<CLIP>(v.z, p, k, relu, lim) & 0xffu) << 16) |
                     (((uint32_t)sq_code<CLIP>(v.w, p, k, relu, lim) & 0xffu) << 24);
        if (MASK) w &= pos_bytes(mk);
        out[i] = w;
        put_f16x4(out16, i, w);
        if (i2 < n4) {
            uint32_t w2 = ((uint32_t)sq_code<CLIP>(v2.x, p, k, relu, lim) & 0xffu) |
                          (((uint32_t)sq_code<CLIP>(v2.y, p, k, relu, lim) & 0xffu) << 8) |
                          (((uint32_t)sq_code<CLIP>(v2.z, p, k, relu, lim) & 0xffu) << 16) |
                          (((uint32_t)sq_code<CLIP>(v2.w, p, k, relu, lim) & 0xffu) << 24);
            if (MASK) w2 &= pos_bytes(mk2);
            out[i2] = w2;
            put_f16x4(out16, i2, w2);
        }
    }
}

// the 4-code kernel over n codes (n % 4 == 0, aligned operands)
template <bool CLIP, bool MASK>
void sq_x4_launch(const void* q, int64_t n, int k, int relu, const RqParams* prm, void* out,
                  __half* out16, const int8_t* mask, cudaStream_t st) {
    k_sq_i32_i8x4<CLIP, MASK><<<grid_for(n / 4), kThreads, 0, st>>>(
        (const int4*)q, n / 4, k, relu, prm, (uint32_t*)out, (uint2*)out16,
        (const uint32_t*)mask);
}

template <typename T, bool CLIP>
__global__ void k_sq_int(const T* __restrict__ q, int64_t n, int k, int relu,
                         const RqParams* __restrict__ prm, void* __restrict__ out, int dtype) {
    const RqParams p = *prm;
    const int64_t lim = qmax(k);
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        int64_t v = (int64_t)q[i];
        if (relu && v < 0) v = 0;
        int64_t c = 0;
        if (p.M) {
            if (CLIP) v = clamp64(v, -(int64_t)p.M, (int64_t)p.M);
            uint64_t num = ((uint64_t)(v + (int64_t)p.M) << k) + p.M;
            c = (int64_t)udiv(num, p.div) - (int64_t(1) << (k - 1));
            c = clamp64(c, -lim, lim);
        }
        store_code(out, dtype, i, c);
    }
}

// RQ (Eqs. (SQ),(SR)): with num = (q + M) 2^(k-1) >= 0, f = floor(num/M) - 2^(k-1),
// rem = num mod M; round up iff u M < rem 2^32 for the element's Philox word u.
// One Philox block serves 8 consecutive elements.
template <typename T>
__global__ void k_rq_int(const T* __restrict__ q, int64_t n, int k,
                         const RqParams* __restrict__ prm, uint64_t seed, uint64_t layer,
                         uint64_t step, uint64_t tag, const unsigned long long* __restrict__ epoch,
                         void* __restrict__ out, int dtype) {
    const RqParams p = *prm;
    const uint64_t ep = *epoch;
    const int64_t nb = (n + 7) / 8;
    // 8 consecutive elements per thread: 16-byte loads and, for int8 codes, one 8-byte store
    const bool vec = ((((uintptr_t)q) & 15) == 0) && (dtype != IQ_I8 || (((uintptr_t)out) & 7) == 0);
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < nb; b += stride) {
        uint64_t w[4];
        philox4x64_10((uint64_t)b, step, tag, ep, seed, layer, w);
        const bool full = vec && b * 8 + 8 <= n;
        T v[8];
        if (full) {
            const uint4* src = reinterpret_cast<const uint4*>(q + b * 8);
#pragma unroll
            for (int j = 0; j < (int)(8 * sizeof(T) / 16); j++)
                reinterpret_cast<uint4*>(v)[j] = __ldg(src + j);
        } else {
#pragma unroll
            for (int j = 0; j < 8; j++) v[j] = b * 8 + j < n ? q[b * 8 + j] : T(0);
        }
        int64_t c8[8];
#pragma unroll
        for (int j = 0; j < 8; j++) {
            int64_t c = 0;
            if (p.M) {
                const uint64_t word = w[j >> 1];
                const uint32_t u = (j & 1) ? (uint32_t)(word >> 32) : (uint32_t)word;
                c = rq_code((int64_t)v[j], p.M, p.div, k, u);
            }
            c8[j] = c;
        }
        if (full && dtype == IQ_I8) {
            uint32_t lo = 0, hi = 0;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                lo |= ((uint32_t)c8[j] & 0xffu) << (8 * j);
                hi |= ((uint32_t)c8[4 + j] & 0xffu) << (8 * j);
            }
            reinterpret_cast<uint2*>(out)[b] = make_uint2(lo, hi);
        } else {
#pragma unroll
            for (int j = 0; j < 8; j++)
                if (b * 8 + j < n) store_code(out, dtype, b * 8 + j, c8[j]);
        }
    }
}

// x[i] = 0 where mask[i] <= 0, in place, and optionally the fp16 copy of the result (x16:
// n % 16 == 0, x, mask and x16 16-byte aligned, 8 codes a thread; else one code a thread)
__global__ void k_mask_inplace(int8_t* x, const int8_t* __restrict__ mask, int64_t n,
                               uint4* __restrict__ x16) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (x16) {
        for (int64_t v = i0; v < n / 8; v += stride) {
            uint2 c = reinterpret_cast<const uint2*>(x)[v];
            const uint2 m = reinterpret_cast<const uint2*>(mask)[v];
            c.x &= pos_bytes(m.x);
            c.y &= pos_bytes(m.y);
            reinterpret_cast<uint2*>(x)[v] = c;
            uint4 h;
            tc::i8x4_to_f16x4(c.x, h.x, h.y);
            tc::i8x4_to_f16x4(c.y, h.z, h.w);
            x16[v] = h;
        }
        return;
    }
    for (int64_t i = i0; i < n; i += stride)
        if (mask[i] <= 0) x[i] = 0;
}

iq_status requant_apply(const void* q, int in_dtype, int64_t n, const double* s_in, int k,
                        int mode, uint64_t seed, uint64_t layer, uint64_t step, uint64_t tag,
                        void* out, int out_dtype, double* s_out, void* ws, cudaStream_t st,
                        bool params_ready, bool clip, __half* out16, const int8_t* mask) {
    if ((out16 || mask) && (out_dtype != IQ_I8 || (mode != IQ_MODE_SQ && mode != IQ_MODE_SQ_RELU)))
        return IQ_ERR_INVALID_ARG;
    if (out16 && (!f16_copy_ok(out, out16, n) || ((uintptr_t)mask & 15)))
        return IQ_ERR_INVALID_ARG;
    unsigned long long* cell = (unsigned long long*)ws;
    RqParams* prm = rq_params_slot(ws);
    bool relu = mode == IQ_MODE_SQ_RELU;
    int g = grid_for(n);
    if (!params_ready) {
        k_rq_finalize<<<1, 1, 0, st>>>(cell, s_in, k, mode, prm, s_out);
        IQ_LAUNCH_CHECK();
    }
    if (n == 0) return IQ_OK;
    const double isz = in_dtype == IQ_I64 ? 8.0 : 4.0;
    const double osz = out_dtype == IQ_I8 ? 1.0 : (out_dtype == IQ_I16 ? 2.0 : 4.0);
    kt_pre(st);
    if (mode == IQ_MODE_SQ || mode == IQ_MODE_SQ_RELU) {
        const bool x4 = in_dtype == IQ_I32 && out_dtype == IQ_I8 && n % 4 == 0 &&
                        (((uintptr_t)q & 15) | ((uintptr_t)out & 3)) == 0;
        // the mask rides on the 4-wide kernel when its codes are 4-byte aligned
        const bool m4 = !mask || ((uintptr_t)mask & 3) == 0;
        if (x4 && m4) {
            using Launch = void (*)(const void*, int64_t, int, int, const RqParams*, void*,
                                    __half*, const int8_t*, cudaStream_t);
            const Launch f = clip ? (mask ? sq_x4_launch<true, true> : sq_x4_launch<true, false>)
                                  : (mask ? sq_x4_launch<false, true> : sq_x4_launch<false, false>);
            f(q, n, k, relu, prm, out, out16, mask, st);
        } else if (in_dtype == IQ_I32 && clip)
            k_sq_int<int32_t, true><<<g, kThreads, 0, st>>>((const int32_t*)q, n, k, relu, prm,
                                                            out, out_dtype);
        else if (in_dtype == IQ_I32)
            k_sq_int<int32_t, false><<<g, kThreads, 0, st>>>((const int32_t*)q, n, k, relu, prm,
                                                             out, out_dtype);
        else
            k_sq_int<int64_t, false><<<g, kThreads, 0, st>>>((const int64_t*)q, n, k, relu, prm,
                                                             out, out_dtype);
    } else {
        int gb = grid_for((n + 7) / 8);
        const unsigned long long* ep = rq_epoch_ptr();
        if (!ep) return IQ_ERR_CUDA;
        if (in_dtype == IQ_I32)
            k_rq_int<int32_t><<<gb, kThreads, 0, st>>>((const int32_t*)q, n, k, prm, seed, layer,
                                                       step, tag, ep, out, out_dtype);
        else
            k_rq_int<int64_t><<<gb, kThreads, 0, st>>>((const int64_t*)q, n, k, prm, seed, layer,
                                                       step, tag, ep, out, out_dtype);
    }
    IQ_LAUNCH_CHECK();
    const bool fused = (out16 || mask) && in_dtype == IQ_I32 && out_dtype == IQ_I8 &&
                       n % 4 == 0 && (((uintptr_t)q & 15) | ((uintptr_t)out & 3)) == 0 &&
                       (!mask || ((uintptr_t)mask & 3) == 0);
    kt_post_bytes(st, (mode == IQ_MODE_SQ || mode == IQ_MODE_SQ_RELU) ? IQ_KERNEL_SQ_CODES
                                                                       : IQ_KERNEL_RQ_CODES,
                  (double)n * (isz + osz + (fused && out16 ? 2.0 : 0.0) +
                               (fused && mask ? 1.0 : 0.0)));
    if ((out16 || mask) && !fused) {
        // the kernels without the fused mask / copy: one pass over the codes, in place
        return codes_mask_copy((int8_t*)out, mask, n, out16, st);
    }
    return IQ_OK;
}

iq_status codes_mask_copy(int8_t* x, const int8_t* mask, int64_t n, __half* x16,
                          cudaStream_t st) {
    if (n == 0 || (!mask && !x16)) return IQ_OK;
    if (!mask) return codes_to_f16(x, x16, n, st);
    k_mask_inplace<<<grid_for(x16 ? n / 8 : n), kThreads, 0, st>>>(x, mask, n, (uint4*)x16);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

iq_status requant_int(const void* q, int in_dtype, int64_t n, const double* s_in, int k,
                      int mode, uint64_t seed, uint64_t layer, uint64_t step, uint64_t tag,
                      void* out, int out_dtype, double* s_out, void* ws, cudaStream_t st) {
    unsigned long long* cell = (unsigned long long*)ws;
    bool relu = mode == IQ_MODE_SQ_RELU;
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, sizeof(unsigned long long), st));
    if (n > 0) {
        int g = grid_for(n);
        kt_pre(st);
        if (in_dtype == IQ_I32)
            k_absmax_int<int32_t><<<g, kThreads, 0, st>>>((const int32_t*)q, n, relu, cell);
        else
            k_absmax_int<int64_t><<<g, kThreads, 0, st>>>((const int64_t*)q, n, relu, cell);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_ABSMAX, (double)n * (in_dtype == IQ_I64 ? 8.0 : 4.0));
    }
    return requant_apply(q, in_dtype, n, s_in, k, mode, seed, layer, step, tag, out, out_dtype,
                         s_out, ws, st);
}

// ------------------------------------------------------------------ image input

// pixel/255 -> SQ8: code = floor((256 p + P) / (2P)) for P = max pixel.
__global__ void k_absmax_u8(const uint8_t* __restrict__ x, int64_t n, unsigned* cell) {
    uint32_t m = 0;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        m = max(m, (uint32_t)x[i]);
    m = warp_max_u32(m);
    if ((threadIdx.x & 31) == 0 && m) atomicMax(cell, m);
}

__global__ void k_image_sq8(const uint8_t* __restrict__ img, int32_t N, int32_t H, int32_t W,
                            int32_t Cin, int nchw, int32_t Cout, const unsigned* __restrict__ cell,
                            int8_t* __restrict__ out) {
    const uint32_t P = *cell;
    const int64_t total = (int64_t)N * H * W * Cout;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        int32_t c = (int32_t)(i % Cout);
        int64_t pix = i / Cout;
        int8_t code = 0;
        if (c < Cin && P) {
            int64_t w = pix % W, h = (pix / W) % H, nn = pix / ((int64_t)W * H);
            int64_t src = nchw ? ((nn * Cin + c) * H + h) * W + w : pix * Cin + c;
            uint32_t p = img[src];
            uint32_t v = (256u * p + P) / (2u * P);
            code = (int8_t)(v > 127u ? 127u : v);
        }
        out[i] = code;
    }
}

__global__ void k_image_scale(const unsigned* __restrict__ cell, double* s) {
    uint32_t P = *cell;
    *s = P ? ldexp(__ddiv_rn((double)P, 255.0), -7) : ldexp(1.0, -7);
}

// ------------------------------------------------------------------ weights and update

// Eq. (WQ1): wq = clip(floor((m + 2^(sh-1)) / 2^sh)), sh = k_u - k_w.
__global__ void k_weight_requant(const int32_t* __restrict__ m, int8_t* __restrict__ wq,
                                 int64_t n, int sh, int k_w) {
    const int64_t lim = qmax(k_w);
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        int64_t v = ((int64_t)m[i] + (int64_t(1) << (sh - 1))) >> sh;
        wq[i] = (int8_t)clamp64(v, -lim, lim);
    }
}

// Eq. (UQ2): dW = UQ(G_q lr, k_u) = clip(rhu(c s_g 2^(k_u-1-lr_log2))) (x2 grid: k_u-2),
// m <- clip(m - dW), then wq = UQ(W_m, k_w).  A gradient code takes one of 255 values,
// so each block first evaluates the fp64 product once per value (the same operations
// every element with that code would perform) into a shared-memory table.
__global__ void k_update(int32_t* __restrict__ master, int8_t* __restrict__ wq,
                         const int8_t* __restrict__ g, const double* __restrict__ s_g,
                         int64_t n, int sh, int k_u, int k_w) {
    __shared__ int32_t tab[256];
    {
        const double s = *s_g;
        const double p2 = ldexp(1.0, sh);
        for (int i = threadIdx.x; i < 255; i += blockDim.x)
            tab[i] = (int32_t)code_of(__dmul_rn(__dmul_rn((double)(i - 127), s), p2), k_u);
    }
    __syncthreads();
    const int64_t lu = qmax(k_u), lw = qmax(k_w);
    const int dsh = k_u - k_w;
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    auto one = [&](int32_t m, int8_t gv, int8_t& w) -> int32_t {
        const int64_t nm = clamp64((int64_t)m - tab[(int)gv + 127], -lu, lu);
        w = (int8_t)clamp64((nm + (int64_t(1) << (dsh - 1))) >> dsh, -lw, lw);
        return (int32_t)nm;
    };
    const bool vec = ((((uintptr_t)master | (uintptr_t)wq | (uintptr_t)g) & 15) == 0);
    const int64_t n4 = vec ? n / 4 : 0;
    // 4 parameters per thread: one 16-byte master load/store, 4-byte gradient and code words
    for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < n4; v += stride) {
        int4 m = reinterpret_cast<int4*>(master)[v];
        const uint32_t gw = reinterpret_cast<const uint32_t*>(g)[v];
        int8_t w0, w1, w2, w3;
        m.x = one(m.x, (int8_t)(gw & 0xffu), w0);
        m.y = one(m.y, (int8_t)((gw >> 8) & 0xffu), w1);
        m.z = one(m.z, (int8_t)((gw >> 16) & 0xffu), w2);
        m.w = one(m.w, (int8_t)(gw >> 24), w3);
        reinterpret_cast<int4*>(master)[v] = m;
        reinterpret_cast<uint32_t*>(wq)[v] = (uint32_t)(uint8_t)w0 | ((uint32_t)(uint8_t)w1 << 8) |
                                              ((uint32_t)(uint8_t)w2 << 16) | ((uint32_t)(uint8_t)w3 << 24);
    }
    for (int64_t i = n4 * 4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        int8_t w;
        master[i] = one(master[i], g[i], w);
        wq[i] = w;
    }
}

__global__ void k_relu_bwd(const int8_t* __restrict__ ea, const int8_t* __restrict__ a,
                           int64_t n, int8_t* __restrict__ e, uint2* __restrict__ e16) {
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e16) {
        // with the fp16 copy (n % 16 == 0, all aligned): 8 codes a thread, so that a warp's
        // 16-byte stores of the copy are contiguous
        const int64_t n8 = n / 8;
        for (int64_t v = i0; v < n8; v += stride) {
            const uint2 x = reinterpret_cast<const uint2*>(ea)[v];
            const uint2 m = reinterpret_cast<const uint2*>(a)[v];
            const uint32_t xs[2] = {x.x, x.y}, ms[2] = {m.x, m.y};
            uint32_t r[2];
#pragma unroll
            for (int j = 0; j < 2; j++) {
                uint32_t t = 0;
#pragma unroll
                for (int b = 0; b < 4; b++) {
                    const int8_t mv = (int8_t)(ms[j] >> (8 * b));
                    const uint32_t xv = (xs[j] >> (8 * b)) & 0xffu;
                    t |= (mv > 0 ? xv : 0u) << (8 * b);
                }
                r[j] = t;
            }
            reinterpret_cast<uint2*>(e)[v] = make_uint2(r[0], r[1]);
            uint4 h;
            tc::i8x4_to_f16x4(r[0], h.x, h.y);
            tc::i8x4_to_f16x4(r[1], h.z, h.w);
            reinterpret_cast<uint4*>(e16)[v] = h;
        }
        return;
    }
    bool vec = (((uintptr_t)ea | (uintptr_t)a | (uintptr_t)e) & 15) == 0;
    int64_t n16 = vec ? n / 16 : 0;
    for (int64_t v = i0; v < n16; v += stride) {
        int4 x = reinterpret_cast<const int4*>(ea)[v];
        int4 m = reinterpret_cast<const int4*>(a)[v];
        int xs[4] = {x.x, x.y, x.z, x.w}, ms[4] = {m.x, m.y, m.z, m.w};
#pragma unroll
        for (int j = 0; j < 4; j++) {
            uint32_t r = 0;
#pragma unroll
            for (int b = 0; b < 4; b++) {
                int8_t mv = (int8_t)(ms[j] >> (8 * b));
                uint32_t xv = ((uint32_t)xs[j] >> (8 * b)) & 0xffu;
                r |= (mv > 0 ? xv : 0u) << (8 * b);
            }
            xs[j] = (int)r;
        }
        reinterpret_cast<int4*>(e)[v] = make_int4(xs[0], xs[1], xs[2], xs[3]);
    }
    for (int64_t i = n16 * 16 + i0; i < n; i += stride) e[i] = a[i] > 0 ? ea[i] : 0;
}

// ------------------------------------------------------------------ per-channel Scale
// Eqs. (ScaleFactor),(ScaleQ) with the maximum taken over each channel instead of the whole
// tensor; q is viewed as [outer][C][inner] (channel-innermost NHWC: inner = 1).

// inner == 1: thread (x, y) owns channel 256 x + threadIdx.x and rows y, y + gridDim.y, ...
// (a warp reads 32 neighbouring channels of a row)
template <typename T>
__global__ void k_pc_max_c(const T* __restrict__ q, int64_t outer, int32_t C, int relu,
                           unsigned long long* __restrict__ M) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    uint64_t m = 0;
    for (int64_t o = blockIdx.y; o < outer; o += gridDim.y) {
        int64_t v = (int64_t)q[o * C + c];
        if (relu && v < 0) v = 0;
        const uint64_t a = (uint64_t)(v < 0 ? -v : v);
        m = a > m ? a : m;
    }
    if (m) atomicMax(M + c, (unsigned long long)m);
}

// inner > 1: one warp per row (o, c) of `inner` contiguous elements
template <typename T>
__global__ void k_pc_max_rows(const T* __restrict__ q, int64_t rows, int32_t C, int64_t inner,
                              int relu, unsigned long long* __restrict__ M) {
    const int lane = threadIdx.x & 31;
    const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t row = w0; row < rows; row += nw) {         // warp-uniform
        uint64_t m = 0;
        for (int64_t i = lane; i < inner; i += 32) {
            int64_t v = (int64_t)q[row * inner + i];
            if (relu && v < 0) v = 0;
            const uint64_t a = (uint64_t)(v < 0 ? -v : v);
            m = a > m ? a : m;
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            const uint64_t t = __shfl_xor_sync(0xffffffffu, m, o);
            m = t > m ? t : m;
        }
        if (lane == 0 && m) atomicMax(M + (row % C), (unsigned long long)m);
    }
}

// per channel: the divisor by 2 M_c and the output scale s_in M_c 2^(1-k)
__global__ void k_pc_params(const unsigned long long* __restrict__ M, int32_t C,
                            const double* __restrict__ s_in, int k, UDiv* __restrict__ div,
                            double* __restrict__ s_out) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    const uint64_t m = M[c];
    div[c] = make_udiv(m ? 2 * m : 1);
    s_out[c] = m ? ldexp(__dmul_rn(*s_in, (double)m), 1 - k) : ldexp(*s_in, 1 - k);
}

// code = clip(floor((2^k (v + M_c) + M_c) / (2 M_c)) - 2^(k-1)), 0 when M_c = 0
template <typename T>
__global__ void k_pc_codes(const T* __restrict__ q, int64_t n, int32_t C, int64_t inner, int k,
                           int relu, const unsigned long long* __restrict__ M,
                           const UDiv* __restrict__ div, void* __restrict__ out, int dtype) {
    const int64_t lim = qmax(k);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)((i / inner) % C);
        const uint64_t m = M[c];
        int64_t v = (int64_t)q[i];
        if (relu && v < 0) v = 0;
        int64_t code = 0;
        if (m) {
            const uint64_t num = ((uint64_t)(v + (int64_t)m) << k) + m;
            code = clamp64((int64_t)udiv(num, div[c]) - (int64_t(1) << (k - 1)), -lim, lim);
        }
        store_code(out, dtype, i, code);
    }
}

// decoupled L2 weight decay: m <- m - floor(m / 2^shift + 1/2), then W_q = UQ(W_m, k_w)
__global__ void k_weight_decay(int32_t* __restrict__ master, int8_t* __restrict__ wq, int64_t n,
                               int shift, int k_u, int k_w) {
    const int64_t lw = qmax(k_w);
    const int dsh = k_u - k_w;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = master[i];
        const int64_t nm = m - ((m + (int64_t(1) << (shift - 1))) >> shift);
        master[i] = (int32_t)nm;
        wq[i] = (int8_t)clamp64((nm + (int64_t(1) << (dsh - 1))) >> dsh, -lw, lw);
    }
}

size_t pc_ws_bytes(int32_t C) {
    return 256 + ((size_t)C * 8 + 255) / 256 * 256 + (size_t)C * sizeof(UDiv) + 256;
}

template <typename T>
iq_status pc_run(const T* q, int64_t outer, int32_t C, int64_t inner, const double* s_in, int k,
                 int relu, void* out, int dtype, double* s_out, void* ws, cudaStream_t st) {
    char* b = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    unsigned long long* M = (unsigned long long*)b;
    UDiv* div = (UDiv*)(b + ((size_t)C * 8 + 255) / 256 * 256);
    IQ_CUDA_CHECK(cudaMemsetAsync(M, 0, (size_t)C * 8, st));
    const int64_t n = outer * C * inner;
    if (n > 0) {
        if (inner == 1) {
            const unsigned gx = (unsigned)((C + kThreads - 1) / kThreads);
            int64_t gy = (152 * 8 + gx - 1) / gx;
            if (gy > outer) gy = outer;
            if (gy > 65535) gy = 65535;
            k_pc_max_c<T><<<dim3(gx, (unsigned)gy), kThreads, 0, st>>>(q, outer, C, relu, M);
        } else {
            k_pc_max_rows<T><<<grid_for(outer * C * 32), kThreads, 0, st>>>(q, outer * C, C,
                                                                            inner, relu, M);
        }
        IQ_LAUNCH_CHECK();
    }
    k_pc_params<<<(C + kThreads - 1) / kThreads, kThreads, 0, st>>>(M, C, s_in, k, div, s_out);
    IQ_LAUNCH_CHECK();
    if (n > 0) {
        k_pc_codes<T><<<grid_for(n), kThreads, 0, st>>>(q, n, C, inner, k, relu, M, div, out,
                                                        dtype);
        IQ_LAUNCH_CHECK();
    }
    return IQ_OK;
}

}  // namespace iq

using namespace iq;

// ==================================================================== C ABI

extern "C" const char* iq_status_str(iq_status s) {
    switch (s) {
        case IQ_OK: return "ok";
        case IQ_ERR_INVALID_ARG: return "invalid argument";
        case IQ_ERR_UNSUPPORTED: return "unsupported";
        case IQ_ERR_WORKSPACE: return "workspace too small";
        case IQ_ERR_OVERFLOW_RISK: return "int32 accumulation could overflow";
        case IQ_ERR_TIMEOUT: return "device wait timed out";
        case IQ_ERR_CUDA: return "CUDA error";
    }
    return "unknown status";
}

extern "C" int iq_version(void) { return 1; }

extern "C" unsigned long long iq_launch_count(void) { return g_launches.load(); }

extern "C" iq_status iq_rq_epoch_advance(iq_stream stream) {
    unsigned long long* e = iq::rq_epoch_ptr();
    if (!e) return IQ_ERR_CUDA;
    iq::k_epoch_update<<<1, 1, 0, (cudaStream_t)stream>>>(e, 1ull, 0);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_rq_epoch_set(uint64_t value, iq_stream stream) {
    unsigned long long* e = iq::rq_epoch_ptr();
    if (!e) return IQ_ERR_CUDA;
    iq::k_epoch_update<<<1, 1, 0, (cudaStream_t)stream>>>(e, (unsigned long long)value, 1);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_quantize_workspace_size(int64_t n, size_t* bytes) {
    if (!bytes || n < 0) return IQ_ERR_INVALID_ARG;
    *bytes = requant_ws_bytes();
    return IQ_OK;
}

static bool dtype_holds(int dtype, int k) {
    return (dtype == IQ_I8 && k <= 8) || (dtype == IQ_I16 && k <= 16) ||
           (dtype == IQ_I32 && k <= 24);
}

extern "C" iq_status iq_quantize(const float* x, int64_t n, int k, int mode, int out_dtype,
                                 void* codes, double* scale, void* ws, size_t ws_bytes,
                                 iq_stream stream) {
    cudaStream_t st = (cudaStream_t)stream;
    if (n < 0 || (n > 0 && (!x || !codes)) || k < 2) return IQ_ERR_INVALID_ARG;
    if (!dtype_holds(out_dtype, k)) return IQ_ERR_INVALID_ARG;
    if (mode == IQ_MODE_UQ || mode == IQ_MODE_UQ2) {
        if (k > 24) return IQ_ERR_INVALID_ARG;
        if (n > 0) {
            k_uq_f32<<<grid_for(n), kThreads, 0, st>>>(x, n, k, mode == IQ_MODE_UQ ? k - 1 : k - 2,
                                                        codes, out_dtype);
            IQ_LAUNCH_CHECK();
        }
        if (scale) {
            k_set_double<<<1, 1, 0, st>>>(scale, ldexp(1.0, mode == IQ_MODE_UQ ? 1 - k : 2 - k));
            IQ_LAUNCH_CHECK();
        }
        return IQ_OK;
    }
    if (mode != IQ_MODE_SQ && mode != IQ_MODE_SQ_RELU) return IQ_ERR_INVALID_ARG;
    if (k > 16 || !scale) return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < requant_ws_bytes()) return IQ_ERR_WORKSPACE;
    unsigned* cell = (unsigned*)ws;
    int relu = mode == IQ_MODE_SQ_RELU;
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, sizeof(unsigned), st));
    if (n > 0) {
        k_absmax_f32<<<grid_for(n / 4 + 1), kThreads, 0, st>>>(x, n, relu, cell);
        IQ_LAUNCH_CHECK();
        k_sq_f32<<<grid_for(n), kThreads, 0, st>>>(x, n, k, relu, cell, codes, out_dtype);
        IQ_LAUNCH_CHECK();
    }
    k_sq_f32_scale<<<1, 1, 0, st>>>(cell, k, scale);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_quantize_image_u8(const uint8_t* img, int32_t n, int32_t h, int32_t w,
                                          int32_t c, int nchw, int32_t c_out, int8_t* codes,
                                          double* scale, void* ws, size_t ws_bytes,
                                          iq_stream stream) {
    cudaStream_t st = (cudaStream_t)stream;
    if (!img || !codes || !scale || n <= 0 || h <= 0 || w <= 0 || c <= 0 || c_out < c)
        return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < requant_ws_bytes()) return IQ_ERR_WORKSPACE;
    unsigned* cell = (unsigned*)ws;
    int64_t nin = (int64_t)n * h * w * c;
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, sizeof(unsigned), st));
    k_absmax_u8<<<grid_for(nin), kThreads, 0, st>>>(img, nin, cell);
    IQ_LAUNCH_CHECK();
    k_image_sq8<<<grid_for((int64_t)n * h * w * c_out), kThreads, 0, st>>>(img, n, h, w, c, nchw,
                                                                           c_out, cell, codes);
    IQ_LAUNCH_CHECK();
    k_image_scale<<<1, 1, 0, st>>>(cell, scale);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_requantize(const void* q, int in_dtype, int64_t n, const double* s_in,
                                   int k, int mode, uint64_t seed, uint64_t layer, uint64_t step,
                                   uint64_t tag, void* codes, int out_dtype, double* s_out,
                                   void* ws, size_t ws_bytes, iq_stream stream) {
    if (n < 0 || (n > 0 && (!q || !codes)) || !s_out) return IQ_ERR_INVALID_ARG;
    if (in_dtype != IQ_I32 && in_dtype != IQ_I64) return IQ_ERR_INVALID_ARG;
    if (k < 2 || k > 16 || !dtype_holds(out_dtype, k)) return IQ_ERR_INVALID_ARG;
    if (mode < IQ_MODE_SQ || mode > IQ_MODE_RQ_GQ2) return IQ_ERR_INVALID_ARG;
    if (mode != IQ_MODE_RQ_GQ2 && !s_in) return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < requant_ws_bytes()) return IQ_ERR_WORKSPACE;
    return requant_int(q, in_dtype, n, s_in, k, mode, seed, layer, step, tag, codes, out_dtype,
                       s_out, ws, (cudaStream_t)stream);
}

extern "C" iq_status iq_requantize_per_channel_workspace_size(int32_t c, size_t* bytes) {
    if (!bytes || c <= 0) return IQ_ERR_INVALID_ARG;
    *bytes = pc_ws_bytes(c);
    return IQ_OK;
}

extern "C" iq_status iq_requantize_per_channel(const void* q, int in_dtype, int64_t outer,
                                               int32_t c, int64_t inner, const double* s_in,
                                               int k, int relu, void* codes, int out_dtype,
                                               double* s_out, void* ws, size_t ws_bytes,
                                               iq_stream stream) {
    if (outer < 0 || inner < 1 || c <= 0 || !s_in || !s_out) return IQ_ERR_INVALID_ARG;
    if (outer > 0 && (!q || !codes)) return IQ_ERR_INVALID_ARG;
    if (in_dtype != IQ_I32 && in_dtype != IQ_I64) return IQ_ERR_INVALID_ARG;
    if (k < 2 || k > 16 || !dtype_holds(out_dtype, k)) return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < pc_ws_bytes(c)) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    if (in_dtype == IQ_I32)
        return pc_run((const int32_t*)q, outer, c, inner, s_in, k, relu, codes, out_dtype, s_out,
                      ws, st);
    return pc_run((const int64_t*)q, outer, c, inner, s_in, k, relu, codes, out_dtype, s_out, ws,
                  st);
}

extern "C" iq_status iq_weight_decay(int32_t* master, int8_t* wq, int64_t n, int shift,
                                     int k_u, int k_w, iq_stream stream) {
    if (!master || !wq || n < 0 || shift < 1 || shift > 40 || k_w < 2 || k_w > 8 ||
        k_u <= k_w || k_u > 31)
        return IQ_ERR_INVALID_ARG;
    if (n == 0) return IQ_OK;
    k_weight_decay<<<grid_for(n), kThreads, 0, (cudaStream_t)stream>>>(master, wq, n, shift, k_u,
                                                                       k_w);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_weight_requant(const int32_t* master, int8_t* wq, int64_t n, int k_u,
                                       int k_w, iq_stream stream) {
    if (!master || !wq || n < 0 || k_w < 2 || k_w > 8 || k_u <= k_w || k_u > 31)
        return IQ_ERR_INVALID_ARG;
    if (n == 0) return IQ_OK;
    k_weight_requant<<<grid_for(n), kThreads, 0, (cudaStream_t)stream>>>(master, wq, n, k_u - k_w,
                                                                          k_w);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_update(int32_t* master, int8_t* wq, const int8_t* g, const double* s_g,
                               int64_t n, int lr_log2, int k_u, int k_w, int x2,
                               iq_stream stream) {
    if (!master || !wq || !g || !s_g || n < 0 || k_w < 2 || k_w > 8 || k_u <= k_w || k_u > 31)
        return IQ_ERR_INVALID_ARG;
    if (lr_log2 < 0 || lr_log2 > 60) return IQ_ERR_INVALID_ARG;
    if (n == 0) return IQ_OK;
    int sh = (x2 ? k_u - 2 : k_u - 1) - lr_log2;
    k_update<<<grid_for(n / 4 + 1, kThreads, 152 * 8), kThreads, 0, (cudaStream_t)stream>>>(
        master, wq, g, s_g, n, sh, k_u, k_w);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_relu_bwd(const int8_t* e_a, const int8_t* a, int64_t n, int8_t* e,
                                 void* e_f16, iq_stream stream) {
    if (!e_a || !a || !e || n < 0) return IQ_ERR_INVALID_ARG;
    // the fp16 copy rides on the 16-code vector loop: every operand 16-byte aligned
    if (e_f16 && (!f16_copy_ok(e, e_f16, n) || (((uintptr_t)e_a | (uintptr_t)a) & 15)))
        return IQ_ERR_INVALID_ARG;
    if (n == 0) return IQ_OK;
    k_relu_bwd<<<grid_for(n / 16 + 1), kThreads, 0, (cudaStream_t)stream>>>(e_a, a, n, e,
                                                                           (uint2*)e_f16);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}
