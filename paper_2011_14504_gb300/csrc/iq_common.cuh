// iq_common.cuh -- device helpers shared by the kernels of the iq library.
//
// Everything here is integer-exact or IEEE fp64 with explicit round-to-nearest
// intrinsics (no FMA contraction), so that the scale metadata follows one fixed
// operation order on every run.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/iq.h"

namespace iq {

typedef __int128 i128;
typedef unsigned __int128 u128;

constexpr int kThreads = 256;

__host__ __device__ inline int64_t qmax(int k) { return (int64_t(1) << (k - 1)) - 1; }

__device__ __forceinline__ int64_t clamp64(int64_t v, int64_t lo, int64_t hi) {
    return v < lo ? lo : (v > hi ? hi : v);
}

// int64 -> fp32 through the two 32-bit halves of |v| (64-bit conversions run on the narrow
// FP64 pipe of this part): |v| = hi 2^32 + lo with hi < 2^24 (|v| < 2^56) is exact in
// hi 2^32, so fma(hi, 2^32, fl(lo)) is fl(lo) when hi = 0 and otherwise within
// 2^8 + u |v| <= 2u |v| of |v| (u = 2^-24): a relative error of at most 2u.
__device__ __forceinline__ float f32_of_i64(long long v) {
    const unsigned long long a = (unsigned long long)(v < 0 ? -v : v);
    const float f = fmaf((float)(uint32_t)(a >> 32), 0x1p32f, __uint2float_rn((uint32_t)a));
    return v < 0 ? -f : f;
}
// an fp32 upper bound of |v|
__device__ __forceinline__ float f32_abs_up(long long v) {
    const unsigned long long a = (unsigned long long)(v < 0 ? -v : v);
    return __fmaf_ru(__uint2float_ru((uint32_t)(a >> 32)), 0x1p32f,
                     __uint2float_ru((uint32_t)a));
}

// floor(y + 1/2) (the rounding of Eq. (UQ)) on an fp64 value: y - floor(y) is
// exact, so comparing it with 1/2 never rounds.
__device__ __forceinline__ double rhu(double y) {
    double f = floor(y);
    return __dadd_rn(f, (__dsub_rn(y, f) >= 0.5) ? 1.0 : 0.0);
}

// rhu clipped to the symmetric k-bit grid; NaN -> 0.
__device__ __forceinline__ int64_t code_of(double y, int k) {
    if (y != y) return 0;
    double lim = (double)qmax(k);
    double r = rhu(y);
    r = r > lim ? lim : r;
    r = r < -lim ? -lim : r;
    return (int64_t)r;
}

// Exact floor(n / d) for 64-bit unsigned n and a fixed divisor 1 <= d < 2^63,
// by multiplication (Granlund & Montgomery, "Division by invariant integers
// using multiplication", PLDI 1994, Sec. 4): with l = ceil(log2 d),
// m' = floor(2^64 (2^l - d) / d) + 1, t = mulhi(m', n),
// q = (t + ((n - t) >> min(l,1))) >> max(l-1, 0).
struct UDiv {
    uint64_t mp;
    int32_t sh1, sh2;
    uint64_t d;
};

__host__ __device__ inline UDiv make_udiv(uint64_t d) {
    int l = 0;
    while (l < 64 && (uint64_t(1) << l) < d) l++;
    UDiv u;
    u128 num = (u128)((l == 64 ? u128(0) : (u128(1) << l)) - d) << 64;
    u.mp = (uint64_t)(num / d) + 1;
    u.sh1 = l < 1 ? l : 1;
    u.sh2 = l - 1 > 0 ? l - 1 : 0;
    u.d = d;
    return u;
}

__device__ __forceinline__ uint64_t udiv(uint64_t n, const UDiv& u) {
    uint64_t t = __umul64hi(u.mp, n);
    return (t + ((n - t) >> u.sh1)) >> u.sh2;
}

// RQ_k of one integer code v (Eqs. (SQ),(SR)) with M = max|v| > 0 and div = the divisor by M:
// f = floor((v + M) 2^(k-1) / M), rem the remainder; up iff u M < rem 2^32 for the element's
// 32-bit random word u, i.e. floor(u M / 2^32) < rem, evaluated as u Mh + umulhi(u, Ml) with
// M = Mh 2^32 + Ml.  Returns the clipped code.
__device__ __forceinline__ int64_t rq_code(int64_t v, uint64_t M, const UDiv& div, int k,
                                           uint32_t u) {
    const uint64_t num = (uint64_t)(v + (int64_t)M) << (k - 1);
    const uint64_t fq = udiv(num, div);
    const uint64_t rem = num - fq * M;
    const uint64_t hi = (uint64_t)u * (M >> 32) + __umulhi(u, (uint32_t)M);
    const int64_t c = (int64_t)fq - (int64_t(1) << (k - 1)) + (hi < rem ? 1 : 0);
    return clamp64(c, -qmax(k), qmax(k));
}

// A tensor-wide max |q| together with the divisor derived from it.
struct RqDiv {
    uint64_t M;
    UDiv div;
};

// Correctly rounded (nearest-even) conversion of a 128-bit unsigned integer to
// fp64: keep the top 64 bits plus a sticky bit, convert those (the 11 extra
// bits decide the rounding exactly as the full value would), rescale by 2^s.
__device__ inline double u128_to_double(u128 v) {
    uint64_t hi = (uint64_t)(v >> 64);
    if (hi == 0) return __ull2double_rn((uint64_t)v);
    int s = 64 - __clzll((long long)hi);  // bits above the low 64
    uint64_t top = (uint64_t)(v >> s);
    uint64_t mask = s >= 64 ? ~uint64_t(0) : ((uint64_t(1) << s) - 1);
    uint64_t rest = (uint64_t)v & mask;
    top |= (rest != 0);
    return ldexp(__ull2double_rn(top), s);
}

// Philox4x64-10 (Salmon et al., SC'11): counter (4 x 64) and key (2 x 64).
__device__ __forceinline__ void philox4x64_10(uint64_t c0, uint64_t c1, uint64_t c2,
                                              uint64_t c3, uint64_t k0, uint64_t k1,
                                              uint64_t out[4]) {
    const uint64_t M0 = 0xD2E7470EE14C6C93ULL, M1 = 0xCA5A826395121157ULL;
    const uint64_t W0 = 0x9E3779B97F4A7C15ULL, W1 = 0xBB67AE8584CAA73BULL;
#pragma unroll
    for (int r = 0; r < 10; r++) {
        uint64_t hi0 = __umul64hi(M0, c0), lo0 = M0 * c0;
        uint64_t hi1 = __umul64hi(M1, c2), lo1 = M1 * c2;
        uint64_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
        k0 += W0; k1 += W1;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

__device__ __forceinline__ int warp_max_i32(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        uint64_t w = __shfl_xor_sync(0xffffffffu, v, o);
        v = w > v ? w : v;
    }
    return v;
}
__device__ __forceinline__ uint32_t warp_max_u32(uint32_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// grid size for an elementwise pass: enough blocks to fill 152 SMs several times
inline int grid_for(int64_t work_items, int threads = kThreads, int max_blocks = 152 * 16) {
    int64_t b = (work_items + threads - 1) / threads;
    if (b < 1) b = 1;
    if (b > max_blocks) b = max_blocks;
    return (int)b;
}

// Host-side bump allocator over the caller's workspace (256-byte aligned slices).
struct WsCursor {
    char* base;
    size_t cap, off;
    explicit WsCursor(void* p, size_t c) : base((char*)p), cap(c), off(0) {}
    template <typename T>
    T* take(size_t n) {
        size_t o = (off + 255) & ~size_t(255);
        off = o + n * sizeof(T);
        return base ? (T*)(base + o) : nullptr;
    }
    bool ok() const { return off <= cap; }
};

}  // namespace iq

#define IQ_CUDA_CHECK(expr)                                  \
    do {                                                     \
        cudaError_t e_ = (expr);                             \
        if (e_ != cudaSuccess) return IQ_ERR_CUDA;           \
    } while (0)

namespace iq {
// number of kernels this library has enqueued (host-side count, for diagnostics)
void count_launch();
}  // namespace iq

#define IQ_LAUNCH_CHECK()                 \
    do {                                  \
        iq::count_launch();               \
        IQ_CUDA_CHECK(cudaGetLastError()); \
    } while (0)
