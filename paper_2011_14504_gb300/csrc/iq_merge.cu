// iq_merge.cu -- quantized sums and concatenations, spatial sums and channel slices:
// the tensor joins of DeepLabv3-ResNet50 (bottleneck residual adds, the sums of the
// errors that reach one tensor, the ASPP concatenation and its image-pooling branch).
//
// The paper (Sec. 5) runs DeepLabv3 fully quantized but does not say how its joins are
// quantized; here each join evaluates the real-valued operation on the codes and then
// applies Q_A / Q_E = SQ(., 8) (Eq. (ScaleQ) with Scale = max|.| of the whole tensor).
#include <algorithm>
#include <climits>

#include "iq_internal.cuh"
#include "iq_stream.cuh"

namespace iq {

namespace {

struct TermDev {
    const void* codes;
    const double* scale;
    const int32_t* gamma;
    const int32_t* beta;
    int32_t is16, c, c_offset, bcast, k_gamma, k_beta, base;   // base: first table row
};

struct Terms {
    TermDev t[IQ_MAX_TERMS];
    int32_t n;
};

// Workspace: [0,256) header (max cell, shift P, output parameters), then F and B tables.
struct CombHdr {
    unsigned long long maxz;
    int32_t P;
    int32_t pad;
    uint64_t M;
    UDiv div;
    float kq;      // fl(128 / M) (0 when M = 0)
    float c130;    // 130 / M rounded up
    unsigned long long bound[IQ_MAX_TERMS];   // per operand max_ch(|a| vmax + |b|), as bits
};
static_assert(sizeof(CombHdr) <= 256, "the join header fits its 256 bytes");

__device__ __forceinline__ double term_a(const TermDev& t, double s, int ch) {
    if (!t.gamma) return s;
    return __dmul_rn(__dmul_rn((double)t.gamma[ch], ldexp(1.0, 2 - t.k_gamma)), s);
}
__device__ __forceinline__ double term_b(const TermDev& t, int ch) {
    return t.beta ? __dmul_rn((double)t.beta[ch], ldexp(1.0, 2 - t.k_beta)) : 0.0;
}

// The tables, over ceil(c / 64) x operands blocks of 64 threads (the fp64 pipe of one SM is
// narrow).  Stage 1: per operand the bound max_ch(|a| vmax + |b|), kept as the bit pattern
// of a non-negative double (such doubles order as their bits; the cells are zeroed first).
constexpr int kTabThreads = 64;

__global__ void __launch_bounds__(kTabThreads) k_comb_bound(Terms T, CombHdr* hdr) {
    const TermDev& t = T.t[blockIdx.y];
    const int ch = blockIdx.x * blockDim.x + threadIdx.x;
    double v = 0.0;
    if (ch < t.c) {
        const double vmax = t.is16 ? 32767.0 : 127.0;
        v = __dadd_rn(__dmul_rn(fabs(term_a(t, *t.scale, ch)), vmax), fabs(term_b(t, ch)));
    }
    const uint64_t m = warp_max_u64((uint64_t)__double_as_longlong(v));
    if ((threadIdx.x & 31) == 0 && m) atomicMax(&hdr->bound[blockIdx.y], (unsigned long long)m);
}

// Stage 2: the shift P from the bounds' sum (in operand order), then F = rhu(a 2^P) and
// B = rhu(b 2^P); block (0, 0) publishes P and clears the max cell of the join's first pass.
__global__ void __launch_bounds__(kTabThreads) k_comb_tab(Terms T, CombHdr* hdr, long long* F,
                                                          long long* B) {
    double bound = 0.0;
    for (int i = 0; i < T.n; i++)
        bound = __dadd_rn(bound, __longlong_as_double((long long)hdr->bound[i]));
    int e;
    frexp(__dadd_rn(bound, 1.0), &e);
    int P = 50 - e;
    if (P > 62) P = 62;
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) {
        hdr->P = P;
        hdr->maxz = 0ull;
    }
    const TermDev& t = T.t[blockIdx.y];
    const int ch = blockIdx.x * blockDim.x + threadIdx.x;
    if (ch >= t.c) return;
    const double s = *t.scale;
    F[t.base + ch] = (long long)rhu(ldexp(term_a(t, s, ch), P));
    B[t.base + ch] = (long long)rhu(ldexp(term_b(t, ch), P));
}

__device__ __forceinline__ int64_t load_code(const TermDev& t, int64_t idx) {
    return t.is16 ? (int64_t)((const int16_t*)t.codes)[idx] : (int64_t)((const int8_t*)t.codes)[idx];
}

// Pass 0: max |z| over the tensor.  Pass 1: the SQ(., 8) codes.
template <int PASS>
__global__ void __launch_bounds__(kThreads) k_comb(Terms T, int concat, int64_t n, int64_t hw,
                                                   int c_out, int relu,
                                                   const long long* __restrict__ F,
                                                   const long long* __restrict__ B,
                                                   CombHdr* hdr, int8_t* __restrict__ out,
                                                   UDiv dc, UDiv dhw) {
    uint64_t M = 0;
    UDiv d2m;
    if (PASS == 1) {
        M = hdr->M;
        d2m = hdr->div;
    }
    const int64_t total = n * hw * (int64_t)c_out;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    uint64_t mx = 0;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += stride) {
        const int64_t pix = (int64_t)udiv((uint64_t)e, dc);
        const int co = (int)(e - pix * c_out);
        const int64_t img = (int64_t)udiv((uint64_t)pix, dhw);
        int64_t z = 0;
#pragma unroll
        for (int i = 0; i < IQ_MAX_TERMS; i++) {
            if (i >= T.n) break;
            const TermDev& t = T.t[i];
            int ch = co;
            if (concat) {
                ch = co - t.c_offset;
                if (ch < 0 || ch >= t.c) continue;
            }
            const int64_t idx = t.bcast ? img * t.c + ch : pix * t.c + ch;
            z += (int64_t)F[t.base + ch] * load_code(t, idx) + (int64_t)B[t.base + ch];
        }
        if (relu && z < 0) z = 0;
        if (PASS == 0) {
            uint64_t a = (uint64_t)(z < 0 ? -z : z);
            mx = a > mx ? a : mx;
        } else {
            int64_t c = 0;
            if (M) {
                uint64_t num = ((uint64_t)(z + (int64_t)M) << 8) + M;
                c = clamp64((int64_t)udiv(num, d2m) - 128, -127, 127);
            }
            out[e] = (int8_t)c;
        }
    }
    if (PASS == 0) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxz, (unsigned long long)mx);
    }
}

// The same two passes, 8 channels per thread: every operand's channel count and offset
// and c_out are multiples of 8 and the code pointers aligned, so each operand contributes
// one 8-byte (int8) or 16-byte (int16) load and its F / B rows four 16-byte loads.
__device__ __forceinline__ void load8(const TermDev& t, int64_t idx, int32_t v[8]) {
    if (t.is16) {
        const int4 q = __ldg(reinterpret_cast<const int4*>((const int16_t*)t.codes + idx));
        const int w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; j++) {
            v[2 * j] = (int32_t)(int16_t)(w[j] & 0xffff);
            v[2 * j + 1] = (int32_t)(w[j] >> 16);
        }
    } else {
        const int2 q = __ldg(reinterpret_cast<const int2*>((const int8_t*)t.codes + idx));
        const int w[2] = {q.x, q.y};
#pragma unroll
        for (int j = 0; j < 8; j++) v[j] = (int32_t)(int8_t)((w[j >> 2] >> (8 * (j & 3))) & 0xff);
    }
}

template <int PASS>
__global__ void __launch_bounds__(kThreads) k_comb8(Terms T, int concat, int64_t nvec, int cgs,
                                                    int relu, const long long* __restrict__ F,
                                                    const long long* __restrict__ B,
                                                    CombHdr* hdr, int8_t* __restrict__ out,
                                                    UDiv dcg, UDiv dhw, int any_bcast) {
    uint64_t M = 0;
    UDiv d2m;
    if (PASS == 1) {
        M = hdr->M;
        d2m = hdr->div;
    }
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    uint64_t mx = 0;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < nvec; u += stride) {
        const int64_t pix = (int64_t)udiv((uint64_t)u, dcg);
        const int co0 = (int)(u - pix * cgs) * 8;
        const int64_t img = any_bcast ? (int64_t)udiv((uint64_t)pix, dhw) : 0;
        int64_t z[8];
#pragma unroll
        for (int j = 0; j < 8; j++) z[j] = 0;
#pragma unroll
        for (int i = 0; i < IQ_MAX_TERMS; i++) {
            if (i >= T.n) break;
            const TermDev& t = T.t[i];
            int ch0 = co0;
            if (concat) {
                ch0 = co0 - t.c_offset;
                if (ch0 < 0 || ch0 >= t.c) continue;
            }
            int32_t v[8];
            load8(t, (t.bcast ? img : pix) * t.c + ch0, v);
            const longlong2* f2 = reinterpret_cast<const longlong2*>(F + t.base + ch0);
            const longlong2* b2 = reinterpret_cast<const longlong2*>(B + t.base + ch0);
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const longlong2 f = __ldg(f2 + j), b = __ldg(b2 + j);
                z[2 * j] += (int64_t)f.x * v[2 * j] + (int64_t)b.x;
                z[2 * j + 1] += (int64_t)f.y * v[2 * j + 1] + (int64_t)b.y;
            }
        }
        if (PASS == 0) {
#pragma unroll
            for (int j = 0; j < 8; j++) {
                int64_t zz = (relu && z[j] < 0) ? 0 : z[j];
                uint64_t a = (uint64_t)(zz < 0 ? -zz : zz);
                mx = a > mx ? a : mx;
            }
        } else {
            uint32_t w[2] = {0u, 0u};
#pragma unroll
            for (int j = 0; j < 8; j++) {
                int64_t zz = (relu && z[j] < 0) ? 0 : z[j];
                int64_t c = 0;
                if (M) {
                    uint64_t num = ((uint64_t)(zz + (int64_t)M) << 8) + M;
                    c = clamp64((int64_t)udiv(num, d2m) - 128, -127, 127);
                }
                w[j >> 2] |= ((uint32_t)c & 0xffu) << (8 * (j & 3));
            }
            *reinterpret_cast<uint2*>(out + u * 8) = make_uint2(w[0], w[1]);
        }
    }
    if (PASS == 0) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxz, (unsigned long long)mx);
    }
}

// The operands covering a channel group of the output (at most two in k_comb4r).
struct Cover {
    int n;              // operands covering the group (0..2)
    int id0, id1;
    int ch0, ch1;       // first channel of the group inside each operand
};

__device__ __forceinline__ void cover_of(const Terms& T, int concat, int co0, Cover& cv) {
    cv.n = 0;
    cv.id0 = cv.id1 = 0;
    cv.ch0 = cv.ch1 = 0;
#pragma unroll
    for (int i = 0; i < IQ_MAX_TERMS; i++) {
        if (i >= T.n) break;
        const int ch = concat ? co0 - T.t[i].c_offset : co0;
        if (ch < 0 || ch >= T.t[i].c) continue;
        if (cv.n == 0) { cv.id0 = i; cv.ch0 = ch; }
        else if (cv.n == 1) { cv.id1 = i; cv.ch1 = ch; }
        cv.n++;
    }
}

__device__ __forceinline__ const TermDev& term_at(const Terms& T, int i) {
    switch (i) {
        case 0: return T.t[0];
        case 1: return T.t[1];
        case 2: return T.t[2];
        case 3: return T.t[3];
        case 4: return T.t[4];
        case 5: return T.t[5];
        case 6: return T.t[6];
        default: return T.t[7];
    }
}

// 4 channels of one pixel as int32 (int16 codes: one 8-byte load, int8: one 4-byte load)
__device__ __forceinline__ void load4p(const void* codes, int is16, int64_t idx, int32_t v[4]) {
    if (is16) {
        const int2 q = __ldg(reinterpret_cast<const int2*>((const int16_t*)codes + idx));
        v[0] = (int32_t)(int16_t)(q.x & 0xffff);
        v[1] = q.x >> 16;
        v[2] = (int32_t)(int16_t)(q.y & 0xffff);
        v[3] = q.y >> 16;
    } else {
        const int q = __ldg(reinterpret_cast<const int*>((const int8_t*)codes + idx));
#pragma unroll
        for (int j = 0; j < 4; j++) v[j] = (int32_t)(int8_t)((q >> (8 * j)) & 0xff);
    }
}

// z of 4 channels: F0 v0 + F1 v1 + (B0 + B1), exact in int64 (|z| < 2^50 by the choice of
// P, and the two offsets are added first, which changes no sum)
__device__ __forceinline__ void comb_z4(const long long (&f0)[4], const long long (&f1)[4],
                                        const long long (&bs)[4], const int32_t (&v0)[4],
                                        const int32_t (&v1)[4], int64_t (&z)[4]) {
#pragma unroll
    for (int j = 0; j < 4; j++) z[j] = (int64_t)f0[j] * v0[j] + (int64_t)f1[j] * v1[j] + bs[j];
}

// The two passes with a fixed 4-channel group per thread: the launch has a multiple of
// c_out / 4 threads, so thread t always owns group t % (c_out / 4), keeps the F rows of the
// (at most two) operands covering it and their summed B rows in registers (24 registers;
// the kernel fits 3 blocks of 256 threads per SM), and walks the pixels
// t / (c_out / 4), + T / (c_out / 4), ... two at a time, both pixels' loads in flight
// together.
template <int PASS>
__global__ void __launch_bounds__(kThreads, 3) k_comb4r(Terms T, int concat, int64_t npix, int cgs,
                                                     int relu, const long long* __restrict__ F,
                                                     const long long* __restrict__ B,
                                                     CombHdr* hdr, int8_t* __restrict__ out,
                                                     UDiv dhw, int any_bcast) {
    uint64_t M = 0;
    UDiv d2m;
    if (PASS == 1) {
        M = hdr->M;
        d2m = hdr->div;
    }
    const int64_t tcount = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int g = (int)(t % cgs);
    const int64_t pstride = tcount / cgs;
    const int co0 = 4 * g;
    Cover cv;
    cover_of(T, concat, co0, cv);
    long long f0[4], f1[4], bs[4];
    const TermDev& t0 = term_at(T, cv.id0);
    const TermDev& t1 = term_at(T, cv.id1);
#pragma unroll
    for (int j = 0; j < 4; j++) {
        f0[j] = cv.n > 0 ? F[t0.base + cv.ch0 + j] : 0;
        f1[j] = cv.n > 1 ? F[t1.base + cv.ch1 + j] : 0;
        bs[j] = (cv.n > 0 ? B[t0.base + cv.ch0 + j] : 0) + (cv.n > 1 ? B[t1.base + cv.ch1 + j] : 0);
    }
    const void* base0 = t0.codes;
    const void* base1 = t1.codes;
    const int is0 = t0.is16, is1 = t1.is16, c0 = t0.c, c1 = t1.c, bc0 = t0.bcast, bc1 = t1.bcast;
    const int n0 = cv.n;
    uint64_t mx = 0;
    auto one = [&](int64_t pix, const int32_t (&v0)[4], const int32_t (&v1)[4]) {
        int64_t z[4];
        comb_z4(f0, f1, bs, v0, v1, z);
        if (PASS == 0) {
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const int64_t zz = (relu && z[j] < 0) ? 0 : z[j];
                const uint64_t a = (uint64_t)(zz < 0 ? -zz : zz);
                mx = a > mx ? a : mx;
            }
        } else {
            uint32_t w = 0u;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const int64_t zz = (relu && z[j] < 0) ? 0 : z[j];
                int64_t c = 0;
                if (M) {
                    const uint64_t num = ((uint64_t)(zz + (int64_t)M) << 8) + M;
                    c = clamp64((int64_t)udiv(num, d2m) - 128, -127, 127);
                }
                w |= ((uint32_t)c & 0xffu) << (8 * j);
            }
            *reinterpret_cast<uint32_t*>(out + pix * (int64_t)cgs * 4 + co0) = w;
        }
    };
    int64_t pix = t / cgs;
    for (; pix + pstride < npix; pix += 2 * pstride) {
        const int64_t pb = pix + pstride;
        const int64_t ia = any_bcast ? (int64_t)udiv((uint64_t)pix, dhw) : 0;
        const int64_t ib = any_bcast ? (int64_t)udiv((uint64_t)pb, dhw) : 0;
        int32_t a0[4] = {0, 0, 0, 0}, a1[4] = {0, 0, 0, 0}, b0[4] = {0, 0, 0, 0},
                b1[4] = {0, 0, 0, 0};
        if (n0 > 0) {
            load4p(base0, is0, (bc0 ? ia : pix) * c0 + cv.ch0, a0);
            load4p(base0, is0, (bc0 ? ib : pb) * c0 + cv.ch0, b0);
        }
        if (n0 > 1) {
            load4p(base1, is1, (bc1 ? ia : pix) * c1 + cv.ch1, a1);
            load4p(base1, is1, (bc1 ? ib : pb) * c1 + cv.ch1, b1);
        }
        one(pix, a0, a1);
        one(pb, b0, b1);
    }
    if (pix < npix) {
        const int64_t ia = any_bcast ? (int64_t)udiv((uint64_t)pix, dhw) : 0;
        int32_t a0[4] = {0, 0, 0, 0}, a1[4] = {0, 0, 0, 0};
        if (n0 > 0) load4p(base0, is0, (bc0 ? ia : pix) * c0 + cv.ch0, a0);
        if (n0 > 1) load4p(base1, is1, (bc1 ? ia : pix) * c1 + cv.ch1, a1);
        one(pix, a0, a1);
    }
    if (PASS == 0) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxz, (unsigned long long)mx);
    }
}

// The two passes for a sum of up to 6 operands that each cover all c_out channels (the ASPP
// error sum: four branch errors and the broadcast pooled one).  As in k_comb4r each thread
// owns one 4-channel group, (blockIdx.x 256 + tid) % (c_out / 4), and walks pixels; the
// operands' F rows of the block's 256 groups are staged once per block in shared memory
// (n 8 KB), their B rows summed per thread in registers, so per 4 outputs an operand costs
// one 4- or 8-byte code load and two 16-byte shared loads.
template <int PASS>
__global__ void __launch_bounds__(kThreads) k_combNs(Terms T, int64_t npix, int cgs, int relu,
                                                     const long long* __restrict__ F,
                                                     const long long* __restrict__ B,
                                                     CombHdr* hdr, int8_t* __restrict__ out,
                                                     UDiv dhw, int any_bcast) {
    extern __shared__ __align__(16) long long sF[];     // [n][256 groups][4]
    const int n = T.n, c_out = 4 * cgs;
    const int w0 = (int)(((int64_t)blockIdx.x * blockDim.x) % cgs);   // the block's first group
    for (int k = threadIdx.x; k < n * kThreads * 4; k += blockDim.x) {
        const int ti = k / (kThreads * 4), r = k - ti * (kThreads * 4);
        const int grp = (w0 + (r >> 2)) % cgs;
        sF[k] = F[term_at(T, ti).base + 4 * grp + (r & 3)];
    }
    __syncthreads();
    uint64_t M = 0;
    UDiv d2m;
    if (PASS == 1) {
        M = hdr->M;
        d2m = hdr->div;
    }
    const int64_t tcount = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int g = (int)(t % cgs);
    const int64_t pstride = tcount / cgs;
    const int co0 = 4 * g;
    long long bs[4] = {0, 0, 0, 0};
#pragma unroll
    for (int i = 0; i < IQ_MAX_TERMS; i++) {
        if (i >= n) break;
        const TermDev& ti = term_at(T, i);
#pragma unroll
        for (int j = 0; j < 4; j++) bs[j] += B[ti.base + co0 + j];
    }
    uint64_t mx = 0;
    for (int64_t pix = t / cgs; pix < npix; pix += pstride) {
        const int64_t img = any_bcast ? (int64_t)udiv((uint64_t)pix, dhw) : 0;
        int64_t z[4] = {bs[0], bs[1], bs[2], bs[3]};
#pragma unroll
        for (int i = 0; i < IQ_MAX_TERMS; i++) {
            if (i >= n) break;
            const TermDev& ti = term_at(T, i);
            int32_t v[4];
            load4p(ti.codes, ti.is16, (ti.bcast ? img : pix) * c_out + co0, v);
            const longlong2* f2 =
                reinterpret_cast<const longlong2*>(sF + (i * kThreads + threadIdx.x) * 4);
            const longlong2 fa = f2[0], fb = f2[1];
            z[0] += (int64_t)fa.x * v[0];
            z[1] += (int64_t)fa.y * v[1];
            z[2] += (int64_t)fb.x * v[2];
            z[3] += (int64_t)fb.y * v[3];
        }
        if (PASS == 0) {
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const int64_t zz = (relu && z[j] < 0) ? 0 : z[j];
                const uint64_t a = (uint64_t)(zz < 0 ? -zz : zz);
                mx = a > mx ? a : mx;
            }
        } else {
            uint32_t w = 0u;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const int64_t zz = (relu && z[j] < 0) ? 0 : z[j];
                int64_t c = 0;
                if (M) {
                    const uint64_t num = ((uint64_t)(zz + (int64_t)M) << 8) + M;
                    c = clamp64((int64_t)udiv(num, d2m) - 128, -127, 127);
                }
                w |= ((uint32_t)c & 0xffu) << (8 * j);
            }
            *reinterpret_cast<uint32_t*>(out + pix * (int64_t)c_out + co0) = w;
        }
    }
    if (PASS == 0) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxz, (unsigned long long)mx);
    }
}

// ---------------------------------------------------------------- fp32-decided joins
//
// The two passes with a fixed group of CPT channels per thread (as k_comb4r with 4), for up
// to NC operands covering each group, with each element first evaluated in fp32:
// zf = fma(F_k, v_k, ...) over the covering operands from fl(sum B), with F_k rounded to
// fp32.  With u = 2^-24 and, over the thread's channels, S = max |sum B| +
// sum_k |F_k| vmax_k, every |zf - z| <= (nc + 2) u S (the B sum and each F converted with a
// relative error of at most 2u, one rounding per fma, every partial sum below S); the
// kernel takes E = (nc + 3) u S, evaluated in fp32 rounded upward, so it bounds the exact
// value.  The exact int64 z is formed only where fp32 cannot decide:
//  - max pass: an element whose |zf| is within 3E_w of the largest |zf| its warp has seen,
//    E_w the largest E of the warp's lanes.  No |zf| of the warp exceeds M + E_w, M = max
//    |z|, and an element with |z| = M has |zf| >= M - E_w, so that element is evaluated
//    exactly (the third E_w covers the rounding of the threshold); the largest exact value
//    over all evaluated elements is M;
//  - codes pass: y = fl(zf fl(128/M) + 1/2) is within D = 130 E / M + 2^-14 of the exact
//    128 z / M + 1/2 (the ratio's and the fma's roundings add at most 2^-15); when
//    floor(y - D) == floor(y + D) that is the code, otherwise the code is
//    floor((256 z + M) / (2M)) with the 64-bit invariant division, as in k_comb4r.
// UNR pixels per iteration keep UNR x NC loads of 8 or 16 bytes in flight per thread; the
// codes stay packed in registers until they are used.

template <int NC>
struct Cover4 {
    int n;
    int id[NC];
    int ch[NC];
};

template <int NC>
__device__ __forceinline__ void cover4_of(const Terms& T, int concat, int co0, Cover4<NC>& cv) {
    cv.n = 0;
#pragma unroll
    for (int k = 0; k < NC; k++) { cv.id[k] = 0; cv.ch[k] = 0; }
#pragma unroll
    for (int i = 0; i < IQ_MAX_TERMS; i++) {
        if (i >= T.n) break;
        const int ch = concat ? co0 - T.t[i].c_offset : co0;
        if (ch < 0 || ch >= T.t[i].c) continue;
#pragma unroll
        for (int k = 0; k < NC; k++)
            if (k == cv.n) { cv.id[k] = i; cv.ch[k] = ch; }
        cv.n++;
    }
}


// CPT codes of one operand as loaded: 16 bytes (CPT = 8 int16 or 16 int8 codes) or
// 8 bytes (CPT = 8 int8 codes)
struct Raw16 {
    uint32_t w[4];
};

template <int CPT>
__device__ __forceinline__ Raw16 load_raw(const char* p, int is16) {
    Raw16 r;
    if (CPT == 16 || is16) {
        const int4 q = __ldg(reinterpret_cast<const int4*>(p));
        r.w[0] = (uint32_t)q.x; r.w[1] = (uint32_t)q.y; r.w[2] = (uint32_t)q.z; r.w[3] = (uint32_t)q.w;
    } else {
        const int2 q = __ldg(reinterpret_cast<const int2*>(p));
        r.w[0] = (uint32_t)q.x; r.w[1] = (uint32_t)q.y; r.w[2] = 0u; r.w[3] = 0u;
    }
    return r;
}

template <int CPT>
__device__ __forceinline__ int32_t raw_code(const Raw16& r, int is16, int j) {
    if (CPT == 8 && is16) {
        const uint32_t w = r.w[j >> 1];
        return (j & 1) ? (int32_t)w >> 16 : (int32_t)(int16_t)(w & 0xffffu);
    }
    return (int32_t)(int8_t)((r.w[j >> 2] >> (8 * (j & 3))) & 0xffu);
}

// The two passes with CPT channels per thread.  PLAIN: every operand is int8 codes
// without gamma / beta, so each has one F for all its channels and B = 0 (the sums of
// errors and the ASPP concatenation); otherwise (the residual joins) F and B are
// per channel, codes int16 or int8, CPT = 8.
template <int PASS, int NC, int CPT, int UNR, bool PLAIN>
__global__ void __launch_bounds__(kThreads, (PLAIN && NC <= 2) ? 3 : 2) k_comb4f(Terms T, int concat, int64_t npix, int cgs,
                                                     int relu, const long long* __restrict__ F,
                                                     const long long* __restrict__ B,
                                                     CombHdr* hdr, int8_t* __restrict__ out,
                                                     UDiv dhw, int any_bcast) {
    constexpr int FW = PLAIN ? 1 : CPT;      // F values held per operand
    const int64_t tcount = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int g = (int)(t % cgs);
    const int64_t pstride = tcount / cgs;
    const int co0 = CPT * g;
    Cover4<NC> cv;
    cover4_of<NC>(T, concat, co0, cv);
    const int nc = cv.n;
    // per covering operand: its codes at the group's first channel, row bytes, type,
    // broadcast flag, first row of F / B, fp32 F; the fp32 B sums; the bound S
    const char* base[NC];
    int rowb[NC], is16[NC], bc[NC], fo[NC];
    float ff[NC][FW];
    float bf[FW];
    long long fi[NC];          // PLAIN: the exact F of each operand
    float S = 0.f;             // fp32 with upward rounding: an upper bound of the exact S
    {
        long long bs[FW];
        float sv[FW];
#pragma unroll
        for (int j = 0; j < FW; j++) { bs[j] = 0; sv[j] = 0.f; }
#pragma unroll
        for (int k = 0; k < NC; k++) {
            const TermDev& tt = term_at(T, cv.id[k]);
            const bool on = k < nc;
            is16[k] = PLAIN ? 0 : tt.is16;
            bc[k] = tt.bcast;
            rowb[k] = tt.c * (tt.is16 ? 2 : 1);
            base[k] = (const char*)tt.codes + (size_t)cv.ch[k] * (tt.is16 ? 2 : 1);
            fo[k] = tt.base + cv.ch[k];
            const float vmax = tt.is16 ? 32767.f : 127.f;
#pragma unroll
            for (int j = 0; j < FW; j++) {
                const long long f = on ? F[fo[k] + j] : 0;
                ff[k][j] = f32_of_i64(f);
                if (PLAIN) fi[k] = f;
                if (!PLAIN) bs[j] += on ? B[fo[k] + j] : 0;
                sv[j] = __fmaf_ru(f32_abs_up(f), vmax, sv[j]);
            }
        }
#pragma unroll
        for (int j = 0; j < FW; j++) {
            bf[j] = f32_of_i64(bs[j]);
            const float sj = __fadd_ru(sv[j], f32_abs_up(bs[j]));
            S = fmaxf(S, sj);
        }
    }
    const float E = __fmul_ru(__fmul_ru((float)(nc + 3), 0x1p-24f), S);
    // the max pass shares its running maximum across the warp, so its margin covers the
    // largest E of the warp's lanes
    float E3 = __fmul_ru(3.f, E);
    if (PASS == 0) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) E3 = fmaxf(E3, __shfl_xor_sync(0xffffffffu, E3, o));
    }
    uint64_t M = 0;
    float kq = 0.f, D = 0.f;
    if (PASS == 1) {
        M = hdr->M;
        kq = hdr->kq;
        D = __fmaf_ru(E, hdr->c130, 0x1p-14f);
    }
    // exact z of channel j of a pixel from its loaded codes (F and B re-read: a rare path)
    auto exact = [&](const Raw16 (&r)[NC], int j) -> int64_t {
        int64_t z = 0;
#pragma unroll
        for (int k = 0; k < NC; k++)
            if (k < nc) {
                const int64_t f = PLAIN ? fi[k] : F[fo[k] + j];
                z += f * raw_code<CPT>(r[k], is16[k], j);
                if (!PLAIN) z += B[fo[k] + j];
            }
        return (relu && z < 0) ? 0 : z;
    };
    float fmx = 0.f;
    uint64_t mx = 0;
    auto one = [&](int64_t pix, const Raw16 (&r)[NC]) {
        const bool valid = pix < npix;
        float zf[CPT];
#pragma unroll
        for (int j = 0; j < CPT; j++) zf[j] = PLAIN ? 0.f : bf[PLAIN ? 0 : j];
#pragma unroll
        for (int k = 0; k < NC; k++)
            if (k < nc) {
#pragma unroll
                for (int j = 0; j < CPT; j++)
                    zf[j] = fmaf(ff[k][PLAIN ? 0 : j], (float)raw_code<CPT>(r[k], is16[k], j),
                                 zf[j]);
            }
        if (PASS == 0) {
            // the pixel's largest |zf| first, so that only elements near the running maximum
            // (usually none of the pixel's) take the exact form
            float a[CPT], am = 0.f;
#pragma unroll
            for (int j = 0; j < CPT; j++) {
                a[j] = fabsf(relu ? fmaxf(zf[j], 0.f) : zf[j]);
                am = fmaxf(am, a[j]);
            }
            if (!valid) am = 0.f;
            fmx = fmaxf(fmx, am);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) fmx = fmaxf(fmx, __shfl_xor_sync(0xffffffffu, fmx, o));
            const float thr = fmx - E3;
            if (valid && am >= thr) {
#pragma unroll
                for (int j = 0; j < CPT; j++)
                    if (a[j] >= thr) {
                        const int64_t z = exact(r, j);
                        const uint64_t az = (uint64_t)(z < 0 ? -z : z);
                        mx = az > mx ? az : mx;
                    }
            }
        } else {
            uint32_t w[CPT / 4];
#pragma unroll
            for (int q = 0; q < CPT / 4; q++) w[q] = 0u;
            if (M) {
#pragma unroll
                for (int j = 0; j < CPT; j++) {
                    const float y = fmaf(relu ? fmaxf(zf[j], 0.f) : zf[j], kq, 0.5f);
                    const float lo = floorf(y - D), hi = floorf(y + D);
                    int64_t c;
                    if (lo == hi) {      // only when D < 1/2, so |y| < 130
                        c = min(max((int)lo, -127), 127);
                    } else {
                        const UDiv d2m = hdr->div;
                        const uint64_t num = ((uint64_t)(exact(r, j) + (int64_t)M) << 8) + M;
                        c = clamp64((int64_t)udiv(num, d2m) - 128, -127, 127);
                    }
                    w[j >> 2] |= ((uint32_t)c & 0xffu) << (8 * (j & 3));
                }
            }
            int8_t* o = out + pix * (int64_t)cgs * CPT + co0;
            if (!valid) return;
            if (CPT == 16)
                *reinterpret_cast<uint4*>(o) = make_uint4(w[0], w[1], w[2], w[3]);
            else
                *reinterpret_cast<uint2*>(o) = make_uint2(w[0], w[1]);
        }
    };
    auto load = [&](int64_t pix, Raw16 (&r)[NC]) {
        const bool valid = pix < npix;
        const int64_t img = (any_bcast && valid) ? (int64_t)udiv((uint64_t)pix, dhw) : 0;
#pragma unroll
        for (int k = 0; k < NC; k++) {
            if (k < nc && valid) {
                r[k] = load_raw<CPT>(base[k] + (bc[k] ? img : pix) * rowb[k], is16[k]);
            } else {
#pragma unroll
                for (int q = 0; q < 4; q++) r[k].w[q] = 0u;
            }
        }
    };
    // every lane of a warp runs the warp's largest number of pixel steps (the max pass
    // shuffles inside the loop); steps past the tensor's end load and store nothing
    const int64_t p0 = t / cgs;
    int64_t steps = p0 < npix ? (npix - p0 + pstride - 1) / pstride : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int64_t w = __shfl_xor_sync(0xffffffffu, steps, o);
        steps = w > steps ? w : steps;
    }
    for (int64_t k0 = 0; k0 < steps; k0 += UNR) {
        Raw16 r[UNR][NC];
#pragma unroll
        for (int u = 0; u < UNR; u++) load(p0 + (k0 + u) * pstride, r[u]);
#pragma unroll
        for (int u = 0; u < UNR; u++) one(p0 + (k0 + u) * pstride, r[u]);
    }
    if (PASS == 0) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxz, (unsigned long long)mx);
    }
}

__global__ void k_comb_params(CombHdr* hdr, double* s_out) {
    const uint64_t M = hdr->maxz;
    hdr->M = M;
    hdr->div = make_udiv(M ? 2 * M : 1);
    hdr->kq = M ? (float)(128.0 / (double)M) : 0.f;
    hdr->c130 = M ? __double2float_ru(__ddiv_ru(130.0, (double)M)) : 0.f;
    *s_out = M ? ldexp((double)M, -hdr->P - 7) : ldexp(1.0, -hdr->P - 7);
}

// ---------------------------------------------------------------- streamed two-operand joins
//
// The two passes of a sum of two operands that both cover every channel of every pixel (the
// residual adds and the sums of two errors), with the operands' rows landed in shared memory
// by bulk copies (iq_stream.cuh): the copy engine keeps about 130 KB per SM in flight, where
// the register-fed k_comb4f keeps 32 KB.  The arithmetic is k_comb4f's, with 4 channels per
// thread (the stream's channel group), and two changes that decide nothing differently:
//  - codes reach fp32 without the conversion unit: a code v of an int16 word biased to
//    u = v + 2^15 (an xor) and placed in the low mantissa bits of 2^23 by a byte permute is
//    the float 2^23 + u, and subtracting 2^23 + 2^15 leaves v exactly (int8: 2^23 + 2^7);
//  - the codes pass clamps y to [-126.5, 127.5] (the clamp of the code to [-127, 127]
//    commutes with the floor there) and takes floor(y) = c from the bits of y + 1.5 2^23
//    rounded downward (its low byte is the code), f = y - c exactly; the code is c when
//    D <= f < 1 - D (D < 1/2): the exact value, within D of y, then has the same floor (a
//    clamped y has f = 1/2 and an exact value beyond the clamp bound); otherwise the element
//    takes the exact division.
// The max pass shares its running maximum across the warp with one max-reduction over the
// fp32 bit patterns (non-negative floats order as their bits) per row.

__device__ __forceinline__ float f32_of_i16_lo(uint32_t wx) {
    return __int_as_float((int)__byte_perm(wx, 0x4B000000u, 0x7410)) - 8421376.0f;
}
__device__ __forceinline__ float f32_of_i16_hi(uint32_t wx) {
    return __int_as_float((int)__byte_perm(wx, 0x4B000000u, 0x7432)) - 8421376.0f;
}
template <int J>
__device__ __forceinline__ float f32_of_i8(uint32_t wx) {
    return __int_as_float((int)__byte_perm(wx, 0x4B000000u, 0x7440 + J)) - 8388736.0f;
}

// the 4 codes of one operand at a row of a stage, as fp32 and as raw words
template <bool W16>
__device__ __forceinline__ void stage_codes4(const uint8_t* p, float (&f)[4], uint2& raw) {
    if (W16) {
        raw = *reinterpret_cast<const uint2*>(p);
        const uint32_t a = raw.x ^ 0x80008000u, b = raw.y ^ 0x80008000u;
        f[0] = f32_of_i16_lo(a); f[1] = f32_of_i16_hi(a);
        f[2] = f32_of_i16_lo(b); f[3] = f32_of_i16_hi(b);
    } else {
        raw.x = *reinterpret_cast<const uint32_t*>(p);
        raw.y = 0u;
        const uint32_t a = raw.x ^ 0x80808080u;
        f[0] = f32_of_i8<0>(a); f[1] = f32_of_i8<1>(a);
        f[2] = f32_of_i8<2>(a); f[3] = f32_of_i8<3>(a);
    }
}
template <bool W16>
__device__ __forceinline__ int32_t raw_code4(const uint2& r, int j) {
    if (W16) {
        const uint32_t w = j < 2 ? r.x : r.y;
        return (j & 1) ? (int32_t)w >> 16 : (int32_t)(int16_t)(w & 0xffffu);
    }
    return (int32_t)(int8_t)((r.x >> (8 * j)) & 0xffu);
}

template <int PASS, bool A16, bool B16, bool PLAIN>
__global__ void __launch_bounds__(kStreamThreads, 1)
    k_comb_s(RowStream rs, Terms T, int relu, const long long* __restrict__ F,
             const long long* __restrict__ B, CombHdr* hdr, int8_t* __restrict__ out,
             uint2* __restrict__ out16, int* __restrict__ err) {
    extern __shared__ __align__(128) uint8_t smem[];
    if (__syncthreads_or(threadIdx.x == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    constexpr int FW = PLAIN ? 1 : 4;
    const int CB4 = rs.CB >> 2;
    const int g = threadIdx.x % CB4, rl = threadIdx.x / CB4;
    const int c0 = blockIdx.x * rs.CB + 4 * g;
    int fo[2];
    float ff[2][FW], bf[FW];
    long long fi[2];
    float S = 0.f;
    {
        long long bs[FW];
        float sv[FW];
#pragma unroll
        for (int j = 0; j < FW; j++) { bs[j] = 0; sv[j] = 0.f; }
#pragma unroll
        for (int k = 0; k < 2; k++) {
            const TermDev& tt = T.t[k];
            fo[k] = tt.base + c0;
            const float vmax = (k == 0 ? A16 : B16) ? 32767.f : 127.f;
#pragma unroll
            for (int j = 0; j < FW; j++) {
                const long long f = F[fo[k] + j];
                ff[k][j] = f32_of_i64(f);
                if (PLAIN) fi[k] = f;
                if (!PLAIN) bs[j] += B[fo[k] + j];
                sv[j] = __fmaf_ru(f32_abs_up(f), vmax, sv[j]);
            }
        }
#pragma unroll
        for (int j = 0; j < FW; j++) {
            bf[j] = f32_of_i64(bs[j]);
            S = fmaxf(S, __fadd_ru(sv[j], f32_abs_up(bs[j])));
        }
    }
    const float E = __fmul_ru(__fmul_ru(5.f, 0x1p-24f), S);    // (nc + 3) u S, nc = 2
    float E3 = __fmul_ru(3.f, E);
    if (PASS == 0) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) E3 = fmaxf(E3, __shfl_xor_sync(0xffffffffu, E3, o));
    }
    uint64_t M = 0;
    float kq = 0.f, D = 0.f, omd = 0.f;
    bool fast = false;
    if (PASS == 1) {
        M = hdr->M;
        kq = hdr->kq;
        D = __fmaf_ru(E, hdr->c130, 0x1p-14f);
        omd = __fsub_rd(1.f, D);
        fast = D < 0.5f;
    }
    auto exact = [&](const uint2& ra, const uint2& rb, int j) -> int64_t {
        int64_t z;
        if (PLAIN) {
            z = fi[0] * raw_code4<A16>(ra, j) + fi[1] * raw_code4<B16>(rb, j);
        } else {
            z = F[fo[0] + j] * raw_code4<A16>(ra, j) + B[fo[0] + j] +
                F[fo[1] + j] * raw_code4<B16>(rb, j) + B[fo[1] + j];
        }
        return (relu && z < 0) ? 0 : z;
    };
    const int eszA = A16 ? 2 : 1, eszB = B16 ? 2 : 1;
    uint32_t fmx = 0u;         // bits of the warp's largest |zf| so far
    uint64_t mx = 0;
    auto row = [&](const uint8_t* st, int r, int64_t r0) {
            const int e = r * rs.CB + 4 * g;
            float fa[4], fb[4];
            uint2 ra, rb;
            stage_codes4<A16>(st + rs.off[0] + e * eszA, fa, ra);
            stage_codes4<B16>(st + rs.off[1] + e * eszB, fb, rb);
            float zf[4];
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const float b0 = PLAIN ? 0.f : bf[PLAIN ? 0 : j];
                zf[j] = fmaf(ff[1][PLAIN ? 0 : j], fb[j], fmaf(ff[0][PLAIN ? 0 : j], fa[j], b0));
            }
            if (PASS == 0) {
                float a[4], am = 0.f;
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    a[j] = fabsf(relu ? fmaxf(zf[j], 0.f) : zf[j]);
                    am = fmaxf(am, a[j]);
                }
                fmx = max(fmx, __reduce_max_sync(0xffffffffu, __float_as_uint(am)));
                const float thr = __uint_as_float(fmx) - E3;
                if (am >= thr) {
#pragma unroll
                    for (int j = 0; j < 4; j++)
                        if (a[j] >= thr) {
                            const int64_t z = exact(ra, rb, j);
                            const uint64_t az = (uint64_t)(z < 0 ? -z : z);
                            mx = az > mx ? az : mx;
                        }
                }
            } else {
                uint32_t w = 0u;
                if (M) {
                    uint32_t tb[4];
                    bool ok[4];
#pragma unroll
                    for (int j = 0; j < 4; j++) {
                        const float y = fminf(fmaxf(fmaf(relu ? fmaxf(zf[j], 0.f) : zf[j], kq,
                                                         0.5f), -126.5f), 127.5f);
                        const float t = __fadd_rd(y, 12582912.0f);
                        const float f = y - (t - 12582912.0f);
                        tb[j] = __float_as_uint(t);
                        ok[j] = f >= D && f < omd;
                    }
                    // one branch per row for the rare elements fp32 does not decide
                    if (!(fast && ok[0] && ok[1] && ok[2] && ok[3])) {
                        const UDiv d2m = hdr->div;
#pragma unroll
                        for (int j = 0; j < 4; j++)
                            if (!(fast && ok[j])) {
                                const uint64_t num =
                                    ((uint64_t)(exact(ra, rb, j) + (int64_t)M) << 8) + M;
                                tb[j] = (uint32_t)(int)clamp64((int64_t)udiv(num, d2m) - 128,
                                                               -127, 127);
                            }
                    }
                    w = __byte_perm(__byte_perm(tb[0], tb[1], 0x0040),
                                    __byte_perm(tb[2], tb[3], 0x0040), 0x5410);
                }
                const int64_t oi = (r0 + r) * rs.C + c0;
                *reinterpret_cast<uint32_t*>(out + oi) = w;
                if (out16) {          // the fp16 copy of the 4 codes
                    uint2 hv;
                    tc::i8x4_to_f16x4(w, hv.x, hv.y);
                    out16[oi >> 2] = hv;
                }
            }
    };
    const bool ok = stream_chunks(rs, smem, err, [&](const uint8_t* st, int rows, int64_t r0) {
        // rl is the same on every lane of a warp (CB >= 128), so the row loop is warp-uniform;
        // a whole chunk runs fully unrolled (the rows' loads and arithmetic interleave)
        if (rows == rs.R) {
#pragma unroll
            for (int u = 0; u < kStreamRPT; u++) row(st, rl + u * rs.RL, r0);
        } else {
            for (int u = 0; u < kStreamRPT; u++) {
                const int r = rl + u * rs.RL;
                if (r >= rows) break;
                row(st, r, r0);
            }
        }
    });
    if (!ok) return;
    if (PASS == 0) {
        mx = warp_max_u64(mx);
        if ((threadIdx.x & 31) == 0 && mx) atomicMax(&hdr->maxz, (unsigned long long)mx);
    }
}

// the dynamic shared memory of one instantiation, set once
template <int PASS, bool A16, bool B16, bool PLAIN>
iq_status comb_s_launch(const RowStream& rs, const Terms& T, int relu, const long long* F,
                        const long long* B, CombHdr* hdr, int8_t* out, uint2* out16, int* err,
                        cudaStream_t st) {
    static bool attr = false;
    auto kern = k_comb_s<PASS, A16, B16, PLAIN>;
    if (!attr) {
        IQ_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)row_stream_smem(rs)));
        attr = true;
    }
    kern<<<row_stream_grid(rs, device_sms()), kStreamThreads, row_stream_smem(rs), st>>>(
        rs, T, relu, F, B, hdr, out, out16, err);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

template <int PASS>
iq_status comb_s_pass(const RowStream& rs, const Terms& T, bool plain, int relu,
                      const long long* F, const long long* B, CombHdr* hdr, int8_t* out,
                      uint2* o16, int* err, cudaStream_t st) {
    const bool a16 = T.t[0].is16 != 0, b16 = T.t[1].is16 != 0;
    if (plain)
        return comb_s_launch<PASS, false, false, true>(rs, T, relu, F, B, hdr, out, o16, err, st);
    if (a16 && b16)
        return comb_s_launch<PASS, true, true, false>(rs, T, relu, F, B, hdr, out, o16, err, st);
    if (a16)
        return comb_s_launch<PASS, true, false, false>(rs, T, relu, F, B, hdr, out, o16, err, st);
    if (b16)
        return comb_s_launch<PASS, false, true, false>(rs, T, relu, F, B, hdr, out, o16, err, st);
    return comb_s_launch<PASS, false, false, false>(rs, T, relu, F, B, hdr, out, o16, err, st);
}

// ---------------------------------------------------------------- spatial sums

// sums[i][j] += sum over a slice of image i's pixels of x[i][p][c_off + j]
__global__ void k_ssum(const int8_t* __restrict__ x, int64_t hw, int c_total, int c_off, int c,
                       int64_t pix_per_block, unsigned long long* __restrict__ sums) {
    const int64_t img = blockIdx.y;
    const int j = blockIdx.z * blockDim.x + threadIdx.x;
    if (j >= c) return;
    const int64_t p0 = (int64_t)blockIdx.x * pix_per_block;
    const int64_t p1 = min(hw, p0 + pix_per_block);
    const int8_t* src = x + (img * hw) * c_total + c_off + j;
    int64_t acc = 0;
    for (int64_t p = p0; p < p1; p++) acc += src[p * c_total];
    if (acc) atomicAdd(&sums[img * c + j], (unsigned long long)acc);
}

// One block: M = max |sum|, the output scale in the oracle's order, then the codes.
__global__ void k_ssum_finish(const unsigned long long* __restrict__ sums, int64_t count,
                              const double* __restrict__ s_x, double den,
                              int8_t* __restrict__ out, double* __restrict__ s_out) {
    __shared__ unsigned long long sM;
    __shared__ UDiv sdiv;
    if (threadIdx.x == 0) sM = 0;
    __syncthreads();
    uint64_t mx = 0;
    for (int64_t i = threadIdx.x; i < count; i += blockDim.x) {
        int64_t v = (int64_t)sums[i];
        uint64_t a = (uint64_t)(v < 0 ? -v : v);
        mx = a > mx ? a : mx;
    }
    mx = warp_max_u64(mx);
    if ((threadIdx.x & 31) == 0) atomicMax(&sM, (unsigned long long)mx);
    __syncthreads();
    const uint64_t M = sM;
    if (threadIdx.x == 0) {
        sdiv = make_udiv(M ? 2 * M : 1);
        const double s = *s_x;
        const double sm = M ? __dmul_rn(s, (double)M) : s;
        *s_out = ldexp(__ddiv_rn(sm, den), -7);
    }
    __syncthreads();
    const UDiv d = sdiv;
    for (int64_t i = threadIdx.x; i < count; i += blockDim.x) {
        int64_t c = 0;
        if (M) {
            uint64_t num = ((uint64_t)((int64_t)sums[i] + (int64_t)M) << 8) + M;
            c = clamp64((int64_t)udiv(num, d) - 128, -127, 127);
        }
        out[i] = (int8_t)c;
    }
}

__global__ void k_scale_div(const double* __restrict__ s, double den, double* __restrict__ out) {
    *out = __ddiv_rn(*s, den);
}

__global__ void k_bcast(const int8_t* __restrict__ e, int64_t n, int64_t hw, int c,
                        int8_t* __restrict__ ex, UDiv dhwc) {
    const int64_t total = n * hw * c;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        const int64_t img = (int64_t)udiv((uint64_t)i, dhwc);
        const int64_t r = i - img * hw * c;
        const int64_t pix = r / c;
        ex[i] = e[img * c + (r - pix * c)];
    }
}

__global__ void k_slice(const int8_t* __restrict__ x, int64_t npix, int c_total, int c_off, int c,
                        int8_t* __restrict__ out, UDiv dc) {
    const int64_t total = npix * c;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        const int64_t p = (int64_t)udiv((uint64_t)i, dc);
        out[i] = x[p * c_total + c_off + (i - p * c)];
    }
}

bool terms_ok(const iq_term* terms, int32_t n_terms) {
    if (!terms || n_terms < 1 || n_terms > IQ_MAX_TERMS) return false;
    for (int i = 0; i < n_terms; i++) {
        const iq_term& t = terms[i];
        if (!t.codes || !t.scale || t.c < 1) return false;
        if (t.dtype != IQ_I8 && t.dtype != IQ_I16) return false;
        if ((t.gamma == nullptr) != (t.beta == nullptr)) return false;
        if (t.gamma && (t.k_gamma < 2 || t.k_gamma > 16 || t.k_beta < 2 || t.k_beta > 16))
            return false;
    }
    return true;
}

size_t comb_ws(const iq_term* terms, int32_t n_terms) {
    size_t rows = 0;
    for (int i = 0; i < n_terms; i++) rows += (size_t)terms[i].c;
    return 256 + 2 * (((rows * 8) + 255) & ~size_t(255));
}

}  // namespace

}  // namespace iq

using namespace iq;

extern "C" iq_status iq_combine_workspace_size(const iq_term* terms, int32_t n_terms,
                                               size_t* bytes) {
    if (!bytes || !terms_ok(terms, n_terms)) return IQ_ERR_INVALID_ARG;
    *bytes = comb_ws(terms, n_terms);
    return IQ_OK;
}

static iq_status combine_codes(const iq_term* terms, int32_t n_terms, int32_t concat, int64_t n,
                               int64_t hw, int32_t c_out, int32_t relu, int8_t* out,
                               double* s_out, uint2* out16, bool& wrote16, void* ws,
                               size_t ws_bytes, iq_stream stream);

extern "C" iq_status iq_combine(const iq_term* terms, int32_t n_terms, int32_t concat, int64_t n,
                                int64_t hw, int32_t c_out, int32_t relu, int8_t* out,
                                double* s_out, void* out_f16, void* ws, size_t ws_bytes,
                                iq_stream stream) {
    if (!terms_ok(terms, n_terms) || !out || !s_out || n < 1 || hw < 1 || c_out < 1)
        return IQ_ERR_INVALID_ARG;
    if (n * hw > (int64_t(1) << 40)) return IQ_ERR_INVALID_ARG;
    if (out_f16 && !f16_copy_ok(out, out_f16, n * hw * (int64_t)c_out)) return IQ_ERR_INVALID_ARG;
    bool wrote16 = false;
    iq_status r = combine_codes(terms, n_terms, concat, n, hw, c_out, relu, out, s_out,
                                (uint2*)out_f16, wrote16, ws, ws_bytes, stream);
    if (r != IQ_OK || !out_f16 || wrote16) return r;
    // the kernels without the fused copy: one conversion pass
    return codes_to_f16(out, (__half*)out_f16, n * hw * (int64_t)c_out, (cudaStream_t)stream);
}

// the joins; out16 is written by the streamed codes pass (wrote16), else left to the caller
static iq_status combine_codes(const iq_term* terms, int32_t n_terms, int32_t concat, int64_t n,
                               int64_t hw, int32_t c_out, int32_t relu, int8_t* out,
                               double* s_out, uint2* out16, bool& wrote16, void* ws,
                               size_t ws_bytes, iq_stream stream) {
    Terms T;
    T.n = n_terms;
    int32_t base = 0;
    for (int i = 0; i < n_terms; i++) {
        const iq_term& s = terms[i];
        if (concat) {
            if (s.c_offset < 0 || s.c_offset + s.c > c_out) return IQ_ERR_INVALID_ARG;
        } else if (s.c != c_out || s.c_offset != 0) {
            return IQ_ERR_INVALID_ARG;
        }
        TermDev& t = T.t[i];
        t.codes = s.codes;
        t.scale = s.scale;
        t.gamma = s.gamma;
        t.beta = s.beta;
        t.is16 = s.dtype == IQ_I16;
        t.c = s.c;
        t.c_offset = concat ? s.c_offset : 0;
        t.bcast = s.bcast != 0;
        t.k_gamma = s.k_gamma;
        t.k_beta = s.k_beta;
        t.base = base;
        base += s.c;
    }
    if (!ws || ws_bytes < comb_ws(terms, n_terms)) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    CombHdr* hdr = (CombHdr*)ws;
    const size_t tab = (((size_t)base * 8) + 255) & ~size_t(255);
    long long* F = (long long*)((char*)ws + 256);
    long long* B = (long long*)((char*)ws + 256 + tab);
    int max_c = 0;
    for (int i = 0; i < n_terms; i++) max_c = std::max(max_c, (int)T.t[i].c);
    if (max_c < 1) return IQ_ERR_INVALID_ARG;
    const dim3 tg((unsigned)((max_c + kTabThreads - 1) / kTabThreads), (unsigned)n_terms);
    IQ_CUDA_CHECK(cudaMemsetAsync(hdr->bound, 0, sizeof(hdr->bound), st));
    k_comb_bound<<<tg, kTabThreads, 0, st>>>(T, hdr);
    IQ_LAUNCH_CHECK();
    k_comb_tab<<<tg, kTabThreads, 0, st>>>(T, hdr, F, B);
    IQ_LAUNCH_CHECK();
    const int64_t total = n * hw * (int64_t)c_out;
    bool vec = c_out % 8 == 0 && ((uintptr_t)out & 7) == 0;
    bool vec4 = c_out % 4 == 0 && ((uintptr_t)out & 3) == 0;
    bool any_bcast = false;
    for (int i = 0; i < n_terms; i++) {
        const TermDev& t = T.t[i];
        vec = vec && t.c % 8 == 0 && t.c_offset % 8 == 0 &&
              ((uintptr_t)t.codes & (t.is16 ? 15 : 7)) == 0;
        vec4 = vec4 && t.c % 4 == 0 && t.c_offset % 4 == 0 &&
               ((uintptr_t)t.codes & (t.is16 ? 7 : 3)) == 0;
        any_bcast = any_bcast || t.bcast;
    }
    // the bytes each pass must move: every operand's codes once (+ the output codes)
    double in_b = 0.0;
    for (int i = 0; i < n_terms; i++)
        in_b += (double)(T.t[i].bcast ? n : n * hw) * T.t[i].c * (T.t[i].is16 ? 2.0 : 1.0);
    const double out_b = (double)total;
    const UDiv dhw = make_udiv((uint64_t)hw);
    // the wide kernels: every operand's channel count and offset and c_out a multiple of the
    // channels per thread, codes 16-byte (8-byte for int8 at 8 channels) aligned; the most
    // operands covering any group (checked per group on the host) and whether all are plain
    // int8 codes decide the variant
    bool plain = true, any16 = false;
    for (int i = 0; i < n_terms; i++) {
        plain = plain && !T.t[i].gamma && !T.t[i].beta && !T.t[i].is16;
        any16 = any16 || T.t[i].is16;
    }
    // two operands that cover every channel of every pixel (residual adds, sums of two
    // errors): the streamed passes, when the stream takes the shape with at least 128
    // channels per slab (a warp's lanes then share their rows)
    if (n_terms == 2 && !concat && !any_bcast && ((uintptr_t)out & 3) == 0) {
        RowStream rs;
        const void* srcs[2] = {T.t[0].codes, T.t[1].codes};
        const int esz[2] = {T.t[0].is16 ? 2 : 1, T.t[1].is16 ? 2 : 1};
        if (row_stream_plan(rs, n * hw, c_out, srcs, esz, 2) && rs.CB >= 128) {
            int* err = device_status_ptr();
            if (!err) return IQ_ERR_CUDA;
            const int rl = relu != 0;
            kt_pre(st);
            iq_status r = comb_s_pass<0>(rs, T, plain, rl, F, B, hdr, out, nullptr, err, st);
            if (r != IQ_OK) return r;
            kt_post_bytes(st, IQ_KERNEL_COMBINE_MAX, in_b);
            k_comb_params<<<1, 1, 0, st>>>(hdr, s_out);
            IQ_LAUNCH_CHECK();
            kt_pre(st);
            r = comb_s_pass<1>(rs, T, plain, rl, F, B, hdr, out, out16, err, st);
            if (r != IQ_OK) return r;
            kt_post_bytes(st, IQ_KERNEL_COMBINE_CODES, in_b + out_b * (out16 ? 3.0 : 1.0));
            wrote16 = out16 != nullptr;
            return IQ_OK;
        }
    }
    const int cpt = plain ? 16 : 8;
    bool wide = c_out % cpt == 0 && ((uintptr_t)out & (cpt - 1)) == 0;
    for (int i = 0; i < n_terms && wide; i++) {
        const TermDev& t = T.t[i];
        const uintptr_t al = (cpt == 16 || t.is16) ? 15 : 7;
        wide = t.c % cpt == 0 && t.c_offset % cpt == 0 && ((uintptr_t)t.codes & al) == 0;
    }
    int maxcover = 0;
    for (int co = 0; co < c_out && wide; co += cpt) {
        int nc = 0;
        for (int i = 0; i < n_terms; i++) {
            const TermDev& t = T.t[i];
            const int ch = concat ? co - t.c_offset : co;
            if (ch >= 0 && ch < t.c) nc++;
        }
        maxcover = nc > maxcover ? nc : maxcover;
    }
    (void)any16;
    if (wide && (plain ? maxcover <= 6 : maxcover <= 2)) {
        const int cgs = c_out / cpt;
        const int64_t npix = n * hw;
        // a multiple of cgs threads, about 8 blocks of 256 per SM
        int64_t gcd = cgs, b2 = kThreads;
        while (b2) { int64_t r = gcd % b2; gcd = b2; b2 = r; }
        const int64_t unit = cgs / gcd;                 // blocks per whole number of groups
        int64_t want = (npix * cgs + kThreads - 1) / kThreads;
        if (want > 152 * 8) want = 152 * 8;
        want = (want + unit - 1) / unit * unit;
        if (want < unit) want = unit;
        const int g = (int)want;
        const int cc = concat != 0, rl = relu != 0;
        for (int pass = 0; pass < 2; pass++) {
            kt_pre(st);
            if (!plain) {
                if (pass == 0)
                    k_comb4f<0, 2, 8, 2, false><<<g, kThreads, 0, st>>>(T, cc, npix, cgs, rl, F, B,
                                                                        hdr, out, dhw, any_bcast);
                else
                    k_comb4f<1, 2, 8, 2, false><<<g, kThreads, 0, st>>>(T, cc, npix, cgs, rl, F, B,
                                                                        hdr, out, dhw, any_bcast);
            } else if (maxcover <= 2) {
                if (pass == 0)
                    k_comb4f<0, 2, 16, 2, true><<<g, kThreads, 0, st>>>(T, cc, npix, cgs, rl, F, B,
                                                                        hdr, out, dhw, any_bcast);
                else
                    k_comb4f<1, 2, 16, 2, true><<<g, kThreads, 0, st>>>(T, cc, npix, cgs, rl, F, B,
                                                                        hdr, out, dhw, any_bcast);
            } else {
                if (pass == 0)
                    k_comb4f<0, 6, 16, 1, true><<<g, kThreads, 0, st>>>(T, cc, npix, cgs, rl, F, B,
                                                                        hdr, out, dhw, any_bcast);
                else
                    k_comb4f<1, 6, 16, 1, true><<<g, kThreads, 0, st>>>(T, cc, npix, cgs, rl, F, B,
                                                                        hdr, out, dhw, any_bcast);
            }
            IQ_LAUNCH_CHECK();
            kt_post_bytes(st, pass == 0 ? IQ_KERNEL_COMBINE_MAX : IQ_KERNEL_COMBINE_CODES,
                          pass == 0 ? in_b : in_b + out_b);
            if (pass == 0) {
                k_comb_params<<<1, 1, 0, st>>>(hdr, s_out);
                IQ_LAUNCH_CHECK();
            }
        }
        return IQ_OK;
    }
    // at most two operands cover any 4-channel group: sums of up to two operands, and
    // concatenations whose ranges overlap at most pairwise (checked per group on the host)
    bool two = vec4;
    for (int co = 0; co < c_out && two; co += 4) {
        int nc = 0;
        for (int i = 0; i < n_terms; i++) {
            const TermDev& t = T.t[i];
            const int ch = concat ? co - t.c_offset : co;
            if (ch >= 0 && ch < t.c) nc++;
        }
        two = nc <= 2;
    }
    if (two) {
        const int cgs = c_out / 4;
        const int64_t npix = n * hw;
        // a multiple of cgs threads, about 8 blocks of 256 per SM
        int64_t gcd = cgs, b2 = kThreads;
        while (b2) { int64_t r = gcd % b2; gcd = b2; b2 = r; }
        const int64_t unit = cgs / gcd;                 // blocks per whole number of groups
        int64_t want = (npix * cgs + kThreads - 1) / kThreads;
        if (want > 152 * 8) want = 152 * 8;
        want = (want + unit - 1) / unit * unit;
        if (want < unit) want = unit;
        const int g = (int)want;
        kt_pre(st);
        k_comb4r<0><<<g, kThreads, 0, st>>>(T, concat != 0, npix, cgs, relu != 0, F, B, hdr, out,
                                            dhw, any_bcast);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_COMBINE_MAX, in_b);
        k_comb_params<<<1, 1, 0, st>>>(hdr, s_out);
        IQ_LAUNCH_CHECK();
        kt_pre(st);
        k_comb4r<1><<<g, kThreads, 0, st>>>(T, concat != 0, npix, cgs, relu != 0, F, B, hdr, out,
                                            dhw, any_bcast);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_COMBINE_CODES, in_b + out_b);
        return IQ_OK;
    }
    if (vec) {
        const int64_t nvec = total / 8;
        const int g = grid_for(nvec, kThreads, 152 * 8);
        const UDiv dcg = make_udiv((uint64_t)(c_out / 8));
        kt_pre(st);
        k_comb8<0><<<g, kThreads, 0, st>>>(T, concat != 0, nvec, c_out / 8, relu != 0, F, B, hdr,
                                           out, dcg, dhw, any_bcast);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_COMBINE_MAX, in_b);
        k_comb_params<<<1, 1, 0, st>>>(hdr, s_out);
        IQ_LAUNCH_CHECK();
        kt_pre(st);
        k_comb8<1><<<g, kThreads, 0, st>>>(T, concat != 0, nvec, c_out / 8, relu != 0, F, B, hdr,
                                           out, dcg, dhw, any_bcast);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_COMBINE_CODES, in_b + out_b);
        return IQ_OK;
    }
    const int g = grid_for(total, kThreads, 152 * 8);
    const UDiv dc = make_udiv((uint64_t)c_out);
    kt_pre(st);
    k_comb<0><<<g, kThreads, 0, st>>>(T, concat != 0, n, hw, c_out, relu != 0, F, B, hdr, out,
                                      dc, dhw);
    IQ_LAUNCH_CHECK();
    kt_post_bytes(st, IQ_KERNEL_COMBINE_MAX, in_b);
    k_comb_params<<<1, 1, 0, st>>>(hdr, s_out);
    IQ_LAUNCH_CHECK();
    kt_pre(st);
    k_comb<1><<<g, kThreads, 0, st>>>(T, concat != 0, n, hw, c_out, relu != 0, F, B, hdr, out,
                                      dc, dhw);
    IQ_LAUNCH_CHECK();
    kt_post_bytes(st, IQ_KERNEL_COMBINE_CODES, in_b + out_b);
    return IQ_OK;
}

extern "C" iq_status iq_spatial_sum_workspace_size(int64_t n, int32_t c, size_t* bytes) {
    if (!bytes || n < 1 || c < 1) return IQ_ERR_INVALID_ARG;
    *bytes = (((size_t)n * c * 8) + 255) & ~size_t(255);
    return IQ_OK;
}

extern "C" iq_status iq_spatial_sum(const int8_t* x, const double* s_x, int64_t n, int64_t hw,
                                    int32_t c_total, int32_t c_off, int32_t c, int32_t mean,
                                    int8_t* out, double* s_out, void* ws, size_t ws_bytes,
                                    iq_stream stream) {
    if (!x || !s_x || !out || !s_out || n < 1 || n > 65535 || hw < 1 || c < 1 || c_off < 0 ||
        c_off + c > c_total)
        return IQ_ERR_INVALID_ARG;
    if (hw * 127 >= (int64_t(1) << 62) / 2) return IQ_ERR_INVALID_ARG;
    const size_t need = (((size_t)n * c * 8) + 255) & ~size_t(255);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    unsigned long long* sums = (unsigned long long*)ws;
    IQ_CUDA_CHECK(cudaMemsetAsync(sums, 0, (size_t)n * c * 8, st));
    const int cz = (c + kThreads - 1) / kThreads;
    // enough pixel slices that the grid covers the SMs a few times over
    int64_t slices = (152 * 8 + n * cz - 1) / (n * cz);
    if (slices > hw) slices = hw;
    if (slices < 1) slices = 1;
    if (slices > 65535) slices = 65535;
    const int64_t per = (hw + slices - 1) / slices;
    slices = (hw + per - 1) / per;
    dim3 grid((unsigned)slices, (unsigned)n, (unsigned)cz);
    k_ssum<<<grid, kThreads, 0, st>>>(x, hw, c_total, c_off, c, per, sums);
    IQ_LAUNCH_CHECK();
    k_ssum_finish<<<1, 1024, 0, st>>>(sums, n * c, s_x, mean ? (double)hw : 1.0, out, s_out);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_avgpool_bwd(const int8_t* e, const double* s_e, int64_t n, int64_t hw,
                                    int32_t c, int8_t* ex, double* s_ex, iq_stream stream) {
    if (!e || !s_e || !s_ex || n < 1 || hw < 1 || c < 1) return IQ_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    k_scale_div<<<1, 1, 0, st>>>(s_e, (double)hw, s_ex);
    IQ_LAUNCH_CHECK();
    if (ex) {
        k_bcast<<<grid_for(n * hw * c), kThreads, 0, st>>>(e, n, hw, c, ex,
                                                            make_udiv((uint64_t)(hw * c)));
        IQ_LAUNCH_CHECK();
    }
    return IQ_OK;
}

extern "C" iq_status iq_channel_slice(const int8_t* x, int64_t npix, int32_t c_total,
                                      int32_t c_off, int32_t c, int8_t* out, iq_stream stream) {
    if (!x || !out || npix < 0 || c < 1 || c_off < 0 || c_off + c > c_total)
        return IQ_ERR_INVALID_ARG;
    if (npix == 0) return IQ_OK;
    k_slice<<<grid_for(npix * c), kThreads, 0, (cudaStream_t)stream>>>(x, npix, c_total, c_off, c,
                                                                      out, make_udiv((uint64_t)c));
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}
