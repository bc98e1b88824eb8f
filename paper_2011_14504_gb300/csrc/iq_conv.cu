// iq_conv.cu -- the 8-bit convolution (the MAC of Sec. 3.2.3 on 8-bit W and A) as
// implicit GEMMs, forward, data gradient and weight gradient, plus the C ABI of the
// conv layer (Sec. 3.2 forward with Q_A or quantized L1BN, Sec. 3.3 backward).
//
// This file holds the portable CUDA-core path: 64x64 output tiles, 32-byte K
// slices staged in shared memory packed 4 codes per word, dp4a MACs with int32
// accumulation.  The tensor-core path (iq_conv_tc.cu) takes the shapes it supports.
#include "iq_internal.cuh"
#include "iq_conv_tc.cuh"

#include <algorithm>

#include <climits>

namespace iq {

enum ConvOp { OP_FWD = 0, OP_DGRAD = 1, OP_WGRAD = 2 };

struct ConvP {
    int N, H, W, C, K, R, S, sh, sw, ph, pw, dh, dw, G, P, Q;
    int Cg, Kg;
    int64_t M;       // GEMM rows: fwd N*P*Q, dgrad N*H*W, wgrad Kg
    int ncols;       // GEMM cols per group: fwd Kg, dgrad Cg, wgrad R*S*Cg
    int kin;         // fwd: Cg rounded up to 32; dgrad: Kg rounded up to 32
    int64_t npq;     // wgrad: N*P*Q
    int64_t chunk;   // wgrad: reduction length per split (multiple of 32)
    int nsplit;      // wgrad: splits per group
};

constexpr int BM = 64, BN = 64, BK = 32;

__device__ __forceinline__ void load8_bytes(const int8_t* p, int nvalid, uint32_t& lo,
                                            uint32_t& hi) {
    uint32_t b[8];
#pragma unroll
    for (int j = 0; j < 8; j++) b[j] = j < nvalid ? (uint32_t)(uint8_t)p[j] : 0u;
    lo = b[0] | (b[1] << 8) | (b[2] << 16) | (b[3] << 24);
    hi = b[4] | (b[5] << 8) | (b[6] << 16) | (b[7] << 24);
}

template <int OP, bool WIDE>
__global__ void __launch_bounds__(256) k_conv_simt(ConvP cp, const int8_t* __restrict__ A_src,
                                                   const int8_t* __restrict__ B_src,
                                                   int32_t* __restrict__ out32,
                                                   long long* __restrict__ out64,
                                                   unsigned long long* __restrict__ s1,
                                                   int* __restrict__ hi_c, int* __restrict__ lo_c,
                                                   unsigned long long* __restrict__ amax) {
    __shared__ __align__(16) uint32_t As[BK / 4][BM];
    __shared__ __align__(16) uint32_t Bs[BK / 4][BN];
    __shared__ int s_n[BK], s_p[BK], s_q[BK];
    __shared__ unsigned long long st_s1[BN];
    __shared__ int st_hi[BN], st_lo[BN];

    const int t = threadIdx.x;
    const int ty = t >> 4, tx = t & 15;
    const int lrow = t >> 2, lk = (t & 3) * 8;
    int g, split = 0;
    if (OP == OP_WGRAD) { g = blockIdx.z / cp.nsplit; split = blockIdx.z % cp.nsplit; }
    else g = blockIdx.z;
    const int64_t m0 = (int64_t)blockIdx.x * BM;
    const int n0 = blockIdx.y * BN;

    // per-thread decode of its load rows
    const int64_t am = m0 + lrow;           // A row
    const int bcol = n0 + lrow;             // B row (GEMM column)
    int a_n = 0, a_p = 0, a_q = 0;
    bool a_ok = am < cp.M;
    if (OP == OP_FWD && a_ok) {
        int64_t pq = (int64_t)cp.P * cp.Q;
        a_n = (int)(am / pq);
        int64_t rem = am - (int64_t)a_n * pq;
        a_p = (int)(rem / cp.Q);
        a_q = (int)(rem - (int64_t)a_p * cp.Q);
    } else if (OP == OP_DGRAD && a_ok) {
        int64_t hw = (int64_t)cp.H * cp.W;
        a_n = (int)(am / hw);
        int64_t rem = am - (int64_t)a_n * hw;
        a_p = (int)(rem / cp.W);   // input row h
        a_q = (int)(rem - (int64_t)a_p * cp.W);  // input col w
    }
    const bool b_ok = bcol < cp.ncols;
    int b_r = 0, b_s = 0, b_c = 0;
    if (OP == OP_WGRAD && b_ok) {
        b_c = bcol % cp.Cg;
        int rs = bcol / cp.Cg;
        b_r = rs / cp.S;
        b_s = rs % cp.S;
    }

    int acc[4][4];
    long long wacc[WIDE ? 4 : 1][WIDE ? 4 : 1];
#pragma unroll
    for (int i = 0; i < 4; i++)
#pragma unroll
        for (int j = 0; j < 4; j++) acc[i][j] = 0;
    if (WIDE) {
#pragma unroll
        for (int i = 0; i < (WIDE ? 4 : 1); i++)
#pragma unroll
            for (int j = 0; j < (WIDE ? 4 : 1); j++) wacc[i][j] = 0;
    }

    // K iteration space
    int64_t ktiles;
    int64_t kbase0 = 0;
    if (OP == OP_FWD) ktiles = (int64_t)cp.R * cp.S * (cp.kin / BK);
    else if (OP == OP_DGRAD) ktiles = (int64_t)cp.R * cp.S * (cp.kin / BK);
    else {
        kbase0 = (int64_t)split * cp.chunk;
        int64_t kend = kbase0 + cp.chunk;
        if (kend > cp.npq) kend = cp.npq;
        ktiles = kend > kbase0 ? (kend - kbase0 + BK - 1) / BK : 0;
    }
    const bool vec8 = (OP == OP_FWD) ? ((cp.Cg % 8) == 0 && (cp.C % 8) == 0)
                                     : (OP == OP_DGRAD) ? ((cp.Kg % 8) == 0 && (cp.K % 8) == 0)
                                                        : false;

    for (int64_t kt = 0; kt < ktiles; kt++) {
        uint32_t alo = 0, ahi = 0, blo = 0, bhi = 0;
        if (OP == OP_FWD || OP == OP_DGRAD) {
            int per = cp.kin / BK;
            int tap = (int)(kt / per);
            int c0 = (int)(kt - (int64_t)tap * per) * BK + lk;
            int r = tap / cp.S, s = tap % cp.S;
            int limit = (OP == OP_FWD) ? cp.Cg : cp.Kg;
            int nvalid = limit - c0;
            nvalid = nvalid < 0 ? 0 : (nvalid > 8 ? 8 : nvalid);
            if (OP == OP_FWD) {
                int hh = a_p * cp.sh + r * cp.dh - cp.ph;
                int ww = a_q * cp.sw + s * cp.dw - cp.pw;
                if (a_ok && nvalid > 0 && hh >= 0 && hh < cp.H && ww >= 0 && ww < cp.W) {
                    const int8_t* p = A_src + (((int64_t)a_n * cp.H + hh) * cp.W + ww) * cp.C +
                                      (int64_t)g * cp.Cg + c0;
                    if (vec8) { int2 v = *reinterpret_cast<const int2*>(p); alo = v.x; ahi = v.y; }
                    else load8_bytes(p, nvalid, alo, ahi);
                }
                if (b_ok && nvalid > 0) {
                    int kg = g * cp.Kg + bcol;
                    const int8_t* p = B_src + (((int64_t)kg * cp.R + r) * cp.S + s) * cp.Cg + c0;
                    if (vec8) { int2 v = *reinterpret_cast<const int2*>(p); blo = v.x; bhi = v.y; }
                    else load8_bytes(p, nvalid, blo, bhi);
                }
            } else {
                int ph_ = a_p + cp.ph - r * cp.dh;
                int pw_ = a_q + cp.pw - s * cp.dw;
                bool ok = a_ok && nvalid > 0 && ph_ >= 0 && pw_ >= 0 && (ph_ % cp.sh) == 0 &&
                          (pw_ % cp.sw) == 0;
                if (ok) {
                    int p = ph_ / cp.sh, q = pw_ / cp.sw;
                    if (p < cp.P && q < cp.Q) {
                        const int8_t* src = A_src + (((int64_t)a_n * cp.P + p) * cp.Q + q) * cp.K +
                                            (int64_t)g * cp.Kg + c0;
                        if (vec8) { int2 v = *reinterpret_cast<const int2*>(src); alo = v.x; ahi = v.y; }
                        else load8_bytes(src, nvalid, alo, ahi);
                    }
                }
                if (b_ok && nvalid > 0) {
                    // transposed weights [G][Cg][R][S][Kg]
                    const int8_t* src = B_src + ((((int64_t)g * cp.Cg + bcol) * cp.R + r) * cp.S + s) *
                                                    cp.Kg + c0;
                    if (vec8) { int2 v = *reinterpret_cast<const int2*>(src); blo = v.x; bhi = v.y; }
                    else load8_bytes(src, nvalid, blo, bhi);
                }
            }
        } else {
            // wgrad: decode the 32 reduction pixels of this tile once
            int64_t kb = kbase0 + kt * BK;
            if (t < BK) {
                int64_t j = kb + t;
                int64_t kend = kbase0 + cp.chunk;
                if (j < cp.npq && j < kend) {
                    int64_t pq = (int64_t)cp.P * cp.Q;
                    int nn = (int)(j / pq);
                    int64_t rem = j - (int64_t)nn * pq;
                    s_n[t] = nn;
                    s_p[t] = (int)(rem / cp.Q);
                    s_q[t] = (int)(rem - (int64_t)s_p[t] * cp.Q);
                } else {
                    s_n[t] = -1;
                }
            }
            __syncthreads();
            uint32_t ab[8], bb[8];
#pragma unroll
            for (int j = 0; j < 8; j++) {
                int jj = lk + j;
                int nn = s_n[jj];
                ab[j] = 0; bb[j] = 0;
                if (nn >= 0) {
                    int64_t pix = ((int64_t)nn * cp.P + s_p[jj]) * cp.Q + s_q[jj];
                    if (a_ok) ab[j] = (uint8_t)A_src[pix * cp.K + (int64_t)g * cp.Kg + am];
                    if (b_ok) {
                        int hh = s_p[jj] * cp.sh + b_r * cp.dh - cp.ph;
                        int ww = s_q[jj] * cp.sw + b_s * cp.dw - cp.pw;
                        if (hh >= 0 && hh < cp.H && ww >= 0 && ww < cp.W)
                            bb[j] = (uint8_t)B_src[(((int64_t)nn * cp.H + hh) * cp.W + ww) * cp.C +
                                                   (int64_t)g * cp.Cg + b_c];
                    }
                }
            }
            alo = ab[0] | (ab[1] << 8) | (ab[2] << 16) | (ab[3] << 24);
            ahi = ab[4] | (ab[5] << 8) | (ab[6] << 16) | (ab[7] << 24);
            blo = bb[0] | (bb[1] << 8) | (bb[2] << 16) | (bb[3] << 24);
            bhi = bb[4] | (bb[5] << 8) | (bb[6] << 16) | (bb[7] << 24);
        }
        As[lk / 4][lrow] = alo;
        As[lk / 4 + 1][lrow] = ahi;
        Bs[lk / 4][lrow] = blo;
        Bs[lk / 4 + 1][lrow] = bhi;
        __syncthreads();
#pragma unroll
        for (int kw = 0; kw < BK / 4; kw++) {
            uint4 av = *reinterpret_cast<const uint4*>(&As[kw][ty * 4]);
            uint4 bv = *reinterpret_cast<const uint4*>(&Bs[kw][tx * 4]);
            int a4[4] = {(int)av.x, (int)av.y, (int)av.z, (int)av.w};
            int b4[4] = {(int)bv.x, (int)bv.y, (int)bv.z, (int)bv.w};
#pragma unroll
            for (int i = 0; i < 4; i++)
#pragma unroll
                for (int j = 0; j < 4; j++) acc[i][j] = __dp4a(a4[i], b4[j], acc[i][j]);
        }
        __syncthreads();
        if (WIDE) {
            // fold the 32-product tile sums into int64 (the reduction exceeds int32 range)
#pragma unroll
            for (int i = 0; i < 4; i++)
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    wacc[i & (WIDE ? 3 : 0)][j & (WIDE ? 3 : 0)] += acc[i][j];
                    acc[i][j] = 0;
                }
        }
    }

    // ---------------- epilogue
    if (OP == OP_FWD) {
        if (t < BN) { st_s1[t] = 0; st_hi[t] = INT_MIN; st_lo[t] = INT_MAX; }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 4; j++) {
            int col = n0 + tx * 4 + j;
            if (col >= cp.ncols) continue;
            long long sum = 0;
            int h = INT_MIN, l = INT_MAX;
            bool any = false;
#pragma unroll
            for (int i = 0; i < 4; i++) {
                int64_t m = m0 + ty * 4 + i;
                if (m >= cp.M) continue;
                int v = acc[i][j];
                out32[m * cp.K + (int64_t)g * cp.Kg + col] = v;
                sum += v; h = max(h, v); l = min(l, v); any = true;
            }
            if (any) {
                atomicAdd(&st_s1[tx * 4 + j], (unsigned long long)sum);
                atomicMax(&st_hi[tx * 4 + j], h);
                atomicMin(&st_lo[tx * 4 + j], l);
            }
        }
        __syncthreads();
        if (t < BN && n0 + t < cp.ncols && s1) {
            int c = g * cp.Kg + n0 + t;
            atomicAdd(&s1[c], st_s1[t]);
            atomicMax(&hi_c[c], st_hi[t]);
            atomicMin(&lo_c[c], st_lo[t]);
        }
    } else if (OP == OP_DGRAD) {
        uint64_t mx = 0;
#pragma unroll
        for (int i = 0; i < 4; i++) {
            int64_t m = m0 + ty * 4 + i;
            if (m >= cp.M) continue;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                int col = n0 + tx * 4 + j;
                if (col >= cp.ncols) continue;
                long long v = WIDE ? wacc[i & (WIDE ? 3 : 0)][j & (WIDE ? 3 : 0)] : acc[i][j];
                if (WIDE) out64[m * cp.C + (int64_t)g * cp.Cg + col] = v;
                else out32[m * cp.C + (int64_t)g * cp.Cg + col] = (int)v;
                uint64_t a = (uint64_t)(v < 0 ? -v : v);
                mx = a > mx ? a : mx;
            }
        }
        mx = warp_max_u64(mx);
        if ((t & 31) == 0 && mx) atomicMax(amax, (unsigned long long)mx);
    } else {
#pragma unroll
        for (int i = 0; i < 4; i++) {
            int64_t k = m0 + ty * 4 + i;
            if (k >= cp.M) continue;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                int col = n0 + tx * 4 + j;
                if (col >= cp.ncols || acc[i][j] == 0) continue;
                atomicAdd(reinterpret_cast<unsigned long long*>(
                              &out64[((int64_t)g * cp.Kg + k) * cp.ncols + col]),
                          (unsigned long long)(long long)acc[i][j]);
            }
        }
    }
}

// dgrad weights: w[K][R][S][Cg] -> wT[G][Cg][R][S][Kg]
__global__ void k_transpose_w(const int8_t* __restrict__ w, int8_t* __restrict__ wt, int K,
                              int R, int S, int Cg, int G) {
    int Kg = K / G;
    int64_t total = (int64_t)K * R * S * Cg;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        int c = (int)(i % Cg);
        int64_t t = i / Cg;
        int s = (int)(t % S); t /= S;
        int r = (int)(t % R);
        int k = (int)(t / R);
        int g = k / Kg, kl = k % Kg;
        wt[((((int64_t)g * Cg + c) * R + r) * S + s) * Kg + kl] = w[i];
    }
}

// ------------------------------------------------------------------ small scale kernels

// Channel padding for the tensor-core kernels (output channels a multiple of 8 in the
// forward, error channels a multiple of 8 in the data gradient):
// dst[i][j] = j < cols ? src[i][j] : 0 for rows of cols_p >= cols bytes.
__global__ void k_pad_cols_i8(const int8_t* __restrict__ src, int64_t rows, int cols, int cols_p,
                              int8_t* __restrict__ dst) {
    const int64_t n = rows * cols_p;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / cols_p;
        const int j = (int)(i - r * cols_p);
        dst[i] = j < cols ? src[r * cols + j] : (int8_t)0;
    }
}
// dst[i][j] = src[i][j] for j < cols from rows of cols_p int32
__global__ void k_compact_cols_i32(const int32_t* __restrict__ src, int64_t rows, int cols,
                                   int cols_p, int32_t* __restrict__ dst) {
    const int64_t n = rows * cols;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / cols;
        dst[i] = src[r * cols_p + (i - r * cols)];
    }
}

__global__ void k_scale_mul_pow2(const double* __restrict__ a, int e, double* __restrict__ out) {
    *out = ldexp(*a, e);
}
__global__ void k_scale_mul(const double* __restrict__ a, const double* __restrict__ b,
                            double* __restrict__ out) {
    *out = __dmul_rn(*a, *b);
}
// M for SQ of the conv output from the per-channel extremes
// One block: M = max |acc| (of ReLU(acc) when relu) from the per-channel extremes, then the
// SQ_8 parameters and the output scale s_in M 2^-7 (the requantizer's finalize step).
__global__ void k_max_from_stats(const int* __restrict__ hi, const int* __restrict__ lo, int C,
                                 int relu, const double* __restrict__ s_in,
                                 unsigned long long* __restrict__ cell, RqParams* __restrict__ prm,
                                 double* __restrict__ s_out, int k = 8) {
    __shared__ unsigned long long red[32];
    uint64_t m = 0;
    for (int c = threadIdx.x; c < C; c += blockDim.x) {
        int64_t h = hi[c], l = lo[c];
        // a channel no extreme was written to (kernels that keep only the extremes of the
        // whole output write channel 0; under ReLU only the maxima, INT_MIN when untouched)
        if (!relu && h < l) continue;
        uint64_t v = relu ? (uint64_t)(h > 0 ? h : 0)
                          : (uint64_t)max(h < 0 ? -h : h, l < 0 ? -l : l);
        m = v > m ? v : m;
    }
    m = warp_max_u64(m);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x < 32) {
        uint64_t r = threadIdx.x < (blockDim.x + 31) / 32 ? red[threadIdx.x] : 0;
        r = warp_max_u64(r);
        if (threadIdx.x == 0) {
            *cell = r;
            const RqParams p = rq_params_make(r, *s_in, k, relu ? IQ_MODE_SQ_RELU : IQ_MODE_SQ);
            *prm = p;
            *s_out = p.s_out;
        }
    }
}

// ------------------------------------------------------------------ geometry helpers

static bool desc_ok(const iq_conv_desc* d) {
    if (!d) return false;
    if (d->n <= 0 || d->h <= 0 || d->w <= 0 || d->c <= 0 || d->k <= 0 || d->r <= 0 || d->s <= 0)
        return false;
    if (d->stride_h <= 0 || d->stride_w <= 0 || d->pad_h < 0 || d->pad_w < 0 || d->dil_h <= 0 ||
        d->dil_w <= 0 || d->groups <= 0)
        return false;
    if (d->c % d->groups || d->k % d->groups) return false;
    if (d->layout != IQ_LAYOUT_NHWC && d->layout != IQ_LAYOUT_NCHW) return false;
    if (d->k_w != 0 && (d->k_w < 2 || d->k_w > 8)) return false;
    if (d->k_a != 0 && (d->k_a < 2 || d->k_a > 8)) return false;
    if (d->flags & ~(IQ_CONV_X_F16_READY | IQ_CONV_E_F16_READY)) return false;
    int p = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1);
    int q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1);
    return p >= 0 && q >= 0;
}

// the code widths of a descriptor (0: the paper's 8 bits)
static int code_kw(const iq_conv_desc* d) { return d->k_w ? d->k_w : 8; }
// Q_A width: the descriptor's, else the bits argument's (batch norm), else 8; -1 when both
// are given and differ
static int code_ka(const iq_conv_desc* d, const iq_bn_bits* bits) {
    if (d->k_a && bits && bits->k_a != d->k_a) return -1;
    return d->k_a ? d->k_a : (bits ? bits->k_a : 8);
}

static ConvP make_params(const iq_conv_desc* d) {
    ConvP c;
    c.N = d->n; c.H = d->h; c.W = d->w; c.C = d->c; c.K = d->k; c.R = d->r; c.S = d->s;
    c.sh = d->stride_h; c.sw = d->stride_w; c.ph = d->pad_h; c.pw = d->pad_w;
    c.dh = d->dil_h; c.dw = d->dil_w; c.G = d->groups;
    c.P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    c.Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    c.Cg = d->c / d->groups;
    c.Kg = d->k / d->groups;
    c.M = 0; c.ncols = 0; c.kin = 0; c.npq = (int64_t)c.N * c.P * c.Q; c.chunk = 0; c.nsplit = 1;
    return c;
}

static int64_t roundup(int64_t a, int64_t b) { return (a + b - 1) / b * b; }

struct FwdWs {
    int32_t* acc;
    BnStats st;
    void* rq;
    double* s_acc;
    void* tc;
    int32_t* accp;     // output channels padded to a multiple of 8: the padded sums
    int8_t* wp;        //   and the weights with zero rows appended
};

// output channels not a multiple of 8 (single group): the tensor-core forward runs on
// weights padded to kpad(d) rows
static int fwd_kpad(const iq_conv_desc* d) {
    return (d->groups == 1 && d->k % 8 && d->c % 4 == 0) ? (d->k + 7) / 8 * 8 : 0;
}

static size_t fwd_ws_layout(const iq_conv_desc* d, int with_acc, void* base, size_t cap,
                            FwdWs* out) {
    ConvP cp = make_params(d);
    WsCursor cur(base, cap);
    FwdWs w;
    const int kp = fwd_kpad(d);
    w.acc = with_acc ? cur.take<int32_t>((size_t)cp.npq * cp.K) : nullptr;
    w.st = bn_stats_carve(cur, kp ? kp : cp.K);
    w.rq = cur.take<char>(requant_ws_bytes());
    w.s_acc = cur.take<double>(1);
    iq_conv_desc dp = *d;
    if (kp) dp.k = kp;
    w.tc = cur.take<char>(conv_fwd_tc_ws_bytes(&dp));
    w.accp = kp ? cur.take<int32_t>((size_t)cp.npq * kp) : nullptr;
    w.wp = kp ? cur.take<int8_t>((size_t)kp * d->r * d->s * d->c) : nullptr;
    if (out) *out = w;
    return cur.off + 256;
}

}  // namespace iq

using namespace iq;

// ==================================================================== C ABI

extern "C" iq_status iq_conv_out_size(const iq_conv_desc* d, int32_t* p, int32_t* q) {
    if (!desc_ok(d) || !p || !q) return IQ_ERR_INVALID_ARG;
    ConvP c = make_params(d);
    *p = c.P;
    *q = c.Q;
    return IQ_OK;
}

// bytes of the NCHW staging buffers in front of the NHWC workspace (0 for NHWC)
static size_t nchw_stage_bytes(const iq_conv_desc* d, int op);

extern "C" iq_status iq_conv_fwd_workspace_size(const iq_conv_desc* d, int with_bn, size_t* bytes) {
    (void)with_bn;
    if (!desc_ok(d) || !bytes) return IQ_ERR_INVALID_ARG;
    *bytes = fwd_ws_layout(d, 1, nullptr, 0, nullptr) + nchw_stage_bytes(d, 1);
    return IQ_OK;
}

static bool dgrad_wide(const iq_conv_desc* d) {
    int64_t krs = (int64_t)(d->k / d->groups) * d->r * d->s;
    return krs * 127 * 127 >= (int64_t(1) << 31);
}

// error channels not a multiple of 8 (single group, stride 1, int32 sums): the tensor-core
// data gradient runs on errors and weights zero-padded to dgrad_kpad(d) channels
static int dgrad_kpad(const iq_conv_desc* d) {
    if (d->groups != 1 || d->stride_h != 1 || d->stride_w != 1 || d->k % 8 == 0 || d->c % 8)
        return 0;
    const int kp = (d->k + 7) / 8 * 8;
    if ((int64_t)kp * d->r * d->s * 16129 >= (int64_t(1) << 31)) return 0;
    iq_conv_desc dp = *d;
    dp.k = kp;
    return conv_dgrad_tc_supported(&dp) ? kp : 0;
}

static size_t dgrad_pad_ws(const iq_conv_desc* d) {
    const int kp = dgrad_kpad(d);
    if (!kp) return 0;
    iq_conv_desc dp = *d;
    dp.k = kp;
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    return conv_dgrad_tc_ws_bytes(&dp) + ((size_t)d->n * P * Q * kp + 255) / 256 * 256 +
           ((size_t)kp * d->r * d->s * d->c + 255) / 256 * 256 + 512;
}

extern "C" iq_status iq_conv_dgrad_workspace_size(const iq_conv_desc* d, size_t* bytes) {
    if (!desc_ok(d) || !bytes) return IQ_ERR_INVALID_ARG;
    WsCursor cur(nullptr, 0);
    cur.take<int8_t>((size_t)d->k * d->r * d->s * (d->c / d->groups));
    cur.take<int64_t>((size_t)d->n * d->h * d->w * d->c);   // int32, or int64 when wide
    cur.take<char>(requant_ws_bytes());
    cur.take<double>(1);
    bn_stats_carve(cur, d->c);
    cur.take<char>(std::max({conv_dgrad_tc_ws_bytes(d), conv_dgrad_tc_stride2_ws_bytes(d),
                             dgrad_pad_ws(d)}));
    *bytes = cur.off + 256 + nchw_stage_bytes(d, 2);
    return IQ_OK;
}

extern "C" iq_status iq_conv_wgrad_workspace_size(const iq_conv_desc* d, size_t* bytes) {
    if (!desc_ok(d) || !bytes) return IQ_ERR_INVALID_ARG;
    WsCursor cur(nullptr, 0);
    cur.take<int64_t>((size_t)d->k * d->r * d->s * (d->c / d->groups));
    cur.take<char>(requant_ws_bytes());
    cur.take<double>(1);
    cur.take<char>(conv_wgrad_tc_ws_bytes(d));
    *bytes = cur.off + 256 + nchw_stage_bytes(d, 3);
    return IQ_OK;
}

static bool crs_overflow(const iq_conv_desc* d) {
    int64_t crs = (int64_t)(d->c / d->groups) * d->r * d->s;
    return crs * 127 * 127 >= (int64_t(1) << 31);
}

// multiply-accumulates of one convolution pass, dense: N P Q K R S C / groups (every tap,
// the zero padding included)
static double conv_macs_dense(const iq_conv_desc* d) {
    const int64_t P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int64_t Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    return (double)d->n * P * Q * d->k * d->r * d->s * (double)(d->c / d->groups);
}

// number of (output index, tap) pairs of one spatial dimension whose input index
// o stride + t dil - pad lies inside [0, extent)
static int64_t inbounds_pairs(int64_t extent, int64_t out, int taps, int stride, int dil,
                              int pad) {
    int64_t n = 0;
    for (int t = 0; t < taps; t++)
        for (int64_t o = 0; o < out; o++) {
            const int64_t i = o * stride + (int64_t)t * dil - pad;
            n += i >= 0 && i < extent;
        }
    return n;
}

// the algorithmic multiply-accumulates: only the taps that read inside the input
static double conv_macs(const iq_conv_desc* d) {
    const int64_t P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int64_t Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    return (double)d->n * d->k * (double)(d->c / d->groups) *
           (double)inbounds_pairs(d->h, P, d->r, d->stride_h, d->dil_h, d->pad_h) *
           (double)inbounds_pairs(d->w, Q, d->s, d->stride_w, d->dil_w, d->pad_w);
}

// ------------------------------------------------------------------ kernel timing

namespace iq {
namespace {

constexpr int kKtCap = 8192;

struct KtState {
    bool on = false;
    int n = 0;
    int op = 0;
    double pending_macs = 0.0;      // the current call's MACs, given to its first launch
    double pending_dense = 0.0;
    cudaEvent_t ev[2 * kKtCap] = {};
    int kernel[kKtCap] = {};
    int opv[kKtCap] = {};
    double macs[kKtCap] = {};
    double dense[kKtCap] = {};
    double bytes[kKtCap] = {};
};

KtState& kt() {
    static KtState* s = new KtState();
    return *s;
}

void kt_record(cudaStream_t st, int kernel, double macs, double dense, double bytes, int op) {
    KtState& k = kt();
    if (!k.on || k.n >= kKtCap || !k.ev[2 * k.n]) return;
    cudaEvent_t& e = k.ev[2 * k.n + 1];
    if (!e && cudaEventCreate(&e) != cudaSuccess) { e = nullptr; return; }
    cudaEventRecord(e, st);
    k.kernel[k.n] = kernel;
    k.opv[k.n] = op;
    k.macs[k.n] = macs;
    k.dense[k.n] = dense;
    k.bytes[k.n] = bytes;
    k.n++;
}

}  // namespace

void kt_set_op(int op, double macs, double dense) {
    KtState& k = kt();
    k.op = op;
    k.pending_macs = macs;
    k.pending_dense = dense;
}

void kt_pre(cudaStream_t st) {
    KtState& k = kt();
    if (!k.on || k.n >= kKtCap) return;
    cudaEvent_t& e = k.ev[2 * k.n];
    if (!e && cudaEventCreate(&e) != cudaSuccess) { e = nullptr; return; }
    cudaEventRecord(e, st);
}

void kt_post(cudaStream_t st, int kernel) {
    KtState& k = kt();
    if (!k.on) return;
    kt_record(st, kernel, k.pending_macs, k.pending_dense, 0.0, k.op);
    k.pending_macs = 0.0;
    k.pending_dense = 0.0;
}

void kt_post_bytes(cudaStream_t st, int kernel, double bytes) {
    kt_record(st, kernel, 0.0, 0.0, bytes, 0);
}

}  // namespace iq

extern "C" iq_status iq_kernel_timing_begin(void) {
    KtState& k = kt();
    k.on = true;
    k.n = 0;
    k.pending_macs = 0.0;
    k.pending_dense = 0.0;
    return IQ_OK;
}

extern "C" iq_status iq_kernel_timing_end(iq_kernel_time* out, int32_t capacity, int32_t* n_out) {
    if (!out || !n_out || capacity < 0) return IQ_ERR_INVALID_ARG;
    KtState& k = kt();
    k.on = false;
    int nout = 0;
    iq_status r = IQ_OK;
    for (int i = 0; i < k.n; i++) {
        float ms = 0.0f;
        if (cudaEventSynchronize(k.ev[2 * i + 1]) != cudaSuccess ||
            cudaEventElapsedTime(&ms, k.ev[2 * i], k.ev[2 * i + 1]) != cudaSuccess) {
            r = IQ_ERR_CUDA;
            continue;
        }
        int j = 0;
        while (j < nout && !(out[j].kernel == k.kernel[i] && out[j].op == k.opv[i])) j++;
        if (j == nout) {
            if (nout == capacity) continue;
            out[j].kernel = k.kernel[i];
            out[j].op = k.opv[i];
            out[j].launches = 0;
            out[j].pad = 0;
            out[j].ms = 0.0;
            out[j].macs = 0.0;
            out[j].dense_macs = 0.0;
            out[j].bytes = 0.0;
            nout++;
        }
        out[j].launches++;
        out[j].ms += ms;
        out[j].macs += k.macs[i];
        out[j].dense_macs += k.dense[i];
        out[j].bytes += k.bytes[i];
    }
    k.n = 0;
    *n_out = nout;
    return r;
}

static iq_status conv_fwd_nhwc(const iq_conv_desc* d, const int8_t* x, const double* s_x,
                               const int8_t* w, const int32_t* gamma, const int32_t* beta,
                               const iq_bn_bits* bits, int use_bn, int relu, int8_t* a,
                               double* s_a, int16_t* xhat, int32_t* bn_codes, double* bn_scales,
                               int64_t* frozen_out, int32_t* acc_out, void* x_f16, void* a_f16,
                               void* ws, size_t ws_bytes, iq_stream stream) {
    if (!desc_ok(d) || !x || !s_x || !w || !a || !s_a) return IQ_ERR_INVALID_ARG;
    const int64_t nx = (int64_t)d->n * d->h * d->w * d->c;
    if (x_f16 && (nx % 16 || (((uintptr_t)x | (uintptr_t)x_f16) & 15))) return IQ_ERR_INVALID_ARG;
    if (a_f16) {
        int32_t pp = 0, qq = 0;
        iq_conv_out_size(d, &pp, &qq);
        if (!f16_copy_ok(a, a_f16, (int64_t)d->n * pp * qq * d->k)) return IQ_ERR_INVALID_ARG;
    }
    if (crs_overflow(d)) return IQ_ERR_OVERFLOW_RISK;
    kt_set_op(1, conv_macs(d), conv_macs_dense(d));
    iq_bn_bits b = bn_bits_or_default(bits);
    const int ka = code_ka(d, bits);
    if (ka < 0) return IQ_ERR_INVALID_ARG;
    b.k_a = ka;
    if (use_bn) {
        if (!gamma || !beta || !bn_bits_valid(b)) return IQ_ERR_INVALID_ARG;
        if (d->k % 4) return IQ_ERR_UNSUPPORTED;
        if (((uintptr_t)a | (uintptr_t)xhat | (uintptr_t)acc_out) & 15) return IQ_ERR_INVALID_ARG;
    }
    cudaStream_t st = (cudaStream_t)stream;
    FwdWs L;
    size_t need = fwd_ws_layout(d, acc_out == nullptr, nullptr, 0, nullptr);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    fwd_ws_layout(d, acc_out == nullptr, ws, ws_bytes, &L);
    int32_t* acc = acc_out ? acc_out : L.acc;
    ConvP cp = make_params(d);
    cp.M = cp.npq;
    cp.ncols = cp.Kg;
    cp.kin = (int)roundup(cp.Cg, BK);

    iq_status r = bn_stats_init(L.st, cp.K, st);
    if (r != IQ_OK) return r;
    k_scale_mul_pow2<<<1, 1, 0, st>>>(s_x, 1 - code_kw(d), L.s_acc);  // s_acc = s_x 2^(1-k_w)
    IQ_LAUNCH_CHECK();
    bool done = false;
    if (x_f16 && !(d->flags & IQ_CONV_X_F16_READY)) {
        r = codes_to_f16(x, (__half*)x_f16, nx, st);
        if (r != IQ_OK) return r;
    }
    // batch norm reads the sums and both extremes; SQ of ReLU(acc) only the maxima
    // (the batch-norm deviation pass computes the per-channel extremes itself)
    const unsigned want = use_bn ? (TC_STATS_SUM | TC_STATS_NOEXT) : (relu ? 0u : TC_STATS_LO);
    const int kp = use_bn ? 0 : fwd_kpad(d);
    if (kp) {
        // zero weight rows up to kp output channels, the padded sums compacted to k columns
        // (the zero channels cannot raise the maximum the requantizer takes)
        iq_conv_desc dp = *d;
        dp.k = kp;
        const int64_t rsc = (int64_t)d->r * d->s * d->c;
        k_pad_cols_i8<<<grid_for((int64_t)kp * rsc), kThreads, 0, st>>>(w, 1, (int)(d->k * rsc),
                                                                         (int)(kp * rsc), L.wp);
        IQ_LAUNCH_CHECK();
        r = bn_stats_init(L.st, kp, st);
        if (r != IQ_OK) return r;
        r = conv_fwd_tc(&dp, x, L.wp, L.accp, L.st.s1, L.st.hi, L.st.lo, L.tc, st, &done,
                        (const __half*)x_f16, want);
        if (r != IQ_OK) return r;
        if (done) {
            k_compact_cols_i32<<<grid_for(cp.npq * cp.K), kThreads, 0, st>>>(L.accp, cp.npq, cp.K,
                                                                            kp, acc);
            IQ_LAUNCH_CHECK();
        }
    } else {
        r = conv_fwd_tc(d, x, w, acc, L.st.s1, L.st.hi, L.st.lo, L.tc, st, &done,
                        (const __half*)x_f16, want);
        if (r != IQ_OK) return r;
    }
    if (!done) {
        dim3 grid((unsigned)((cp.M + BM - 1) / BM), (unsigned)((cp.ncols + BN - 1) / BN), cp.G);
        kt_pre(st);
        k_conv_simt<OP_FWD, false><<<grid, 256, 0, st>>>(cp, x, w, acc, nullptr, L.st.s1, L.st.hi,
                                                  L.st.lo, nullptr);
        IQ_LAUNCH_CHECK();
        kt_post(st, IQ_KERNEL_CONV_SIMT);
    }
    if (use_bn)
        return bn_fwd_after_stats(acc, cp.M, cp.K, L.s_acc, gamma, beta, b, L.st, xhat, a, s_a,
                                  bn_codes, bn_scales, frozen_out, st, (__half*)a_f16);
    // Q_A = SQ(act(acc), 8) with M from the per-channel extremes
    unsigned long long* cell = (unsigned long long*)L.rq;
    k_max_from_stats<<<1, 1024, 0, st>>>(L.st.hi, L.st.lo, cp.K, relu, L.s_acc, cell,
                                         rq_params_slot(L.rq), s_a, ka);
    IQ_LAUNCH_CHECK();
    if (frozen_out)      // M, the maximum of act(acc) Q_A divides by
        IQ_CUDA_CHECK(cudaMemcpyAsync(frozen_out, cell, sizeof(int64_t), cudaMemcpyDeviceToDevice,
                                      st));
    return requant_apply(acc, IQ_I32, cp.npq * cp.K, L.s_acc, ka,
                         relu ? IQ_MODE_SQ_RELU : IQ_MODE_SQ, 0, 0, 0, 0, a, IQ_I8, s_a, L.rq, st,
                         true, false, (__half*)a_f16);
}

// frozen Q_A parameters from the calibration maximum M = frozen[0]
__global__ void k_frozen_sq_params(const int64_t* __restrict__ frozen, int k, int relu,
                                   RqParams* __restrict__ prm) {
    const int64_t M = frozen[0];
    *prm = rq_params_make(M > 0 ? (uint64_t)M : 0, 1.0, k, relu ? IQ_MODE_SQ_RELU : IQ_MODE_SQ);
}

// The inference forward with frozen statistics: the conv into int32 accumulators (no
// statistics), then the calibration call's output map in one pass.
static iq_status conv_fwd_frozen_nhwc(const iq_conv_desc* d, const int8_t* x, const int8_t* w,
                                      const int64_t* frozen, const iq_bn_bits* bits, int use_bn,
                                      int relu, int8_t* a, int16_t* xhat, void* x_f16, void* ws,
                                      size_t ws_bytes, iq_stream stream) {
    if (!desc_ok(d) || !x || !w || !frozen || !a) return IQ_ERR_INVALID_ARG;
    const int64_t nx = (int64_t)d->n * d->h * d->w * d->c;
    if (x_f16 && (nx % 16 || (((uintptr_t)x | (uintptr_t)x_f16) & 15))) return IQ_ERR_INVALID_ARG;
    if (crs_overflow(d)) return IQ_ERR_OVERFLOW_RISK;
    iq_bn_bits b = bn_bits_or_default(bits);
    const int ka = code_ka(d, bits);
    if (ka < 0) return IQ_ERR_INVALID_ARG;
    b.k_a = ka;
    if (use_bn) {
        if (!bn_bits_valid(b)) return IQ_ERR_INVALID_ARG;
        if (d->k % 4) return IQ_ERR_UNSUPPORTED;
        if (((uintptr_t)a | (uintptr_t)xhat) & 15) return IQ_ERR_INVALID_ARG;
    } else if (xhat) {
        return IQ_ERR_INVALID_ARG;
    }
    kt_set_op(1, conv_macs(d), conv_macs_dense(d));
    cudaStream_t st = (cudaStream_t)stream;
    FwdWs L;
    size_t need = fwd_ws_layout(d, 1, nullptr, 0, nullptr);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    fwd_ws_layout(d, 1, ws, ws_bytes, &L);
    int32_t* acc = L.acc;
    ConvP cp = make_params(d);
    cp.M = cp.npq;
    cp.ncols = cp.Kg;
    cp.kin = (int)roundup(cp.Cg, BK);
    if (x_f16 && !(d->flags & IQ_CONV_X_F16_READY)) {
        iq_status r = codes_to_f16(x, (__half*)x_f16, nx, st);
        if (r != IQ_OK) return r;
    }
    const int kp = fwd_kpad(d);
    iq_status r = bn_stats_init(L.st, kp ? kp : cp.K, st);
    if (r != IQ_OK) return r;
    bool done = false;
    if (kp) {
        iq_conv_desc dp = *d;
        dp.k = kp;
        const int64_t rsc = (int64_t)d->r * d->s * d->c;
        k_pad_cols_i8<<<grid_for((int64_t)kp * rsc), kThreads, 0, st>>>(w, 1, (int)(d->k * rsc),
                                                                         (int)(kp * rsc), L.wp);
        IQ_LAUNCH_CHECK();
        r = conv_fwd_tc(&dp, x, L.wp, L.accp, L.st.s1, L.st.hi, L.st.lo, L.tc, st, &done,
                        (const __half*)x_f16, TC_STATS_NOEXT);
        if (r != IQ_OK) return r;
        if (done) {
            k_compact_cols_i32<<<grid_for(cp.npq * cp.K), kThreads, 0, st>>>(L.accp, cp.npq, cp.K,
                                                                            kp, acc);
            IQ_LAUNCH_CHECK();
        }
    } else {
        r = conv_fwd_tc(d, x, w, acc, L.st.s1, L.st.hi, L.st.lo, L.tc, st, &done,
                        (const __half*)x_f16, TC_STATS_NOEXT);
        if (r != IQ_OK) return r;
    }
    if (!done) {
        dim3 grid((unsigned)((cp.M + BM - 1) / BM), (unsigned)((cp.ncols + BN - 1) / BN), cp.G);
        kt_pre(st);
        k_conv_simt<OP_FWD, false><<<grid, 256, 0, st>>>(cp, x, w, acc, nullptr, L.st.s1, L.st.hi,
                                                  L.st.lo, nullptr);
        IQ_LAUNCH_CHECK();
        kt_post(st, IQ_KERNEL_CONV_SIMT);
    }
    if (use_bn) return bn_apply_fixed(acc, cp.M, cp.K, frozen, b.k_xhat, b.k_a, xhat, a, st);
    k_frozen_sq_params<<<1, 1, 0, st>>>(frozen, ka, relu, rq_params_slot(L.rq));
    IQ_LAUNCH_CHECK();
    return requant_apply(acc, IQ_I32, cp.npq * cp.K, L.s_acc, ka,
                         relu ? IQ_MODE_SQ_RELU : IQ_MODE_SQ, 0, 0, 0, 0, a, IQ_I8, L.s_acc, L.rq,
                         st, true, true);
}

static iq_status conv_dgrad_nhwc(const iq_conv_desc* d, const int8_t* e, const double* s_e,
                                 const int8_t* w, int8_t* dx, double* s_dx, int32_t* acc_out,
                                 void* e_f16, const int8_t* dx_mask, void* dx_f16, void* ws,
                                 size_t ws_bytes, iq_stream stream) {
    if (!desc_ok(d) || !e || !s_e || !w || !dx || !s_dx) return IQ_ERR_INVALID_ARG;
    const int64_t ndx = (int64_t)d->n * d->h * d->w * d->c;
    if (dx_f16 && (!f16_copy_ok(dx, dx_f16, ndx) || ((uintptr_t)dx_mask & 15)))
        return IQ_ERR_INVALID_ARG;
    __half* dx16 = (__half*)dx_f16;
    const bool wide = dgrad_wide(d);
    if (wide && acc_out) return IQ_ERR_UNSUPPORTED;   // the sums need 64 bits: no int32 copy
    if ((int64_t)(d->k / d->groups) * d->r * d->s >= (int64_t(1) << 31) / 4)
        return IQ_ERR_OVERFLOW_RISK;
    size_t need = 0;
    iq_conv_dgrad_workspace_size(d, &need);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    kt_set_op(2, conv_macs(d), conv_macs_dense(d));
    cudaStream_t st = (cudaStream_t)stream;
    ConvP cp = make_params(d);
    WsCursor cur(ws, ws_bytes);
    int8_t* wt = cur.take<int8_t>((size_t)d->k * d->r * d->s * cp.Cg);
    int64_t* accw = cur.take<int64_t>((size_t)d->n * d->h * d->w * d->c);
    void* rq = cur.take<char>(requant_ws_bytes());
    double* s_in = cur.take<double>(1);
    BnStats stats = bn_stats_carve(cur, d->c);
    const size_t tcb = std::max({conv_dgrad_tc_ws_bytes(d), conv_dgrad_tc_stride2_ws_bytes(d),
                                 dgrad_pad_ws(d)});
    void* tcws = cur.take<char>(tcb);
    const int64_t total = (int64_t)d->n * d->h * d->w * d->c;
    unsigned long long* cell = (unsigned long long*)rq;
    k_scale_mul_pow2<<<1, 1, 0, st>>>(s_e, 1 - code_kw(d), s_in);   // the W_q step 2^(1-k_w)
    IQ_LAUNCH_CHECK();
    int32_t* acc = acc_out ? acc_out : reinterpret_cast<int32_t*>(accw);
    if (e_f16 && !(d->flags & IQ_CONV_E_F16_READY)) {
        const int64_t ne = (int64_t)d->n * cp.P * cp.Q * d->k;
        iq_status r0 = codes_to_f16(e, (__half*)e_f16, ne, st);
        if (r0 != IQ_OK) return r0;
    }
    // tensor-core path: stride 1, as a forward pass over the errors
    if (conv_dgrad_tc_supported(d)) {
        bool done = false;
        iq_status r;
        if (wide) {
            IQ_CUDA_CHECK(cudaMemsetAsync(accw, 0, sizeof(int64_t) * total, st));
            r = conv_dgrad_tc(d, e, w, nullptr, (long long*)accw, nullptr, nullptr, nullptr, tcws,
                              st, &done, (const __half*)e_f16);
            if (r != IQ_OK) return r;
            if (done) {
                r = requant_int(accw, IQ_I64, total, s_in, 8, IQ_MODE_SQ, 0, 0, 0, 0, dx, IQ_I8,
                                s_dx, rq, st);
                if (r != IQ_OK || (!dx_mask && !dx16)) return r;
                return codes_mask_copy(dx, dx_mask, total, dx16, st);
            }
        } else {
            r = bn_stats_init(stats, d->c, st);
            if (r != IQ_OK) return r;
            r = conv_dgrad_tc(d, e, w, acc, nullptr, stats.s1, stats.hi, stats.lo, tcws, st, &done,
                              (const __half*)e_f16);
            if (r != IQ_OK) return r;
            if (done) {
                k_max_from_stats<<<1, 1024, 0, st>>>(stats.hi, stats.lo, d->c, 0, s_in, cell,
                                                     rq_params_slot(rq), s_dx);
                IQ_LAUNCH_CHECK();
                return requant_apply(acc, IQ_I32, total, s_in, 8, IQ_MODE_SQ, 0, 0, 0, 0, dx,
                                     IQ_I8, s_dx, rq, st, true, false, dx16, dx_mask);
            }
        }
    }
    // error channels padded to a multiple of 8: zero error channels and zero weight rows
    if (const int kp = !wide ? dgrad_kpad(d) : 0) {
        iq_conv_desc dp = *d;
        dp.k = kp;
        const int64_t npq = (int64_t)d->n * cp.P * cp.Q;
        const int64_t rsc = (int64_t)d->r * d->s * d->c;
        char* b = (char*)tcws;
        int8_t* ep = reinterpret_cast<int8_t*>(b);
        int8_t* wp = reinterpret_cast<int8_t*>(b + ((size_t)npq * kp + 255) / 256 * 256);
        void* tws = b + ((size_t)npq * kp + 255) / 256 * 256 + ((size_t)kp * rsc + 255) / 256 * 256;
        k_pad_cols_i8<<<grid_for(npq * kp), kThreads, 0, st>>>(e, npq, d->k, kp, ep);
        IQ_LAUNCH_CHECK();
        k_pad_cols_i8<<<grid_for((int64_t)kp * rsc), kThreads, 0, st>>>(w, 1, (int)(d->k * rsc),
                                                                         (int)(kp * rsc), wp);
        IQ_LAUNCH_CHECK();
        iq_status r = bn_stats_init(stats, d->c, st);
        if (r != IQ_OK) return r;
        bool done = false;
        r = conv_dgrad_tc(&dp, ep, wp, acc, nullptr, stats.s1, stats.hi, stats.lo, tws, st, &done,
                          nullptr);
        if (r != IQ_OK) return r;
        if (done) {
            k_max_from_stats<<<1, 1024, 0, st>>>(stats.hi, stats.lo, d->c, 0, s_in, cell,
                                                 rq_params_slot(rq), s_dx);
            IQ_LAUNCH_CHECK();
            return requant_apply(acc, IQ_I32, total, s_in, 8, IQ_MODE_SQ, 0, 0, 0, 0, dx, IQ_I8,
                                 s_dx, rq, st, true, false, dx16, dx_mask);
        }
    }
    // stride 2: the four parity phases of the input as stride-1 problems on the tensor cores
    if (!wide && d->stride_h == 2 && d->stride_w == 2) {
        iq_status r = bn_stats_init(stats, d->c, st);
        if (r != IQ_OK) return r;
        bool done = false;
        r = conv_dgrad_tc_stride2(d, e, w, acc, stats.s1, stats.hi, stats.lo, tcws, tcb, st,
                                  &done, (const __half*)e_f16);
        if (r != IQ_OK) return r;
        if (done) {
            k_max_from_stats<<<1, 1024, 0, st>>>(stats.hi, stats.lo, d->c, 0, s_in, cell,
                                                 rq_params_slot(rq), s_dx);
            IQ_LAUNCH_CHECK();
            return requant_apply(acc, IQ_I32, total, s_in, 8, IQ_MODE_SQ, 0, 0, 0, 0, dx, IQ_I8,
                                 s_dx, rq, st, true, false, dx16, dx_mask);
        }
    }
    int64_t wn = (int64_t)d->k * d->r * d->s * cp.Cg;
    k_transpose_w<<<grid_for(wn), kThreads, 0, st>>>(w, wt, d->k, d->r, d->s, cp.Cg, d->groups);
    IQ_LAUNCH_CHECK();
    IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, sizeof(unsigned long long), st));
    cp.M = (int64_t)d->n * d->h * d->w;
    cp.ncols = cp.Cg;
    cp.kin = (int)roundup(cp.Kg, BK);
    dim3 grid((unsigned)((cp.M + BM - 1) / BM), (unsigned)((cp.ncols + BN - 1) / BN), cp.G);
    if (wide) {
        kt_pre(st);
        k_conv_simt<OP_DGRAD, true><<<grid, 256, 0, st>>>(cp, e, wt, nullptr, (long long*)accw,
                                                          nullptr, nullptr, nullptr, cell);
        IQ_LAUNCH_CHECK();
        kt_post(st, IQ_KERNEL_CONV_SIMT);
        return requant_apply(accw, IQ_I64, total, s_in, 8, IQ_MODE_SQ, 0, 0, 0, 0, dx, IQ_I8,
                             s_dx, rq, st, false, false, dx16, dx_mask);
    }
    kt_pre(st);
    k_conv_simt<OP_DGRAD, false><<<grid, 256, 0, st>>>(cp, e, wt, acc, nullptr, nullptr, nullptr,
                                                       nullptr, cell);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_CONV_SIMT);
    return requant_apply(acc, IQ_I32, total, s_in, 8, IQ_MODE_SQ, 0, 0, 0, 0, dx, IQ_I8, s_dx, rq,
                         st, false, false, dx16, dx_mask);
}

static iq_status conv_wgrad_nhwc(const iq_conv_desc* d, const int8_t* e, const double* s_e,
                                 const int8_t* x, const double* s_x, int gq_mode, uint64_t seed,
                                 uint64_t layer, uint64_t step, int8_t* g, double* s_g,
                                 int64_t* g_acc_out, const void* e_f16, const void* x_f16,
                                 void* ws, size_t ws_bytes, iq_stream stream) {
    if ((((uintptr_t)e_f16 | (uintptr_t)x_f16) & 15)) return IQ_ERR_INVALID_ARG;
    if (!desc_ok(d) || !e || !s_e || !x || !s_x || !g || !s_g) return IQ_ERR_INVALID_ARG;
    if (gq_mode != 1 && gq_mode != 2) return IQ_ERR_INVALID_ARG;
    size_t need = 0;
    iq_conv_wgrad_workspace_size(d, &need);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    kt_set_op(3, conv_macs(d), conv_macs_dense(d));
    ConvP cp = make_params(d);
    // |G| < npq 127^2 must stay below 2^40 for the requantizer
    if ((double)cp.npq * 16129.0 >= 1099511627776.0) return IQ_ERR_OVERFLOW_RISK;
    cudaStream_t st = (cudaStream_t)stream;
    WsCursor cur(ws, ws_bytes);
    int64_t gn = (int64_t)d->k * d->r * d->s * cp.Cg;
    int64_t* gw = cur.take<int64_t>((size_t)gn);
    void* rq = cur.take<char>(requant_ws_bytes());
    double* s_in = cur.take<double>(1);
    void* tcws = cur.take<char>(conv_wgrad_tc_ws_bytes(d));
    int64_t* G = g_acc_out ? g_acc_out : gw;
    k_scale_mul<<<1, 1, 0, st>>>(s_e, s_x, s_in);
    IQ_LAUNCH_CHECK();
    {
        // the tensor-core path writes every element of G and, usually, its max |G| into the
        // requantizer's cell
        bool done = false, amax_done = false;
        unsigned long long* cell = (unsigned long long*)rq;
        IQ_CUDA_CHECK(cudaMemsetAsync(cell, 0, sizeof(unsigned long long), st));
        const int32_t* g32 = nullptr;
        iq_status r = conv_wgrad_tc(d, e, x, (long long*)G, tcws, st, &done, cell, &amax_done,
                                    (const __half*)e_f16, (const __half*)x_f16,
                                    g_acc_out ? nullptr : &g32);
        if (r != IQ_OK) return r;
        const int mode = gq_mode == 1 ? IQ_MODE_RQ_GQ1 : IQ_MODE_RQ_GQ2;
        if (done && g32)
            return requant_apply(g32, IQ_I32, gn, s_in, 8, mode, seed, layer, step, 0, g, IQ_I8,
                                 s_g, rq, st);
        if (done && amax_done)
            return requant_apply(G, IQ_I64, gn, s_in, 8, mode, seed, layer, step, 0, g, IQ_I8,
                                 s_g, rq, st);
        if (done)
            return requant_int(G, IQ_I64, gn, s_in, 8, mode, seed, layer, step, 0, g, IQ_I8,
                               s_g, rq, st);
    }
    IQ_CUDA_CHECK(cudaMemsetAsync(G, 0, sizeof(int64_t) * gn, st));
    cp.M = cp.Kg;
    cp.ncols = d->r * d->s * cp.Cg;
    int64_t tiles = ((cp.M + BM - 1) / BM) * ((cp.ncols + BN - 1) / BN) * cp.G;
    int64_t want_split = (152 * 8 + tiles - 1) / tiles;
    int64_t max_split = (cp.npq + 1023) / 1024;   // chunk >= 1024 reduction pixels
    if (want_split > max_split) want_split = max_split;
    if (want_split < 1) want_split = 1;
    cp.chunk = roundup((cp.npq + want_split - 1) / want_split, BK);
    if (cp.chunk > 65536) cp.chunk = 65536;      // int32 partial sums: 65536 * 127^2 < 2^31
    cp.nsplit = (int)((cp.npq + cp.chunk - 1) / cp.chunk);
    dim3 grid((unsigned)((cp.M + BM - 1) / BM), (unsigned)((cp.ncols + BN - 1) / BN),
              (unsigned)(cp.G * cp.nsplit));
    kt_pre(st);
    k_conv_simt<OP_WGRAD, false><<<grid, 256, 0, st>>>(cp, e, x, nullptr, (long long*)G, nullptr,
                                                       nullptr, nullptr, nullptr);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_CONV_SIMT);
    return requant_int(G, IQ_I64, gn, s_in, 8, gq_mode == 1 ? IQ_MODE_RQ_GQ1 : IQ_MODE_RQ_GQ2,
                       seed, layer, step, 0, g, IQ_I8, s_g, rq, st);
}

// ==================================================================== NCHW layout
// Sec. 3 states the problem without a memory layout; the kernels compute in NHWC (channels
// innermost, the TMA boxes' contiguous dimension).  With IQ_LAYOUT_NCHW the entry points
// transpose their activation / error inputs (NCHW -> NHWC) and filters (KCRS -> KRSC) into
// the workspace, run the NHWC computation, and transpose the outputs back.

namespace iq {
namespace {

// dst[b][c][r] = src[b][r][c] for b < gridDim.z: 32 x 32 tiles through shared memory
template <typename T>
__global__ void k_transpose_b(const T* __restrict__ src, T* __restrict__ dst, int64_t rows,
                              int64_t cols) {
    __shared__ T tile[32][33];
    const int64_t off = (int64_t)blockIdx.z * rows * cols;
    const int64_t r0 = (int64_t)blockIdx.y * 32, c0 = (int64_t)blockIdx.x * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int64_t r = r0 + i, c = c0 + threadIdx.x;
        if (r < rows && c < cols) tile[i][threadIdx.x] = src[off + r * cols + c];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int64_t c = c0 + i, r = r0 + threadIdx.x;
        if (r < rows && c < cols) dst[off + c * rows + r] = tile[threadIdx.x][i];
    }
}

iq_status transpose_b(const void* src, void* dst, int64_t batches, int64_t rows, int64_t cols,
                      int esize, cudaStream_t st) {
    if (batches < 1 || rows < 1 || cols < 1) return IQ_OK;
    const int64_t gx = (cols + 31) / 32, gy = (rows + 31) / 32;
    if (batches > 65535 || gy > 65535 || gx > 0x7fffffff) return IQ_ERR_UNSUPPORTED;
    const dim3 grid((unsigned)gx, (unsigned)gy, (unsigned)batches), blk(32, 8);
    switch (esize) {
        case 1: k_transpose_b<int8_t><<<grid, blk, 0, st>>>((const int8_t*)src, (int8_t*)dst, rows, cols); break;
        case 2: k_transpose_b<int16_t><<<grid, blk, 0, st>>>((const int16_t*)src, (int16_t*)dst, rows, cols); break;
        case 4: k_transpose_b<int32_t><<<grid, blk, 0, st>>>((const int32_t*)src, (int32_t*)dst, rows, cols); break;
        default: k_transpose_b<long long><<<grid, blk, 0, st>>>((const long long*)src, (long long*)dst, rows, cols); break;
    }
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

// NCHW image tensor [n][c][hw] <-> NHWC [n][hw][c]
iq_status to_nhwc(const void* src, void* dst, int64_t n, int64_t c, int64_t hw, int es,
                  cudaStream_t st) {
    return transpose_b(src, dst, n, c, hw, es, st);
}
iq_status to_nchw(const void* src, void* dst, int64_t n, int64_t c, int64_t hw, int es,
                  cudaStream_t st) {
    return transpose_b(src, dst, n, hw, c, es, st);
}

struct NchwWs {
    size_t off_x, off_w, off_y, off_y16, off_acc, off_rest;
};

size_t al256(size_t v) { return (v + 255) / 256 * 256; }

// the NCHW staging buffers of one call: input codes, filters, output codes (int8), int16
// codes, sums (int64 bytes per element), then the NHWC computation's own workspace
NchwWs nchw_layout(int64_t nin, int64_t nw, int64_t nout) {
    NchwWs L;
    L.off_x = 0;
    L.off_w = L.off_x + al256((size_t)nin);
    L.off_y = L.off_w + al256((size_t)nw);
    L.off_y16 = L.off_y + al256((size_t)nout);
    L.off_acc = L.off_y16 + al256((size_t)nout * 2);
    L.off_rest = L.off_acc + al256((size_t)nout * 8);
    return L;
}

void conv_sizes(const iq_conv_desc* d, int64_t* nin, int64_t* nw, int64_t* nout, int64_t* pq) {
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    *nin = (int64_t)d->n * d->h * d->w * d->c;
    *nw = (int64_t)d->k * d->r * d->s * (d->c / d->groups);
    *nout = (int64_t)d->n * P * Q * d->k;
    *pq = (int64_t)P * Q;
}

}  // namespace
}  // namespace iq

extern "C" iq_status iq_conv_fwd(const iq_conv_desc* d, const int8_t* x, const double* s_x,
                                 const int8_t* w, const int32_t* gamma, const int32_t* beta,
                                 const iq_bn_bits* bits, int use_bn, int relu, int8_t* a,
                                 double* s_a, int16_t* xhat, int32_t* bn_codes, double* bn_scales,
                                 int64_t* frozen_out, int32_t* acc_out, void* x_f16,
                                 void* a_f16, void* ws, size_t ws_bytes, iq_stream stream) {
    if (!desc_ok(d)) return IQ_ERR_INVALID_ARG;
    if (d->layout == IQ_LAYOUT_NHWC)
        return conv_fwd_nhwc(d, x, s_x, w, gamma, beta, bits, use_bn, relu, a, s_a, xhat,
                             bn_codes, bn_scales, frozen_out, acc_out, x_f16, a_f16, ws,
                             ws_bytes, stream);
    if (!x || !s_x || !w || !a || !s_a) return IQ_ERR_INVALID_ARG;
    int64_t nin, nw, nout, pq;
    conv_sizes(d, &nin, &nw, &nout, &pq);
    const NchwWs L = nchw_layout(nin, nw, nout);
    if (!ws || ws_bytes < L.off_rest + 256) return IQ_ERR_WORKSPACE;
    char* b = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    ws_bytes -= (size_t)(b - (char*)ws);
    iq_conv_desc dn = *d;
    dn.layout = IQ_LAYOUT_NHWC;
    cudaStream_t st = (cudaStream_t)stream;
    const int cg = d->c / d->groups;
    iq_status r = to_nhwc(x, b + L.off_x, d->n, d->c, (int64_t)d->h * d->w, 1, st);
    if (r == IQ_OK) r = transpose_b(w, b + L.off_w, d->k, cg, (int64_t)d->r * d->s, 1, st);
    if (r != IQ_OK) return r;
    int8_t* an = (int8_t*)(b + L.off_y);
    int16_t* xn = xhat ? (int16_t*)(b + L.off_y16) : nullptr;
    int32_t* accn = acc_out ? (int32_t*)(b + L.off_acc) : nullptr;
    r = conv_fwd_nhwc(&dn, (const int8_t*)(b + L.off_x), s_x, (const int8_t*)(b + L.off_w), gamma,
                      beta, bits, use_bn, relu, an, s_a, xn, bn_codes, bn_scales, frozen_out,
                      accn, x_f16, a_f16, b + L.off_rest, ws_bytes - L.off_rest, stream);
    if (r != IQ_OK) return r;
    r = to_nchw(an, a, d->n, d->k, pq, 1, st);
    if (r == IQ_OK && xhat) r = to_nchw(xn, xhat, d->n, d->k, pq, 2, st);
    if (r == IQ_OK && acc_out) r = to_nchw(accn, acc_out, d->n, d->k, pq, 4, st);
    return r;
}

extern "C" iq_status iq_conv_dgrad(const iq_conv_desc* d, const int8_t* e, const double* s_e,
                                   const int8_t* w, int8_t* dx, double* s_dx, int32_t* acc_out,
                                   void* e_f16, const int8_t* dx_mask, void* dx_f16, void* ws,
                                   size_t ws_bytes, iq_stream stream) {
    if (!desc_ok(d)) return IQ_ERR_INVALID_ARG;
    if (d->layout == IQ_LAYOUT_NHWC)
        return conv_dgrad_nhwc(d, e, s_e, w, dx, s_dx, acc_out, e_f16, dx_mask, dx_f16, ws,
                               ws_bytes, stream);
    if (dx_mask || dx_f16) return IQ_ERR_UNSUPPORTED;      // NHWC only
    if (!e || !s_e || !w || !dx || !s_dx) return IQ_ERR_INVALID_ARG;
    int64_t nin, nw, nout, pq;
    conv_sizes(d, &nin, &nw, &nout, &pq);
    // staging: errors (the "input" slot holds nout codes), filters, dx codes and sums
    const NchwWs L = nchw_layout(nout, nw, nin);
    if (!ws || ws_bytes < L.off_rest + 256) return IQ_ERR_WORKSPACE;
    char* b = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    ws_bytes -= (size_t)(b - (char*)ws);
    iq_conv_desc dn = *d;
    dn.layout = IQ_LAYOUT_NHWC;
    cudaStream_t st = (cudaStream_t)stream;
    const int cg = d->c / d->groups;
    iq_status r = to_nhwc(e, b + L.off_x, d->n, d->k, pq, 1, st);
    if (r == IQ_OK) r = transpose_b(w, b + L.off_w, d->k, cg, (int64_t)d->r * d->s, 1, st);
    if (r != IQ_OK) return r;
    int8_t* dxn = (int8_t*)(b + L.off_y);
    int32_t* accn = acc_out ? (int32_t*)(b + L.off_acc) : nullptr;
    r = conv_dgrad_nhwc(&dn, (const int8_t*)(b + L.off_x), s_e, (const int8_t*)(b + L.off_w), dxn,
                        s_dx, accn, e_f16, nullptr, nullptr, b + L.off_rest,
                        ws_bytes - L.off_rest, stream);
    if (r != IQ_OK) return r;
    const int64_t hw = (int64_t)d->h * d->w;
    r = to_nchw(dxn, dx, d->n, d->c, hw, 1, st);
    if (r == IQ_OK && acc_out) r = to_nchw(accn, acc_out, d->n, d->c, hw, 4, st);
    return r;
}

extern "C" iq_status iq_conv_wgrad(const iq_conv_desc* d, const int8_t* e, const double* s_e,
                                   const int8_t* x, const double* s_x, int gq_mode, uint64_t seed,
                                   uint64_t layer, uint64_t step, int8_t* g, double* s_g,
                                   int64_t* g_acc_out, const void* e_f16, const void* x_f16,
                                   void* ws, size_t ws_bytes, iq_stream stream) {
    if (!desc_ok(d)) return IQ_ERR_INVALID_ARG;
    if (d->layout == IQ_LAYOUT_NHWC)
        return conv_wgrad_nhwc(d, e, s_e, x, s_x, gq_mode, seed, layer, step, g, s_g, g_acc_out,
                               e_f16, x_f16, ws, ws_bytes, stream);
    if (!e || !s_e || !x || !s_x || !g || !s_g) return IQ_ERR_INVALID_ARG;
    int64_t nin, nw, nout, pq;
    conv_sizes(d, &nin, &nw, &nout, &pq);
    // staging: x in the input slot, e in the output-code slot (nout codes), gradient codes in
    // the filter slot, int64 sums in the sum slot (nw <= the slot's elements is checked)
    const int64_t nmax = nout > nw ? nout : nw;
    const NchwWs L = nchw_layout(nin, nw, nmax);
    if (!ws || ws_bytes < L.off_rest + 256) return IQ_ERR_WORKSPACE;
    char* b = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    ws_bytes -= (size_t)(b - (char*)ws);
    iq_conv_desc dn = *d;
    dn.layout = IQ_LAYOUT_NHWC;
    cudaStream_t st = (cudaStream_t)stream;
    const int cg = d->c / d->groups;
    iq_status r = to_nhwc(x, b + L.off_x, d->n, d->c, (int64_t)d->h * d->w, 1, st);
    if (r == IQ_OK) r = to_nhwc(e, b + L.off_y, d->n, d->k, pq, 1, st);
    if (r != IQ_OK) return r;
    int8_t* gn = (int8_t*)(b + L.off_w);
    int64_t* accn = g_acc_out ? (int64_t*)(b + L.off_acc) : nullptr;
    r = conv_wgrad_nhwc(&dn, (const int8_t*)(b + L.off_y), s_e, (const int8_t*)(b + L.off_x),
                        s_x, gq_mode, seed, layer, step, gn, s_g, accn, e_f16, x_f16,
                        b + L.off_rest, ws_bytes - L.off_rest, stream);
    if (r != IQ_OK) return r;
    // KRSC -> KCRS per output channel
    r = transpose_b(gn, g, d->k, (int64_t)d->r * d->s, cg, 1, st);
    if (r == IQ_OK && g_acc_out)
        r = transpose_b(accn, g_acc_out, d->k, (int64_t)d->r * d->s, cg, 8, st);
    return r;
}

static size_t nchw_stage_bytes(const iq_conv_desc* d, int op) {
    if (d->layout != IQ_LAYOUT_NCHW) return 0;
    int64_t nin, nw, nout, pq;
    iq::conv_sizes(d, &nin, &nw, &nout, &pq);
    if (op == 1) return iq::nchw_layout(nin, nw, nout).off_rest + 256;
    if (op == 2) return iq::nchw_layout(nout, nw, nin).off_rest + 256;
    return iq::nchw_layout(nin, nw, nout > nw ? nout : nw).off_rest + 256;
}

extern "C" iq_status iq_conv_fwd_frozen(const iq_conv_desc* d, const int8_t* x, const int8_t* w,
                                        const int64_t* frozen, const iq_bn_bits* bits,
                                        int use_bn, int relu, int8_t* a, int16_t* xhat,
                                        void* x_f16, void* ws, size_t ws_bytes,
                                        iq_stream stream) {
    if (!desc_ok(d)) return IQ_ERR_INVALID_ARG;
    if (d->layout == IQ_LAYOUT_NHWC)
        return conv_fwd_frozen_nhwc(d, x, w, frozen, bits, use_bn, relu, a, xhat, x_f16, ws,
                                    ws_bytes, stream);
    if (!x || !w || !a) return IQ_ERR_INVALID_ARG;
    int64_t nin, nw, nout, pq;
    iq::conv_sizes(d, &nin, &nw, &nout, &pq);
    const iq::NchwWs L = iq::nchw_layout(nin, nw, nout);
    if (!ws || ws_bytes < L.off_rest + 256) return IQ_ERR_WORKSPACE;
    char* b = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    ws_bytes -= (size_t)(b - (char*)ws);
    iq_conv_desc dn = *d;
    dn.layout = IQ_LAYOUT_NHWC;
    cudaStream_t st = (cudaStream_t)stream;
    iq_status r = iq::to_nhwc(x, b + L.off_x, d->n, d->c, (int64_t)d->h * d->w, 1, st);
    if (r == IQ_OK)
        r = iq::transpose_b(w, b + L.off_w, d->k, d->c / d->groups, (int64_t)d->r * d->s, 1, st);
    if (r != IQ_OK) return r;
    int8_t* an = (int8_t*)(b + L.off_y);
    int16_t* xn = xhat ? (int16_t*)(b + L.off_y16) : nullptr;
    r = conv_fwd_frozen_nhwc(&dn, (const int8_t*)(b + L.off_x), (const int8_t*)(b + L.off_w),
                             frozen, bits, use_bn, relu, an, xn, x_f16, b + L.off_rest,
                             ws_bytes - L.off_rest, stream);
    if (r != IQ_OK) return r;
    r = iq::to_nchw(an, a, d->n, d->k, pq, 1, st);
    if (r == IQ_OK && xhat) r = iq::to_nchw(xn, xhat, d->n, d->k, pq, 2, st);
    return r;
}
