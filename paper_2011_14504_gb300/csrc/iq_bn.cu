// iq_bn.cu -- quantized L1 batch normalization (Sec. 3.2.2) with ReLU and Q_A
// (Eq. (AQ1)), forward and backward (Sec. 3.3.1).
//
// Data: acc / errors are [m][C] row-major (NHWC flattened), C % 4 == 0.
// Every per-channel pass uses one launch shape: T threads in total with
// T % (C/4) == 0, so thread t always owns the same 4 channels (t % (C/4)) and
// keeps their partial sums in registers; blocks combine in shared memory and
// add into global integer accumulators (order-independent, hence deterministic).
// Loads are 16 bytes (4 int32 accumulators, or 4 int8 / int16 codes).
#include "iq_internal.cuh"
#include "iq_stream.cuh"

#include <climits>

namespace iq {

namespace {

struct ChanGrid {
    int blocks;
    int64_t threads;
};

int64_t gcd64(int64_t a, int64_t b) {
    while (b) { int64_t t = a % b; a = b; b = t; }
    return a;
}

ChanGrid chan_grid(int64_t m, int32_t C4, int max_blocks = 152 * 8) {
    int64_t unit = C4 / gcd64(kThreads, C4);  // blocks so that unit*256 % C4 == 0
    int64_t want = (m * C4 + kThreads - 1) / kThreads;
    if (want > max_blocks) want = max_blocks;
    if (want < 1) want = 1;
    want = (want + unit - 1) / unit * unit;
    ChanGrid g;
    g.blocks = (int)want;
    g.threads = want * kThreads;
    return g;
}

// Launch shape of the per-channel reduction passes (L1 deviation, backward sums): blocks of CG channel groups (4
// channels each) x RL row lanes (CG RL = 256), grid (channel-group tiles, row tiles).  A warp
// reads 4 CG consecutive channels of one row; the RL lanes of a channel group are combined
// in shared memory, so each block adds one partial per channel to the global accumulators.
struct RowGrid {
    int cg, rl;
    dim3 grid;
};

RowGrid row_grid(int64_t m, int32_t C4, int target_blocks = 152 * 8, int cg_max = 32) {
    RowGrid g;
    g.cg = cg_max;
    while (g.cg > 1 && g.cg > C4) g.cg >>= 1;
    g.rl = kThreads / g.cg;
    const int64_t bx = (C4 + g.cg - 1) / g.cg;
    int64_t by = (m + g.rl - 1) / g.rl;
    int64_t cap = target_blocks / bx;
    if (cap < 1) cap = 1;
    if (by > cap) by = cap;
    if (by > 65535) by = 65535;
    g.grid = dim3((unsigned)bx, (unsigned)by);
    return g;
}

__device__ __forceinline__ void unpack4_i8(int v, int out[4]) {
#pragma unroll
    for (int j = 0; j < 4; j++) out[j] = (int)(int8_t)(v >> (8 * j));
}

}  // namespace

// ------------------------------------------------------------------ workspace

size_t bn_fwd_ws_bytes(int32_t C) {
    WsCursor c(nullptr, 0);
    bn_stats_carve(c, C);
    return c.off + 256;
}

BnStats bn_stats_carve(WsCursor& cur, int32_t C) {
    BnStats s;
    s.s1 = cur.take<unsigned long long>(C);
    s.hi = cur.take<int>(C);
    s.lo = cur.take<int>(C);
    s.dev = cur.take<unsigned long long>(C);
    s.ngt = cur.take<unsigned long long>(C);
    s.F = cur.take<long long>(C);
    s.B = cur.take<long long>(C);
    s.G = cur.take<long long>(C);
    s.H = cur.take<long long>(C);
    s.codes = cur.take<int>(2 * (size_t)C);
    s.px = cur.take<int>(4);
    s.scal = cur.take<double>(IQ_BN_SCALES);
    s.red = cur.take<unsigned long long>(8);
    return s;
}

__global__ void k_bn_init(BnStats s, int32_t C) {
    for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < C; c += gridDim.x * blockDim.x) {
        s.s1[c] = 0; s.dev[c] = 0; s.ngt[c] = 0;
        s.hi[c] = INT_MIN; s.lo[c] = INT_MAX;
        if (c == 0)
            for (int i = 0; i < 8; i++) s.red[i] = 0ull;
    }
}

iq_status bn_stats_init(const BnStats& s, int32_t C, cudaStream_t st) {
    k_bn_init<<<(C + 255) / 256, 256, 0, st>>>(s, C);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

// ------------------------------------------------------------------ Eq. (BN2): sums, extremes

__global__ void __launch_bounds__(kThreads) k_bn_stats(const int32_t* __restrict__ acc,
                                                       int64_t m, int32_t C, BnStats s) {
    __shared__ unsigned long long sh_s1[1024];
    __shared__ int sh_hi[1024], sh_lo[1024];
    const int C4 = C >> 2;
    const bool use_sh = C <= 1024;
    if (use_sh)
        for (int c = threadIdx.x; c < C; c += blockDim.x) { sh_s1[c] = 0; sh_hi[c] = INT_MIN; sh_lo[c] = INT_MAX; }
    __syncthreads();
    const int64_t T = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int g = (int)(t % C4);
    const int64_t rstride = T / C4;
    long long s1[4] = {0, 0, 0, 0};
    int hi[4] = {INT_MIN, INT_MIN, INT_MIN, INT_MIN}, lo[4] = {INT_MAX, INT_MAX, INT_MAX, INT_MAX};
    const int4* a4 = reinterpret_cast<const int4*>(acc);
    for (int64_t r = t / C4; r < m; r += rstride) {
        int4 v = a4[r * C4 + g];
        int vs[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int j = 0; j < 4; j++) { s1[j] += vs[j]; hi[j] = max(hi[j], vs[j]); lo[j] = min(lo[j], vs[j]); }
    }
#pragma unroll
    for (int j = 0; j < 4; j++) {
        int c = 4 * g + j;
        if (use_sh) {
            atomicAdd(&sh_s1[c], (unsigned long long)s1[j]);
            atomicMax(&sh_hi[c], hi[j]);
            atomicMin(&sh_lo[c], lo[j]);
        } else {
            atomicAdd(&s.s1[c], (unsigned long long)s1[j]);
            atomicMax(&s.hi[c], hi[j]);
            atomicMin(&s.lo[c], lo[j]);
        }
    }
    if (use_sh) {
        __syncthreads();
        for (int c = threadIdx.x; c < C; c += blockDim.x) {
            atomicAdd(&s.s1[c], sh_s1[c]);
            atomicMax(&s.hi[c], sh_hi[c]);
            atomicMin(&s.lo[c], sh_lo[c]);
        }
    }
}

iq_status bn_stats_pass(const int32_t* acc, int64_t m, int32_t C, const BnStats& s,
                        cudaStream_t st) {
    ChanGrid g = chan_grid(m, C / 4);
    k_bn_stats<<<g.blocks, kThreads, 0, st>>>(acc, m, C, s);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

// ------------------------------------------------------------------ Eq. (BN5): deviation sums
// sum_i |m acc_i - S1| = m * sum_i |acc_i - f| + rho * (m - 2 #(acc_i > f)),
// f = floor(S1/m), rho = S1 - f m; this pass sums |acc - f| and counts acc > f.

__device__ __forceinline__ int64_t floordiv_i64(int64_t a, int64_t b) {
    int64_t q = a / b;
    if ((a % b) != 0 && a < 0) q -= 1;
    return q;
}

__global__ void __launch_bounds__(kThreads) k_bn_dev(const int32_t* __restrict__ acc, int64_t m,
                                                     int32_t C, int CG, BnStats s) {
    __shared__ unsigned long long sh_d[kThreads * 4], sh_n[kThreads * 4];
    __shared__ int sh_h[kThreads * 4], sh_l[kThreads * 4];
    const int C4 = C >> 2;
    const int cg = threadIdx.x % CG, rl = threadIdx.x / CG, RL = blockDim.x / CG;
    const int g = blockIdx.x * CG + cg;
    const bool act = g < C4;
    int64_t f[4] = {0, 0, 0, 0};
    if (act) {
#pragma unroll
        for (int j = 0; j < 4; j++) f[j] = floordiv_i64((int64_t)s.s1[4 * g + j], m);
    }
    unsigned long long d[4] = {0, 0, 0, 0}, n[4] = {0, 0, 0, 0};
    // the per-channel extremes too (the conv epilogue may leave them to this pass)
    int hi[4] = {INT_MIN, INT_MIN, INT_MIN, INT_MIN}, lo[4] = {INT_MAX, INT_MAX, INT_MAX, INT_MAX};
    const int4* a4 = reinterpret_cast<const int4*>(acc);
    const int64_t step = (int64_t)gridDim.y * RL;
    auto row = [&](const int4 v) {
        const int vs[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const int64_t dv = (int64_t)vs[j] - f[j];
            d[j] += (unsigned long long)(dv < 0 ? -dv : dv);
            n[j] += dv > 0;
            hi[j] = max(hi[j], vs[j]);
            lo[j] = min(lo[j], vs[j]);
        }
    };
    if (act) {
        int64_t r = (int64_t)blockIdx.y * RL + rl;
        // four rows per iteration: their loads in flight together
        for (; r + 3 * step < m; r += 4 * step) {
            int4 v[4];
#pragma unroll
            for (int u = 0; u < 4; u++) v[u] = a4[(r + u * step) * C4 + g];
#pragma unroll
            for (int u = 0; u < 4; u++) row(v[u]);
        }
        for (; r < m; r += step) row(a4[r * C4 + g]);
    }
#pragma unroll
    for (int j = 0; j < 4; j++) {
        sh_d[rl * CG * 4 + 4 * cg + j] = d[j];
        sh_n[rl * CG * 4 + 4 * cg + j] = n[j];
        sh_h[rl * CG * 4 + 4 * cg + j] = hi[j];
        sh_l[rl * CG * 4 + 4 * cg + j] = lo[j];
    }
    __syncthreads();
    const int col = threadIdx.x;
    if (col < CG * 4) {
        const int c = 4 * blockIdx.x * CG + col;
        if (c < C) {
            unsigned long long td = 0, tn = 0;
            int th = INT_MIN, tl = INT_MAX;
            for (int i = 0; i < RL; i++) {
                td += sh_d[i * CG * 4 + col];
                tn += sh_n[i * CG * 4 + col];
                th = max(th, sh_h[i * CG * 4 + col]);
                tl = min(tl, sh_l[i * CG * 4 + col]);
            }
            atomicAdd(&s.dev[c], td);
            atomicAdd(&s.ngt[c], tn);
            if (th >= tl) {
                atomicMax(&s.hi[c], th);
                atomicMin(&s.lo[c], tl);
            }
        }
    }
}

// ------------------------------------------------------------------ finalize (one block)

__device__ __forceinline__ int frexp_exp(double v) {
    int e;
    frexp(v, &e);
    return e;
}

// The fp64 steps below follow the oracle's operation order one for one:
// mu_B = (S1 s_acc)/m, sigma_B = (T s_acc)/(m m), codes by rhu of v 2^(k-2),
// xhat(v) = (v s_acc - mu_q)/den, a_c = (s_acc/den) qx, b_c = (-mu_q/den) qx, ...
// The per-channel work is spread over C/64 blocks of 64 threads (the fp64 pipe of one SM
// is narrow); each tensor-wide maximum of non-negative doubles is an atomicMax on its bit
// pattern, and every stage that needs one is a separate launch.
constexpr int kFinThreads = 64;

__device__ __forceinline__ void red_max(unsigned long long* cell, double v) {
    if (v > 0.0) atomicMax(cell, (unsigned long long)__double_as_longlong(v));
}
__device__ __forceinline__ double red_get(const unsigned long long* cell) {
    return __longlong_as_double((long long)*cell);
}

// stage 1: mu_q / sigma_q codes; max |xhat| at the channel extremes (red[0]); max |acc| (red[1])
__global__ void __launch_bounds__(kFinThreads) k_bn_fin1(BnStats s, int64_t m, int32_t C,
                                                         const double* __restrict__ s_acc_p,
                                                         iq_bn_bits b) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    const double s_acc = *s_acc_p;
    const double md = (double)m;
    const double mu_step = ldexp(1.0, 2 - b.k_mu), sg_step = ldexp(1.0, 2 - b.k_sigma);
    int64_t S1 = (int64_t)s.s1[c];
    int64_t f = floordiv_i64(S1, m);
    int64_t rho = S1 - f * m;
    i128 T = (i128)m * (i128)(int64_t)s.dev[c] + (i128)rho * (i128)(m - 2 * (int64_t)s.ngt[c]);
    double mu_b = __ddiv_rn(__dmul_rn((double)S1, s_acc), md);
    double sg_b = __ddiv_rn(__dmul_rn(u128_to_double((u128)T), s_acc), __dmul_rn(md, md));
    int64_t cm = code_of(ldexp(mu_b, b.k_mu - 2), b.k_mu);
    int64_t cs = code_of(ldexp(sg_b, b.k_sigma - 2), b.k_sigma);
    s.codes[c] = (int32_t)cm;
    s.codes[C + c] = (int32_t)cs;
    double muq = __dmul_rn((double)cm, mu_step);
    double den = __dmul_rn((double)(cs + 1), sg_step);
    double xh = __ddiv_rn(__dsub_rn(__dmul_rn((double)s.hi[c], s_acc), muq), den);
    double xl = __ddiv_rn(__dsub_rn(__dmul_rn((double)s.lo[c], s_acc), muq), den);
    red_max(&s.red[0], fmax(fabs(xh), fabs(xl)));
    red_max(&s.red[1], fmax(fabs((double)s.hi[c]), fabs((double)s.lo[c])));
}

__device__ __forceinline__ void bn_xmap(const BnStats& s, int c, int32_t C, double s_acc,
                                        double qx, const iq_bn_bits& b, double* a, double* bb) {
    const double mu_step = ldexp(1.0, 2 - b.k_mu), sg_step = ldexp(1.0, 2 - b.k_sigma);
    double muq = __dmul_rn((double)s.codes[c], mu_step);
    double den = __dmul_rn((double)(s.codes[C + c] + 1), sg_step);
    *a = __dmul_rn(__ddiv_rn(s_acc, den), qx);
    *bb = __dmul_rn(__ddiv_rn(-muq, den), qx);
}

// stage 2: the bound of the acc -> X map (red[2])
__global__ void __launch_bounds__(kFinThreads) k_bn_fin2(BnStats s, int32_t C,
                                                         const double* __restrict__ s_acc_p,
                                                         iq_bn_bits b) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    const double mx = red_get(&s.red[0]);
    if (c >= C || !(mx > 0.0)) return;
    const double qx = __ddiv_rn(ldexp(1.0, b.k_xhat - 1), mx);
    double a, bb;
    bn_xmap(s, c, C, *s_acc_p, qx, b, &a, &bb);
    red_max(&s.red[2], __dadd_rn(__dmul_rn(fabs(a), red_get(&s.red[1])), fabs(bb)));
}

__device__ __forceinline__ int shift_of(double lmax) {
    int p = 62 - frexp_exp(__dadd_rn(lmax, 1.0));
    return p > 62 ? 62 : (p < 1 ? 1 : p);
}

// stage 3: F, B with the shift P_x; max ReLU(y) at the channel extremes (red[3])
__global__ void __launch_bounds__(kFinThreads) k_bn_fin3(BnStats s, int32_t C,
                                                         const double* __restrict__ s_acc_p,
                                                         const int32_t* __restrict__ gam,
                                                         const int32_t* __restrict__ bet,
                                                         iq_bn_bits b) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    const double mx = red_get(&s.red[0]);
    const double s_xhat = mx > 0.0 ? ldexp(mx, 1 - b.k_xhat) : ldexp(1.0, 1 - b.k_xhat);
    const int64_t xq = qmax(b.k_xhat);
    int px = 1;
    if (mx > 0.0) {
        const double qx = __ddiv_rn(ldexp(1.0, b.k_xhat - 1), mx);
        px = shift_of(red_get(&s.red[2]));
        double a, bb;
        bn_xmap(s, c, C, *s_acc_p, qx, b, &a, &bb);
        s.F[c] = (long long)rhu(ldexp(a, px));
        s.B[c] = (long long)rhu(ldexp(bb, px)) + (1LL << (px - 1));
    } else {
        s.F[c] = 0;
        s.B[c] = 0;
    }
    const double gstep = ldexp(1.0, 2 - b.k_gamma), bstep = ldexp(1.0, 2 - b.k_beta);
    const int64_t xs[2] = {s.hi[c], s.lo[c]};
    const double t1 = __dmul_rn(__dmul_rn((double)gam[c], gstep), s_xhat);
    double my = 0.0;
    for (int j = 0; j < 2; j++) {
        long long t = (long long)s.F[c] * xs[j] + s.B[c];
        int64_t xc = clamp64(t >> px, -xq, xq);
        double y = __dadd_rn(__dmul_rn(t1, (double)xc), __dmul_rn((double)bet[c], bstep));
        my = fmax(my, y);
    }
    red_max(&s.red[3], my);
}

// stage 4: the bound of the X -> A map (red[4])
__global__ void __launch_bounds__(kFinThreads) k_bn_fin4(BnStats s, int32_t C,
                                                         const int32_t* __restrict__ gam,
                                                         const int32_t* __restrict__ bet,
                                                         iq_bn_bits b) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    const double my = red_get(&s.red[3]);
    if (c >= C || !(my > 0.0)) return;
    const double mx = red_get(&s.red[0]);
    const double s_xhat = mx > 0.0 ? ldexp(mx, 1 - b.k_xhat) : ldexp(1.0, 1 - b.k_xhat);
    const double gstep = ldexp(1.0, 2 - b.k_gamma), bstep = ldexp(1.0, 2 - b.k_beta);
    const double qa = __ddiv_rn(ldexp(1.0, b.k_a - 1), my);
    double t1 = __dmul_rn(__dmul_rn((double)gam[c], gstep), s_xhat);
    double bq = __dmul_rn((double)bet[c], bstep);
    red_max(&s.red[4], __dadd_rn(__dmul_rn(fabs(__dmul_rn(t1, qa)), (double)qmax(b.k_xhat)),
                                 fabs(__dmul_rn(bq, qa))));
}

// stage 5: G, H with the shift P_a; the shifts and scales of the layer
__global__ void __launch_bounds__(kFinThreads) k_bn_fin5(BnStats s, int32_t C,
                                                         const double* __restrict__ s_acc_p,
                                                         const int32_t* __restrict__ gam,
                                                         const int32_t* __restrict__ bet,
                                                         iq_bn_bits b) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    const double mx = red_get(&s.red[0]), my = red_get(&s.red[3]);
    const double s_xhat = mx > 0.0 ? ldexp(mx, 1 - b.k_xhat) : ldexp(1.0, 1 - b.k_xhat);
    const double s_a = my > 0.0 ? ldexp(my, 1 - b.k_a) : ldexp(1.0, 1 - b.k_a);
    int pa = 1;
    if (my > 0.0) pa = shift_of(red_get(&s.red[4]));
    if (c < C) {
        if (my > 0.0) {
            const double gstep = ldexp(1.0, 2 - b.k_gamma), bstep = ldexp(1.0, 2 - b.k_beta);
            const double qa = __ddiv_rn(ldexp(1.0, b.k_a - 1), my);
            double t1 = __dmul_rn(__dmul_rn((double)gam[c], gstep), s_xhat);
            double bq = __dmul_rn((double)bet[c], bstep);
            s.G[c] = (long long)rhu(ldexp(__dmul_rn(t1, qa), pa));
            s.H[c] = (long long)rhu(ldexp(__dmul_rn(bq, qa), pa)) + (1LL << (pa - 1));
        } else {
            s.G[c] = 0;
            s.H[c] = 0;
        }
    }
    if (c == 0) {
        s.px[0] = mx > 0.0 ? shift_of(red_get(&s.red[2])) : 1;
        s.px[1] = pa;
        s.scal[IQ_BN_S_XHAT] = s_xhat;
        s.scal[IQ_BN_M_XHAT] = mx;
        s.scal[IQ_BN_M_Y] = my;
        s.scal[IQ_BN_S_ACC] = *s_acc_p;
        s.scal[IQ_BN_S_A] = s_a;
        for (int i = IQ_BN_S_A + 1; i < IQ_BN_SCALES; i++) s.scal[i] = 0.0;
    }
}

// ------------------------------------------------------------------ fused requant pass
// X = clip(floor((F acc + B) / 2^Px)), A = clip(floor((G X + H) / 2^Pa), 0, 2^(k_a-1)-1)

__global__ void __launch_bounds__(kThreads) k_bn_requant(const int32_t* __restrict__ acc,
                                                         int64_t m, int32_t C, BnStats s,
                                                         int kx, int ka,
                                                         int16_t* __restrict__ X,
                                                         int8_t* __restrict__ A,
                                                         uint2* __restrict__ A16) {
    const int C4 = C >> 2;
    const int64_t T = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int g = (int)(t % C4);
    const int64_t rstride = T / C4;
    const int px = s.px[0], pa = s.px[1];
    const int64_t xq = qmax(kx), aq = qmax(ka);
    long long F[4], B[4], G[4], H[4];
#pragma unroll
    for (int j = 0; j < 4; j++) {
        F[j] = s.F[4 * g + j]; B[j] = s.B[4 * g + j];
        G[j] = s.G[4 * g + j]; H[j] = s.H[4 * g + j];
    }
    const int4* a4 = reinterpret_cast<const int4*>(acc);
    auto row = [&](int64_t v, const int4 in) {
        const int vs[4] = {in.x, in.y, in.z, in.w};
        int xo[4];
        uint32_t ao = 0;
#pragma unroll
        for (int j = 0; j < 4; j++) {
            long long tx = F[j] * (long long)vs[j] + B[j];
            int64_t xc = clamp64(tx >> px, -xq, xq);
            xo[j] = (int)xc;
            long long ta = G[j] * xc + H[j];
            int64_t ac = clamp64(ta >> pa, 0, aq);
            ao |= ((uint32_t)ac & 0xffu) << (8 * j);
        }
        if (X) {
            uint2 xv;
            xv.x = ((uint32_t)(uint16_t)xo[0]) | ((uint32_t)(uint16_t)xo[1] << 16);
            xv.y = ((uint32_t)(uint16_t)xo[2]) | ((uint32_t)(uint16_t)xo[3] << 16);
            reinterpret_cast<uint2*>(X)[v] = xv;
        }
        reinterpret_cast<uint32_t*>(A)[v] = ao;
        if (A16) {                    // the fp16 copy of the 4 A codes
            uint2 hv;
            tc::i8x4_to_f16x4(ao, hv.x, hv.y);
            A16[v] = hv;
        }
    };
    int64_t r = t / C4;
    // two rows per iteration: both loads in flight together
    for (; r + rstride < m; r += 2 * rstride) {
        const int64_t v0 = r * C4 + g, v1 = (r + rstride) * C4 + g;
        const int4 in0 = a4[v0], in1 = a4[v1];
        row(v0, in0);
        row(v1, in1);
    }
    if (r < m) row(r * C4 + g, a4[r * C4 + g]);
}

// ------------------------------------------------------------------ streamed forward passes
// The deviation and requantization passes over row chunks staged in shared memory by bulk
// copies (iq_stream.cuh); the arithmetic is that of k_bn_dev / k_bn_requant.

// |v - f| for int32 v and f: below 2^32, exact in 32-bit unsigned arithmetic
__device__ __forceinline__ uint32_t absdiff_u32(int v, int f) {
    return v >= f ? (uint32_t)v - (uint32_t)f : (uint32_t)f - (uint32_t)v;
}

__global__ void __launch_bounds__(kStreamThreads, 1) k_bn_dev_s(RowStream rs, BnStats s,
                                                                  int* __restrict__ err) {
    extern __shared__ __align__(128) uint8_t smem[];
    if (__syncthreads_or(threadIdx.x == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    const int CB4 = rs.CB >> 2;
    const int g = threadIdx.x % CB4, rl = threadIdx.x / CB4;
    const int c0 = blockIdx.x * rs.CB + 4 * g;
    int f[4];                        // floor(S1 / m): a mean of int32 values, so int32
#pragma unroll
    for (int j = 0; j < 4; j++) f[j] = (int)floordiv_i64((int64_t)s.s1[c0 + j], rs.m);
    unsigned long long d[4] = {0, 0, 0, 0}, n[4] = {0, 0, 0, 0};
    int hi[4] = {INT_MIN, INT_MIN, INT_MIN, INT_MIN}, lo[4] = {INT_MAX, INT_MAX, INT_MAX, INT_MAX};
    const bool ok = stream_chunks(rs, smem, err, [&](const uint8_t* st, int rows, int64_t) {
        const int4* v4 = reinterpret_cast<const int4*>(st);
#pragma unroll
        for (int u = 0; u < kStreamRPT; u++) {
            const int r = rl + u * rs.RL;
            if (r >= rows) break;
            const int4 v = v4[r * CB4 + g];
            const int vs[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int j = 0; j < 4; j++) {
                d[j] += absdiff_u32(vs[j], f[j]);
                n[j] += vs[j] > f[j];
                hi[j] = max(hi[j], vs[j]);
                lo[j] = min(lo[j], vs[j]);
            }
        }
    });
    if (!ok) return;
    // the row lanes of each channel, through shared memory (the stages are free now)
    unsigned long long* sd = reinterpret_cast<unsigned long long*>(smem);    // [RL][CB]
    unsigned long long* sn = sd + kStreamThreads * 4;
    int* sh = reinterpret_cast<int*>(sn + kStreamThreads * 4);
    int* sl = sh + kStreamThreads * 4;
#pragma unroll
    for (int j = 0; j < 4; j++) {
        const int i = rl * rs.CB + 4 * g + j;
        sd[i] = d[j]; sn[i] = n[j]; sh[i] = hi[j]; sl[i] = lo[j];
    }
    __syncthreads();
    for (int col = threadIdx.x; col < rs.CB; col += blockDim.x) {
        unsigned long long td = 0, tn = 0;
        int th = INT_MIN, tl = INT_MAX;
        for (int i = 0; i < rs.RL; i++) {
            const int k = i * rs.CB + col;
            td += sd[k]; tn += sn[k]; th = max(th, sh[k]); tl = min(tl, sl[k]);
        }
        const int c = blockIdx.x * rs.CB + col;
        atomicAdd(&s.dev[c], td);
        atomicAdd(&s.ngt[c], tn);
        if (th >= tl) {
            atomicMax(&s.hi[c], th);
            atomicMin(&s.lo[c], tl);
        }
    }
}

__global__ void __launch_bounds__(kStreamThreads, 1) k_bn_requant_s(RowStream rs, BnStats s,
                                                                      int kx, int ka,
                                                                      int16_t* __restrict__ X,
                                                                      int8_t* __restrict__ A,
                                                                      uint2* __restrict__ A16,
                                                                      int* __restrict__ err) {
    extern __shared__ __align__(128) uint8_t smem[];
    if (__syncthreads_or(threadIdx.x == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    const int CB4 = rs.CB >> 2;
    const int g = threadIdx.x % CB4, rl = threadIdx.x / CB4;
    const int c0 = blockIdx.x * rs.CB + 4 * g;
    const int px = s.px[0], pa = s.px[1];
    const int64_t xq = qmax(kx), aq = qmax(ka);
    long long F[4], B[4], G[4], H[4];
#pragma unroll
    for (int j = 0; j < 4; j++) {
        F[j] = s.F[c0 + j]; B[j] = s.B[c0 + j];
        G[j] = s.G[c0 + j]; H[j] = s.H[c0 + j];
    }
    stream_chunks(rs, smem, err, [&](const uint8_t* st, int rows, int64_t r0) {
        const int4* v4 = reinterpret_cast<const int4*>(st);
#pragma unroll
        for (int u = 0; u < kStreamRPT; u++) {
            const int r = rl + u * rs.RL;
            if (r >= rows) break;
            const int4 v = v4[r * CB4 + g];
            const int vs[4] = {v.x, v.y, v.z, v.w};
            int xo[4];
            uint32_t ao = 0;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const long long tx = F[j] * (long long)vs[j] + B[j];
                const int64_t xc = clamp64(tx >> px, -xq, xq);
                xo[j] = (int)xc;
                const long long ta = G[j] * xc + H[j];
                const int64_t ac = clamp64(ta >> pa, 0, aq);
                ao |= ((uint32_t)ac & 0xffu) << (8 * j);
            }
            const int64_t e = (r0 + r) * rs.C + c0;      // element index of channel c0
            if (X) {
                uint2 xv;
                xv.x = ((uint32_t)(uint16_t)xo[0]) | ((uint32_t)(uint16_t)xo[1] << 16);
                xv.y = ((uint32_t)(uint16_t)xo[2]) | ((uint32_t)(uint16_t)xo[3] << 16);
                *reinterpret_cast<uint2*>(X + e) = xv;
            }
            *reinterpret_cast<uint32_t*>(A + e) = ao;
            if (A16) {                // the fp16 copy of the 4 A codes
                uint2 hv;
                tc::i8x4_to_f16x4(ao, hv.x, hv.y);
                A16[e >> 2] = hv;
            }
        }
    });
}

// the streamed kernels' dynamic shared memory, set once per kernel
template <class K>
iq_status stream_attr(K kernel, bool& done) {
    if (!done) {
        IQ_CUDA_CHECK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)(kStreamStages * kStreamElems * 4 +
                                                 2 * kStreamStages * sizeof(uint64_t))));
        done = true;
    }
    return IQ_OK;
}

// ------------------------------------------------------------------ frozen statistics
// The element maps of the forward pass with constants fixed by an earlier call (fixed =
// F[C], B[C], G[C], H[C], P_x, P_a): X = clip(floor((F acc + B) / 2^P_x)) with the product in
// 128 bits (an accumulator beyond the calibration range cannot overflow it), A = clip(floor((G
// X + H) / 2^P_a), 0, aq) (|X| <= 2^15 keeps the second map within int64 by the choice of P_a).

// floor((F v + B) / 2^px) clipped to [-q, q], t = F v + B exact in 128 bits, 1 <= px <= 62
__device__ __forceinline__ int64_t map128_clip(long long F, int v, long long B, int px,
                                               int64_t q) {
    const long long lo = F * (long long)v;                       // low 64 bits
    long long hi = __mul64hi(F, (long long)v);                   // signed high 64 bits
    const unsigned long long l2 = (unsigned long long)lo + (unsigned long long)B;
    hi += (long long)(l2 < (unsigned long long)lo) + (B < 0 ? -1LL : 0LL);
    const unsigned long long rl = (l2 >> px) | ((unsigned long long)hi << (64 - px));
    const long long rh = hi >> px;                               // the shifted value rh:rl
    if (rh > 0) return q;
    if (rh == 0) return rl > (unsigned long long)q ? q : (int64_t)rl;
    if (rh < -1) return -q;
    const long long vv = (long long)rl;                          // rh == -1
    return (vv >= 0 || vv < -q) ? -q : vv;
}

__global__ void __launch_bounds__(kThreads) k_bn_apply_fixed(const int32_t* __restrict__ acc,
                                                             int64_t m, int32_t C,
                                                             const int64_t* __restrict__ fx,
                                                             int kx, int ka,
                                                             int16_t* __restrict__ X,
                                                             int8_t* __restrict__ A) {
    const int C4 = C >> 2;
    const int64_t T = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int g = (int)(t % C4);
    const int64_t rstride = T / C4;
    const int px = (int)fx[4 * (int64_t)C], pa = (int)fx[4 * (int64_t)C + 1];
    const int64_t xq = qmax(kx), aq = qmax(ka);
    long long F[4], B[4], G[4], H[4];
#pragma unroll
    for (int j = 0; j < 4; j++) {
        F[j] = fx[4 * g + j]; B[j] = fx[C + 4 * g + j];
        G[j] = fx[2 * C + 4 * g + j]; H[j] = fx[3 * C + 4 * g + j];
    }
    const int4* a4 = reinterpret_cast<const int4*>(acc);
    auto row = [&](int64_t v, const int4 in) {
        const int vs[4] = {in.x, in.y, in.z, in.w};
        int xo[4];
        uint32_t ao = 0;
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const int64_t xc = map128_clip(F[j], vs[j], B[j], px, xq);
            xo[j] = (int)xc;
            const long long ta = G[j] * xc + H[j];
            const int64_t ac = clamp64(ta >> pa, 0, aq);
            ao |= ((uint32_t)ac & 0xffu) << (8 * j);
        }
        if (X) {
            uint2 xv;
            xv.x = ((uint32_t)(uint16_t)xo[0]) | ((uint32_t)(uint16_t)xo[1] << 16);
            xv.y = ((uint32_t)(uint16_t)xo[2]) | ((uint32_t)(uint16_t)xo[3] << 16);
            reinterpret_cast<uint2*>(X)[v] = xv;
        }
        reinterpret_cast<uint32_t*>(A)[v] = ao;
    };
    int64_t r = t / C4;
    for (; r + rstride < m; r += 2 * rstride) {
        const int64_t v0 = r * C4 + g, v1 = (r + rstride) * C4 + g;
        const int4 in0 = a4[v0], in1 = a4[v1];
        row(v0, in0);
        row(v1, in1);
    }
    if (r < m) row(r * C4 + g, a4[r * C4 + g]);
}

iq_status bn_apply_fixed(const int32_t* acc, int64_t m, int32_t C, const int64_t* fixed, int kx,
                         int ka, int16_t* X, int8_t* A, cudaStream_t st) {
    if (m == 0) return IQ_OK;
    ChanGrid g2 = chan_grid(m, C / 4, 152 * 16);
    kt_pre(st);
    k_bn_apply_fixed<<<g2.blocks, kThreads, 0, st>>>(acc, m, C, fixed, kx, ka, X, A);
    IQ_LAUNCH_CHECK();
    kt_post_bytes(st, IQ_KERNEL_BN_REQUANT, (double)m * C * (X ? 7.0 : 5.0));
    return IQ_OK;
}

__global__ void k_bn_export(BnStats s, int32_t C, const int32_t* __restrict__ codes_ws,
                            double* __restrict__ s_a, int32_t* __restrict__ bn_codes,
                            double* __restrict__ bn_scales, int64_t* __restrict__ bn_fixed) {
    int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t == 0) {
        if (s_a) *s_a = s.scal[IQ_BN_S_A];
        if (bn_scales)
            for (int i = 0; i < IQ_BN_SCALES; i++) bn_scales[i] = s.scal[i];
        if (bn_fixed) { bn_fixed[4 * C] = s.px[0]; bn_fixed[4 * C + 1] = s.px[1]; }
    }
    for (int c = t; c < C; c += gridDim.x * blockDim.x) {
        if (bn_codes) { bn_codes[c] = codes_ws[c]; bn_codes[C + c] = codes_ws[C + c]; }
        if (bn_fixed) {
            bn_fixed[c] = s.F[c]; bn_fixed[C + c] = s.B[c];
            bn_fixed[2 * C + c] = s.G[c]; bn_fixed[3 * C + c] = s.H[c];
        }
    }
}

iq_status bn_fwd_after_stats(const int32_t* acc, int64_t m, int32_t C, const double* s_acc,
                             const int32_t* gamma, const int32_t* beta, const iq_bn_bits& b,
                             const BnStats& s, int16_t* xhat, int8_t* a, double* s_a,
                             int32_t* bn_codes, double* bn_scales, int64_t* bn_fixed,
                             cudaStream_t st, __half* a16) {
    if (a16 && !f16_copy_ok(a, a16, m * C)) return IQ_ERR_INVALID_ARG;
    RowStream rs;
    const void* srcs[1] = {acc};
    const int esz[1] = {4};
    const bool streamed = row_stream_plan(rs, m, C, srcs, esz, 1);
    int* err = device_status_ptr();
    if (!err) return IQ_ERR_CUDA;
    kt_pre(st);
    if (streamed) {
        static bool attr = false;
        iq_status r = stream_attr(k_bn_dev_s, attr);
        if (r != IQ_OK) return r;
        k_bn_dev_s<<<row_stream_grid(rs, device_sms()), kStreamThreads, row_stream_smem(rs), st>>>(
            rs, s, err);
    } else {
        RowGrid rg = row_grid(m, C / 4);
        k_bn_dev<<<rg.grid, kThreads, 0, st>>>(acc, m, C, rg.cg, s);
    }
    IQ_LAUNCH_CHECK();
    kt_post_bytes(st, IQ_KERNEL_BN_DEV, 4.0 * (double)m * C);
    const int fb = (C + kFinThreads - 1) / kFinThreads;
    k_bn_fin1<<<fb, kFinThreads, 0, st>>>(s, m, C, s_acc, b);
    IQ_LAUNCH_CHECK();
    k_bn_fin2<<<fb, kFinThreads, 0, st>>>(s, C, s_acc, b);
    IQ_LAUNCH_CHECK();
    k_bn_fin3<<<fb, kFinThreads, 0, st>>>(s, C, s_acc, gamma, beta, b);
    IQ_LAUNCH_CHECK();
    k_bn_fin4<<<fb, kFinThreads, 0, st>>>(s, C, gamma, beta, b);
    IQ_LAUNCH_CHECK();
    k_bn_fin5<<<fb, kFinThreads, 0, st>>>(s, C, s_acc, gamma, beta, b);
    IQ_LAUNCH_CHECK();
    kt_pre(st);
    if (streamed) {
        static bool attr = false;
        iq_status r = stream_attr(k_bn_requant_s, attr);
        if (r != IQ_OK) return r;
        k_bn_requant_s<<<row_stream_grid(rs, device_sms()), kStreamThreads, row_stream_smem(rs),
                         st>>>(rs, s, b.k_xhat, b.k_a, xhat, a, (uint2*)a16, err);
    } else {
        ChanGrid g2 = chan_grid(m, C / 4, 152 * 16);
        k_bn_requant<<<g2.blocks, kThreads, 0, st>>>(acc, m, C, s, b.k_xhat, b.k_a, xhat, a,
                                                     (uint2*)a16);
    }
    IQ_LAUNCH_CHECK();
    kt_post_bytes(st, IQ_KERNEL_BN_REQUANT,
                  (double)m * C * ((xhat ? 7.0 : 5.0) + (a16 ? 2.0 : 0.0)));
    k_bn_export<<<(C + 255) / 256, 256, 0, st>>>(s, C, s.codes, s_a, bn_codes, bn_scales,
                                                 bn_fixed);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

// ==================================================================== backward
// hist  : e_y = e_a [a > 0]; per channel the histogram of the nonzero e_y codes (count and
//         sum of X per code), sum sign X, the extreme e_y of each sign class of X, and
//         max |e_y gamma|
// fin 1 : E_2 = SQ_{k_e2}(e_y gamma) constants
// hfin  : per channel sum e_y, sum e_y X, sum E_2, sum E_2 X and the E_2 extremes per sign
//         class, all exactly from the histogram (below)
// fin 2 : d x_i = w_c (E_2 + kap_c sgn + lam_c); M = max |d x|; fixed-point SQ8 map
// pass 3: e = clip(floor((fw E_2 + fk sgn + fl) / 2^P))
//
// E_2 = SQ(e_y gamma) divides by the tensor-wide maximum of |e_y gamma|, which is known only
// after every element has been read; but per channel E_2 is a function of the 8-bit code e_y
// alone.  So one pass over the elements gathers, per channel and code v, the count n_v and
// the sum S_v of X over the elements with e_y = v, and every sum of Sec. 3.3.1's backward
// statistics follows exactly: sum e_y = sum_v v n_v, sum e_y X = sum_v v S_v, sum E_2 =
// sum_v E_2(v) n_v, sum E_2 X = sum_v E_2(v) S_v (E_2(0) = 0, so code 0 needs no bin).
// E_2(v) = SQ(v gamma_c) is monotone in v, so the E_2 extremes of a sign class of X are E_2
// at the class's extreme codes.

// Division by 2M for E_2 = SQ(z, k_e2): the numerator 2^k (z + M) + M is below 2^32 for the
// paper's widths (|z| <= 127 * 127, k_e2 <= 16), where a 32-bit invariant divisor (Granlund
// & Montgomery, Sec. 4, at N = 32) replaces the 64-bit one.
// Per channel the output code depends on (sign X, e_y) alone, so it is tabulated once per
// call (k_bnb_tab3, the same arithmetic as the per-element form) and pass 3 looks it up in
// shared memory.
constexpr int kTab3 = 3 * 256;      // (sign X + 1) 256 + e_y + 128
constexpr int kTab3P = kTab3 + 4;   // a table row in shared memory, padded by one word
constexpr int kTabCG = 8;           // channel groups (32 channels) per block of pass 3
constexpr int kHistCh = 32;         // channels per block of the histogram pass
constexpr int kHistRows = 65536;    // rows per block at most: |S_v| < 2^15 2^16 in int32
constexpr int kHistSmem = 2 * kHistCh * 256 * (int)sizeof(int);

struct E2Div {
    uint64_t M;
    UDiv div;          // 64-bit divisor by 2M
    uint32_t mp;       // 32-bit multiplier, shifts
    int32_t sh1, sh2;
    int32_t use32;
};

struct BnBwd {
    unsigned long long* sb;   // sum e_y
    unsigned long long* sg;   // sum e_y X
    unsigned long long* se;   // sum E_2
    unsigned long long* sex;  // sum E_2 X
    unsigned long long* ss;   // sum sign X
    int* emin;                // [3C] per sign class (-1, 0, +1)
    int* emax;                // [3C]
    long long* fw;
    long long* fk;
    long long* fl;
    unsigned* zmax;           // [1]
    int* pe;                  // [1]
    E2Div* e2div;             // [1]
    int2* hist;               // [gy][C][256]: per row tile of the histogram pass, (n_v, S_v)
    int16_t* t2;              // [C][256]: E_2 of e_y = -128 .. 127
    int8_t* t3;               // [C][3][256]: the output code of (sign X, e_y)
    double* scal;             // [2]: s_e2, s_out
    double* kap;              // [C] per-channel constants of d x (fin 2)
    double* lam;
    double* wc;
    unsigned long long* red;  // [4]: maxima of non-negative doubles (bit patterns)
};

// row tiles of the histogram pass: about three blocks per SM, at most kHistRows rows each
static int hist_tiles(int64_t m, int32_t C) {
    const int64_t gx = (C + kHistCh - 1) / kHistCh;
    int64_t gy = (152 * 3 + gx - 1) / gx;
    const int64_t by_rows = (m + 31) / 32;
    if (gy > by_rows) gy = by_rows;
    const int64_t need = (m + kHistRows - 1) / kHistRows;
    if (gy < need) gy = need;
    if (gy < 1) gy = 1;
    return (int)gy;
}

// the channel counts of the streamed / tiled backward passes: row_stream_plan's, and whole
// 64-channel slabs
static bool bnb_fast(int32_t C) {
    return ((C >= 64 && C <= 1024 && (C & (C - 1)) == 0) || (C > 1024 && C % 1024 == 0));
}

static BnBwd bnb_carve(WsCursor& cur, int64_t m, int32_t C) {
    BnBwd w;
    w.sb = cur.take<unsigned long long>(C);
    w.sg = cur.take<unsigned long long>(C);
    w.se = cur.take<unsigned long long>(C);
    w.sex = cur.take<unsigned long long>(C);
    w.ss = cur.take<unsigned long long>(C);
    w.emin = cur.take<int>(3 * (size_t)C);
    w.emax = cur.take<int>(3 * (size_t)C);
    w.fw = cur.take<long long>(C);
    w.fk = cur.take<long long>(C);
    w.fl = cur.take<long long>(C);
    w.zmax = cur.take<unsigned>(1);
    w.pe = cur.take<int>(1);
    w.e2div = cur.take<E2Div>(1);
    w.scal = cur.take<double>(2);
    w.kap = cur.take<double>(C);
    w.lam = cur.take<double>(C);
    w.wc = cur.take<double>(C);
    w.red = cur.take<unsigned long long>(4);
    w.t3 = cur.take<int8_t>((size_t)kTab3 * C);
    w.t2 = cur.take<int16_t>((size_t)256 * C);
    // the histogram pass runs only where the row streamer does not
    w.hist = cur.take<int2>(bnb_fast(C) && m < (int64_t(1) << 31) ? 0 : (size_t)hist_tiles(m, C) * C * 256);
    return w;
}

__global__ void k_bnb_init(BnBwd w, int32_t C) {
    for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < C; c += gridDim.x * blockDim.x) {
        w.sb[c] = 0; w.sg[c] = 0; w.se[c] = 0; w.sex[c] = 0; w.ss[c] = 0;
        for (int j = 0; j < 3; j++) { w.emin[3 * c + j] = INT_MAX; w.emax[3 * c + j] = INT_MIN; }
        if (c == 0) {
            *w.zmax = 0;
            for (int i = 0; i < 4; i++) w.red[i] = 0ull;
        }
    }
}

__device__ __forceinline__ void load4_e_a_x(int64_t v, const int8_t* ea, const int8_t* a,
                                            const int16_t* X, int e[4], int am[4], int x[4]) {
    unpack4_i8(reinterpret_cast<const int*>(ea)[v], e);
    unpack4_i8(reinterpret_cast<const int*>(a)[v], am);
    uint2 xv = reinterpret_cast<const uint2*>(X)[v];
    x[0] = (int)(int16_t)(xv.x & 0xffffu); x[1] = (int)(int16_t)(xv.x >> 16);
    x[2] = (int)(int16_t)(xv.y & 0xffffu); x[3] = (int)(int16_t)(xv.y >> 16);
}

// The histogram pass.  A block is 8 channel groups (32 channels) x 32 row lanes; each
// thread reads 4 channels of a row (the e_a and activation codes, the X codes).  The block
// keeps (n_v, S_v) of its 32 channels in shared memory (shared-memory atomics, for nonzero
// codes only) and writes them to its row tile's slab of the scratch histogram; the sign
// sums and the per-class extreme codes (four channels packed in the bytes of a word,
// byte-wise SIMD maxima / minima) are reduced over the warp and added atomically.
__global__ void __launch_bounds__(kThreads, 3) k_bnb_hist(const int8_t* __restrict__ ea,
                                                          const int8_t* __restrict__ a,
                                                          const int16_t* __restrict__ X,
                                                          const int32_t* __restrict__ gam,
                                                          int64_t m, int32_t C, BnBwd w) {
    extern __shared__ int hsm[];                 // [2][32][256]: n_v, then S_v
    for (int i = threadIdx.x; i < 2 * kHistCh * 256; i += blockDim.x) hsm[i] = 0;
    __syncthreads();
    const int C4 = C >> 2;
    const int lane = threadIdx.x & 31;
    const int cg = threadIdx.x & 7, rl = threadIdx.x >> 3;
    const int g = blockIdx.x * 8 + cg;
    const bool act = g < C4;
    int ss[4] = {0, 0, 0, 0};
    // extreme e_y per sign class of X (-, 0, +); empty: max 0x80 < min 0x7f
    uint32_t mx[3] = {0x80808080u, 0x80808080u, 0x80808080u};
    uint32_t mn[3] = {0x7f7f7f7fu, 0x7f7f7f7fu, 0x7f7f7f7fu};
    if (act) {
        int* hn = hsm + 4 * cg * 256 + 128;      // channel 4 cg, code 0
        int* hs = hn + kHistCh * 256;
        auto row = [&](const uint32_t ev, const uint32_t av, const uint2 xv) {
            const uint32_t ey = ev & __vcmpgts4(av, 0u);
            const int x[4] = {(int)(int16_t)(xv.x & 0xffffu), (int)xv.x >> 16,
                              (int)(int16_t)(xv.y & 0xffffu), (int)xv.y >> 16};
            uint32_t neg = 0u, pos = 0u;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                neg |= x[j] < 0 ? 0xffu << (8 * j) : 0u;
                pos |= x[j] > 0 ? 0xffu << (8 * j) : 0u;
                ss[j] += (x[j] > 0) - (x[j] < 0);
                const int v = (int)(int8_t)(ey >> (8 * j));
                if (v) {
                    atomicAdd(hn + j * 256 + v, 1);
                    atomicAdd(hs + j * 256 + v, x[j]);
                }
            }
            const uint32_t cls[3] = {neg, ~(neg | pos), pos};
#pragma unroll
            for (int q = 0; q < 3; q++) {
                mx[q] = __vmaxs4(mx[q], (ey & cls[q]) | (0x80808080u & ~cls[q]));
                mn[q] = __vmins4(mn[q], (ey & cls[q]) | (0x7f7f7f7fu & ~cls[q]));
            }
        };
        const uint32_t* e4 = reinterpret_cast<const uint32_t*>(ea);
        const uint32_t* a4 = reinterpret_cast<const uint32_t*>(a);
        const uint2* x4 = reinterpret_cast<const uint2*>(X);
        const int64_t step = (int64_t)gridDim.y * 32;
        int64_t r = (int64_t)blockIdx.y * 32 + rl;
        // two rows per iteration: both rows' loads in flight together
        for (; r + step < m; r += 2 * step) {
            const int64_t v0 = r * C4 + g, v1 = (r + step) * C4 + g;
            const uint32_t e0 = __ldg(e4 + v0), a0 = __ldg(a4 + v0);
            const uint2 x0 = __ldg(x4 + v0);
            const uint32_t e1 = __ldg(e4 + v1), a1 = __ldg(a4 + v1);
            const uint2 x1 = __ldg(x4 + v1);
            row(e0, a0, x0);
            row(e1, a1, x1);
        }
        if (r < m) {
            const int64_t v0 = r * C4 + g;
            row(__ldg(e4 + v0), __ldg(a4 + v0), __ldg(x4 + v0));
        }
    }
    // the warp's four row lanes of each channel group: lanes cg, cg + 8, cg + 16, cg + 24
#pragma unroll
    for (int o = 8; o < 32; o <<= 1) {
#pragma unroll
        for (int j = 0; j < 4; j++) ss[j] += __shfl_xor_sync(0xffffffffu, ss[j], o);
#pragma unroll
        for (int q = 0; q < 3; q++) {
            mx[q] = __vmaxs4(mx[q], __shfl_xor_sync(0xffffffffu, mx[q], o));
            mn[q] = __vmins4(mn[q], __shfl_xor_sync(0xffffffffu, mn[q], o));
        }
    }
    uint32_t zm = 0;
    if (lane < 8 && act) {
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const int c = 4 * g + j;
            if (ss[j]) atomicAdd(&w.ss[c], (unsigned long long)(long long)ss[j]);
            int amax = 0;
#pragma unroll
            for (int q = 0; q < 3; q++) {
                const int hi = (int)(int8_t)(mx[q] >> (8 * j)), lo = (int)(int8_t)(mn[q] >> (8 * j));
                if (lo > hi) continue;           // no element of this class
                atomicMin(&w.emin[3 * c + q], lo);
                atomicMax(&w.emax[3 * c + q], hi);
                amax = max(amax, max(abs(lo), abs(hi)));
            }
            zm = max(zm, (uint32_t)amax * (uint32_t)abs(gam[c]));
        }
    }
    zm = warp_max_u32(zm);
    if (lane == 0 && zm) atomicMax(w.zmax, zm);
    __syncthreads();
    // the block's 32 channels x 256 codes into its row tile's slab, 16 bytes a store
    const int64_t c0 = (int64_t)blockIdx.x * kHistCh;
    const int nch = (int)min((int64_t)kHistCh, (int64_t)C - c0);
    int4* dst = reinterpret_cast<int4*>(w.hist + ((int64_t)blockIdx.y * C + c0) * 256);
    for (int i = threadIdx.x; i < nch * 128; i += blockDim.x) {
        const int b0 = 2 * i;                     // bins b0, b0 + 1 of the block's channels
        dst[i] = make_int4(hsm[b0], hsm[kHistCh * 256 + b0], hsm[b0 + 1],
                           hsm[kHistCh * 256 + b0 + 1]);
    }
}

// E_2 = SQ_{k}(z) with M2 = max|z|: floor((2^k (z + M2) + M2) / (2 M2)) - 2^(k-1)
__global__ void k_bnb_fin1(BnBwd w, const double* __restrict__ s_e, int k_gamma, int k_e2) {
    uint32_t M2 = *w.zmax;
    double s_z = __dmul_rn(*s_e, ldexp(1.0, 2 - k_gamma));
    w.scal[0] = M2 ? ldexp(__dmul_rn(s_z, (double)M2), 1 - k_e2) : ldexp(s_z, 1 - k_e2);
    E2Div d;
    d.M = M2;
    const uint64_t dv = M2 ? 2ull * M2 : 1ull;
    d.div = make_udiv(dv);
    int l = 0;
    while ((uint64_t(1) << l) < dv) l++;
    d.use32 = (((uint64_t)2 * M2) << k_e2) + M2 < (uint64_t(1) << 32) && l <= 31;
    d.mp = d.use32 ? (uint32_t)((((uint64_t(1) << l) - dv) << 32) / dv + 1) : 0u;
    d.sh1 = l < 1 ? l : 1;
    d.sh2 = l - 1 > 0 ? l - 1 : 0;
    *w.e2div = d;
}

__device__ __forceinline__ int e2_code(int z, const E2Div& d, int k) {
    if (!d.M) return 0;
    int64_t c;
    if (d.use32) {
        const uint32_t num = ((uint32_t)(z + (int32_t)d.M) << k) + (uint32_t)d.M;
        const uint32_t t = __umulhi(d.mp, num);
        c = (int64_t)((t + ((num - t) >> d.sh1)) >> d.sh2) - (int64_t(1) << (k - 1));
    } else {
        uint64_t num = ((uint64_t)((int64_t)z + (int64_t)d.M) << k) + d.M;
        c = (int64_t)udiv(num, d.div) - (int64_t(1) << (k - 1));
    }
    return (int)clamp64(c, -qmax(k), qmax(k));
}

// Per channel (one warp each, eight codes a lane): the four sums over the histogram's row
// tiles and the E_2 extremes per sign class (replacing the extreme codes in emin / emax).
__global__ void k_bnb_hfin(const int32_t* __restrict__ gam, int64_t m, int32_t C, int gy,
                           int k_e2, BnBwd w) {
    const int c = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (c >= C) return;                           // whole warps leave together
    const E2Div d = *w.e2div;
    const int gc = gam[c];
    long long n[8] = {0, 0, 0, 0, 0, 0, 0, 0}, sv[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int t = 0; t < gy; t++) {
        const int4* src = reinterpret_cast<const int4*>(w.hist + ((int64_t)t * C + c) * 256);
#pragma unroll
        for (int i = 0; i < 4; i++) {
            const int4 v = src[lane * 4 + i];     // bins 8 lane + 2 i, + 1
            n[2 * i] += v.x; sv[2 * i] += v.y; n[2 * i + 1] += v.z; sv[2 * i + 1] += v.w;
        }
    }
    long long sb = 0, sg = 0, se = 0, sex = 0;
#pragma unroll
    for (int i = 0; i < 8; i++) {
        if (!n[i]) continue;
        const int v = 8 * lane + i - 128;
        const int e2 = e2_code(v * gc, d, k_e2);
        sb += (long long)v * n[i];
        sg += (long long)v * sv[i];
        se += (long long)e2 * n[i];
        sex += (long long)e2 * sv[i];
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        sb += __shfl_xor_sync(0xffffffffu, sb, o);
        sg += __shfl_xor_sync(0xffffffffu, sg, o);
        se += __shfl_xor_sync(0xffffffffu, se, o);
        sex += __shfl_xor_sync(0xffffffffu, sex, o);
    }
    if (lane < 3) {
        const int q = lane;
        const int lo = w.emin[3 * c + q], hi = w.emax[3 * c + q];
        if (lo <= hi) {
            const int e0 = e2_code(lo * gc, d, k_e2), e1 = e2_code(hi * gc, d, k_e2);
            w.emin[3 * c + q] = min(e0, e1);
            w.emax[3 * c + q] = max(e0, e1);
        }
    }
    if (lane == 0) {
        w.sb[c] = (unsigned long long)sb;
        w.sg[c] = (unsigned long long)sg;
        w.se[c] = (unsigned long long)se;
        w.sex[c] = (unsigned long long)sex;
    }
}

// the block's 32 channel tables (rows of `row` bytes) into shared memory, 16 bytes a thread
__device__ __forceinline__ void load_tables(const void* __restrict__ src, int64_t c0, int nch,
                                            int row, uint8_t* dst) {
    const int4* s4 = reinterpret_cast<const int4*>((const uint8_t*)src + c0 * row);
    int4* d4 = reinterpret_cast<int4*>(dst);
    const int n16 = nch * row / 16;
    for (int i = threadIdx.x; i < n16; i += blockDim.x) d4[i] = s4[i];
}

// Per channel (oracle order): gx = (SEX s_x)/m; kap = -gx; lam = gx (SS/m) - SE/m;
// w = s_e2 / ((c_sigma + 1) sg_step); d x = w ((E_2 + kap sgn) + lam).  Three launches of
// C/64 blocks: M = max |d x| at the extremes of each sign class (red[0]), then the bound of
// the fixed-point map (red[1]), then its constants.
__global__ void __launch_bounds__(kFinThreads) k_bnb_fin2a(BnBwd w, int64_t m, int32_t C,
                                                           const int32_t* __restrict__ csig,
                                                           const double* __restrict__ bn_scales,
                                                           int k_sigma) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    const double md = (double)m;
    const double s_x = bn_scales[IQ_BN_S_XHAT];
    const double s_e2 = w.scal[0];
    const double sg_step = ldexp(1.0, 2 - k_sigma);
    double gx = __ddiv_rn(__dmul_rn((double)(long long)w.sex[c], s_x), md);
    double kap = -gx;
    double lam = __dsub_rn(__dmul_rn(gx, __ddiv_rn((double)(long long)w.ss[c], md)),
                           __ddiv_rn((double)(long long)w.se[c], md));
    double wc = __ddiv_rn(s_e2, __dmul_rn((double)(csig[c] + 1), sg_step));
    w.kap[c] = kap;
    w.lam[c] = lam;
    w.wc[c] = wc;
    double M = 0.0;
    for (int q = 0; q < 3; q++) {
        int lo = w.emin[3 * c + q], hi = w.emax[3 * c + q];
        if (lo > hi) continue;  // empty sign class
        double sg = (double)(q - 1);
        double ks = __dmul_rn(kap, sg);
        double d0 = __dmul_rn(wc, __dadd_rn(__dadd_rn((double)lo, ks), lam));
        double d1 = __dmul_rn(wc, __dadd_rn(__dadd_rn((double)hi, ks), lam));
        M = fmax(M, fmax(fabs(d0), fabs(d1)));
    }
    red_max(&w.red[0], M);
}

__global__ void __launch_bounds__(kFinThreads) k_bnb_fin2b(BnBwd w, int32_t C, int k_e2, int k_e) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    const double M = red_get(&w.red[0]);
    if (c >= C || M == 0.0) return;
    const double qe = __ddiv_rn(ldexp(1.0, k_e - 1), M);
    const double emax = (double)qmax(k_e2);
    const double kap = w.kap[c], lam = w.lam[c];
    double om = __dmul_rn(w.wc[c], qe);
    red_max(&w.red[1], __dadd_rn(__dadd_rn(__dmul_rn(fabs(om), emax), fabs(__dmul_rn(om, kap))),
                                 fabs(__dmul_rn(om, lam))));
}

__global__ void __launch_bounds__(kFinThreads) k_bnb_fin2c(BnBwd w, int32_t C, int k_e,
                                                           double* __restrict__ s_out) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    const double M = red_get(&w.red[0]);
    if (M == 0.0) {
        if (c < C) { w.fw[c] = 0; w.fk[c] = 0; w.fl[c] = 0; }
        if (c == 0) { *w.pe = 1; w.scal[1] = ldexp(1.0, 1 - k_e); *s_out = w.scal[1]; }
        return;
    }
    const int pe = shift_of(red_get(&w.red[1]));
    if (c < C) {
        const double qe = __ddiv_rn(ldexp(1.0, k_e - 1), M);
        const double kap = w.kap[c], lam = w.lam[c];
        double om = __dmul_rn(w.wc[c], qe);
        w.fw[c] = (long long)rhu(ldexp(om, pe));
        w.fk[c] = (long long)rhu(ldexp(__dmul_rn(om, kap), pe));
        w.fl[c] = (long long)rhu(ldexp(__dmul_rn(om, lam), pe)) + (1LL << (pe - 1));
    }
    if (c == 0) { *w.pe = pe; w.scal[1] = ldexp(M, 1 - k_e); *s_out = w.scal[1]; }
}

// the output-code table: t3[c][(s + 1) 256 + e_y + 128] = clip(floor((fw E_2 + fk s + fl) /
// 2^P)) with E_2 = SQ_kE2(e_y gamma_c)
__global__ void k_bnb_tab3(const int32_t* __restrict__ gam, int32_t C, int k_e2, int k_e,
                           BnBwd w) {
    const E2Div d = *w.e2div;
    const int pe = *w.pe;
    const int64_t eq = qmax(k_e);
    const int64_t n = (int64_t)C * kTab3;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i / kTab3), r = (int)(i - (int64_t)c * kTab3);
        const int sgn = (r >> 8) - 1, ey = (r & 255) - 128;
        const int e2 = e2_code(ey * gam[c], d, k_e2);
        const long long tt = w.fw[c] * (long long)e2 + w.fk[c] * (long long)sgn + w.fl[c];
        w.t3[i] = (int8_t)clamp64(tt >> pe, -eq, eq);
    }
}

// ------------------------------------------------------------------ tiled backward passes
// For C a power of two >= 64 or a multiple of 1024 the backward runs as three passes over 2-D
// tiles (the histogram pass above is the fallback for other C): A, max |e_y| per channel,
// sum sign X and the extreme codes of each sign class of X; B, the per-channel sums of e_y,
// e_y X, E_2 and E_2 X; and the output pass.  The integer ALU work of the statistics is split
// between A and B so that each stays near the memory rate.  A block owns a slab of kTileC = 64
// channels, whose per-channel tables (E_2 of the code, or the output code of (sign X, code))
// sit in shared memory, and row chunks of kTileR rows of it, each chunk one TMA tile per array
// (e_a, the activation codes, X; rows past m read as zeros and are not counted).
constexpr int kTileC = 64;
constexpr int kTileR = 128;
constexpr int kTileStages = 4;
constexpr int kTileStage = kTileR * kTileC * 4;          // int8 e_a, int8 a, int16 X
constexpr int kTab2P = 258;                              // E_2 table row, padded (int16)
constexpr int kTileSmem = 1024 + kTileStages * kTileStage + 2 * kTileStages * 8;

// byte permute with sign replication (a selector nibble with its msb set copies the sign of
// the selected byte): 0x9180 / 0xb3a2 widen bytes 0, 1 / 2, 3 to two signed 16-bit lanes
__device__ __forceinline__ uint32_t prmt_sext(uint32_t a, uint32_t sel) {
    uint32_t r;
    asm("prmt.b32 %0, %1, 0, %2;" : "=r"(r) : "r"(a), "r"(sel));
    return r;
}

__device__ __forceinline__ uint8_t* align1k(uint8_t* p) {
    return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// the E_2 table: t2[c][e_y + 128] = SQ_kE2(e_y gamma_c)
__global__ void k_bnb_tab2(const int32_t* __restrict__ gam, int32_t C, int k_e2, BnBwd w) {
    const E2Div d = *w.e2div;
    const int64_t n = (int64_t)C * 256;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i >> 8), ey = (int)(i & 255) - 128;
        w.t2[i] = (int16_t)e2_code(ey * gam[c], d, k_e2);
    }
}

// thread 0: chunk k of the slab's three tiles into `st`
__device__ __forceinline__ void tile_issue(const CUtensorMap* me, const CUtensorMap* ma,
                                           const CUtensorMap* mxh, uint8_t* st, uint64_t* bar,
                                           int64_t k) {
    tc::mbar_arrive_expect_tx(bar, kTileStage);
    const int x = blockIdx.x * kTileC, y = (int)(k * kTileR);
    tc::tma_load_2d(st, me, bar, x, y);
    tc::tma_load_2d(st + kTileR * kTileC, ma, bar, x, y);
    tc::tma_load_2d(st + 2 * kTileR * kTileC, mxh, bar, x, y);
}

// PTX prmt with its sign-replicating selectors (a selector nibble with bit 3 set fills the
// byte with the sign of the byte it selects); __byte_perm uses only the low 3 bits
__device__ __forceinline__ uint32_t prmt_sx(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// Pass A over tiles: sum sign X per channel, and the extreme code e_y of each sign class of X
// (-, 0, +), two channels per word in int16 lanes (packed 16-bit min / max; the codes are
// widened by sign-replicating byte permutes, the class masks taken from the sign bytes of X
// and min(X, 1) per lane); max |e_y| per channel (for max |e_y gamma|) follows from the
// class extremes.
__global__ void __launch_bounds__(kStreamThreads, 1)
    k_bnb_a_t(const __grid_constant__ CUtensorMap me, const __grid_constant__ CUtensorMap ma,
              const __grid_constant__ CUtensorMap mxh, int64_t m, int32_t C,
              const int32_t* __restrict__ gam, BnBwd w, int* __restrict__ err) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1k(smem_raw);
    if (__syncthreads_or(threadIdx.x == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    const int c_base = blockIdx.x * kTileC;
    const int g = threadIdx.x & 15, rl = threadIdx.x >> 4;       // 16 groups x 32 row lanes
    long long ss[4] = {0, 0, 0, 0};
    // per sign class q (X < 0, X = 0, X > 0) the extremes of e_y, two channels per word as
    // packed int16 (native 16-bit min / max): [q][0, 1] max of channels (0,1), (2,3); [q][2, 3]
    // the minima.  Empty: max 0x8000 (below every code), min 0x7fff.
    uint32_t ext[3][4];
#pragma unroll
    for (int q = 0; q < 3; q++) {
        ext[q][0] = ext[q][1] = 0x80008000u;
        ext[q][2] = ext[q][3] = 0x7fff7fffu;
    }
    const int64_t nchunk = (m + kTileR - 1) / kTileR;
    const bool ok = pipe_chunks<kTileStages>(
        nchunk, kTileR, m, kTileStage, smem, err,
        [&](uint8_t* st, uint64_t* bar, int64_t k) { tile_issue(&me, &ma, &mxh, st, bar, k); },
        [&](const uint8_t* st, int rows, int64_t) {
            const uint32_t* e4 = reinterpret_cast<const uint32_t*>(st);
            const uint32_t* a4 = reinterpret_cast<const uint32_t*>(st + kTileR * kTileC);
            const uint2* x4 = reinterpret_cast<const uint2*>(st + 2 * kTileR * kTileC);
            // the chunk's counts per channel, two int16 lanes a word: X < 0 and X != 0
            uint32_t nneg[2] = {0u, 0u}, nnz[2] = {0u, 0u};
#pragma unroll
            for (int u = 0; u < kTileR / 32; u++) {
                const int r = rl + 32 * u;
                if (r >= rows) break;
                const int i = r * 16 + g;
                const uint32_t a = a4[i];
                // byte j of am: 0xff where A_j > 0 (nonzero with a clear sign bit)
                const uint32_t nzb = ((a & 0x7f7f7f7fu) + 0x7f7f7f7fu) | a;
                const uint32_t am = prmt_sx(nzb, 0u, 0xBA98) & ~prmt_sx(a, 0u, 0xBA98);
                const uint32_t ey = e4[i] & am;
                // e_y of channels (0,1) and (2,3) sign-extended to int16 lanes
                const uint32_t ey16[2] = {prmt_sx(ey, 0u, 0x9180), prmt_sx(ey, 0u, 0xB3A2)};
                const uint2 xv = x4[i];
                const uint32_t xw[2] = {xv.x, xv.y};
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    // per int16 lane: 0xffff where X < 0 (its sign), 1 / 0xffff where X != 0
                    const uint32_t neg = prmt_sx(xw[h], 0u, 0xBB99);
                    uint32_t nz1;
                    asm("min.u16x2 %0, %1, %2;" : "=r"(nz1) : "r"(xw[h]), "r"(0x00010001u));
                    const uint32_t nz = nz1 * 0xffffu;
                    nneg[h] += neg & 0x00010001u;
                    nnz[h] += nz1;
                    const uint32_t cls[3] = {neg, ~nz, nz & ~neg};
#pragma unroll
                    for (int q = 0; q < 3; q++) {
                        const uint32_t vx = (ey16[h] & cls[q]) | (0x80008000u & ~cls[q]);
                        const uint32_t vn = (ey16[h] & cls[q]) | (0x7fff7fffu & ~cls[q]);
                        asm("max.s16x2 %0, %0, %1;" : "+r"(ext[q][h]) : "r"(vx));
                        asm("min.s16x2 %0, %0, %1;" : "+r"(ext[q][2 + h]) : "r"(vn));
                    }
                }
            }
            // sum sign X = #(X > 0) - #(X < 0) = #(X != 0) - 2 #(X < 0)
#pragma unroll
            for (int j = 0; j < 4; j++) {
                const int sh = 16 * (j & 1);
                ss[j] += (int)((nnz[j >> 1] >> sh) & 0xffffu) -
                         2 * (int)((nneg[j >> 1] >> sh) & 0xffffu);
            }
        });
    if (!ok) return;
    long long* sq = reinterpret_cast<long long*>(smem);                // [32][64]
    uint32_t* sp = reinterpret_cast<uint32_t*>(sq + 32 * kTileC);      // [12][512]
#pragma unroll
    for (int j = 0; j < 4; j++) sq[rl * kTileC + 4 * g + j] = ss[j];
#pragma unroll
    for (int q = 0; q < 3; q++)
#pragma unroll
        for (int w = 0; w < 4; w++) sp[(4 * q + w) * kStreamThreads + threadIdx.x] = ext[q][w];
    __syncthreads();
    const int col = threadIdx.x;
    uint32_t zm = 0;
    if (col < kTileC) {
        long long t = 0;
        for (int i = 0; i < 32; i++) t += sq[i * kTileC + col];
        const int c = c_base + col;
        atomicAdd(&w.ss[c], (unsigned long long)t);
        const int gg = col >> 2, j = col & 3, wd = j >> 1, sh = 16 * (j & 1);
        int amax = 0;                              // max |e_y| over every class
#pragma unroll
        for (int q = 0; q < 3; q++) {
            int hi = -32768, lo = 32767;
            for (int i = 0; i < 32; i++) {
                const int k = i * 16 + gg;
                hi = max(hi, (int)(int16_t)(sp[(4 * q + wd) * kStreamThreads + k] >> sh));
                lo = min(lo, (int)(int16_t)(sp[(4 * q + 2 + wd) * kStreamThreads + k] >> sh));
            }
            if (lo > hi) continue;                 // no element of this class
            amax = max(amax, max(abs(hi), abs(lo)));
            atomicMin(&w.emin[3 * c + q], lo);     // codes; k_bnb_ext maps them to E_2
            atomicMax(&w.emax[3 * c + q], hi);
        }
        zm = (uint32_t)amax * (uint32_t)abs(gam[c]);
    }
    if (threadIdx.x < 64) {
        zm = warp_max_u32(zm);
        if ((threadIdx.x & 31) == 0 && zm) atomicMax(w.zmax, zm);
    }
}

// E_2 is monotone in e_y: the E_2 extremes of a sign class are E_2 at its extreme codes
__global__ void k_bnb_ext(int32_t C, BnBwd w) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;         // 3 c + q
    if (i >= 3 * C) return;
    const int lo = w.emin[i], hi = w.emax[i];
    if (lo > hi) return;
    const int16_t* t = w.t2 + (int64_t)(i / 3) * 256 + 128;
    const int e0 = t[lo], e1 = t[hi];
    w.emin[i] = min(e0, e1);
    w.emax[i] = max(e0, e1);
}

// Pass B over tiles: per channel sum e_y, sum e_y X, sum E_2 and sum E_2 X, E_2 from the
// slab's table in shared memory
__global__ void __launch_bounds__(kStreamThreads, 1)
    k_bnb_b_t(const __grid_constant__ CUtensorMap me, const __grid_constant__ CUtensorMap ma,
              const __grid_constant__ CUtensorMap mxh, int64_t m, int32_t C, BnBwd w,
              int* __restrict__ err) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1k(smem_raw);
    int16_t* tab = reinterpret_cast<int16_t*>(smem + kTileStages * kTileStage + 2 * kTileStages * 8);
    if (__syncthreads_or(threadIdx.x == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    const int c_base = blockIdx.x * kTileC;
    for (int i = threadIdx.x; i < kTileC * 128; i += blockDim.x) {
        const int ch = i >> 7, k2 = i & 127;            // two entries a word
        reinterpret_cast<uint32_t*>(tab + ch * kTab2P)[k2] =
            reinterpret_cast<const uint32_t*>(w.t2 + (int64_t)(c_base + ch) * 256)[k2];
    }
    __syncthreads();
    const int g = threadIdx.x & 15, rl = threadIdx.x >> 4;
    const int16_t* tb = tab + 4 * g * kTab2P + 128;
    long long sb[4] = {0, 0, 0, 0}, sg[4] = {0, 0, 0, 0}, se[4] = {0, 0, 0, 0};
    long long sx[4] = {0, 0, 0, 0};
    const int64_t nchunk = (m + kTileR - 1) / kTileR;
    const bool ok = pipe_chunks<kTileStages>(
        nchunk, kTileR, m, kTileStage, smem, err,
        [&](uint8_t* st, uint64_t* bar, int64_t k) { tile_issue(&me, &ma, &mxh, st, bar, k); },
        [&](const uint8_t* st, int rows, int64_t) {
            const uint32_t* e4 = reinterpret_cast<const uint32_t*>(st);
            const uint32_t* a4 = reinterpret_cast<const uint32_t*>(st + kTileR * kTileC);
            const uint2* x4 = reinterpret_cast<const uint2*>(st + 2 * kTileR * kTileC);
            // the chunk's partial sums in 32 bits (kTileR / 32 rows a thread: |e_y X| < 2^22,
            // |E_2| < 2^15; a pair of E_2 X products < 2^31)
            int cb[4] = {0, 0, 0, 0}, cg[4] = {0, 0, 0, 0}, ce[4] = {0, 0, 0, 0};
#pragma unroll
            for (int u = 0; u < kTileR / 32; u += 2) {
                int p2[4] = {0, 0, 0, 0};
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    const int r = rl + 32 * (u + h);
                    if (r >= rows) break;
                    const int i = r * 16 + g;
                    const uint32_t ey = e4[i] & __vcmpgts4(a4[i], 0u);
                    const uint2 xv = x4[i];
                    const int x[4] = {(int)(int16_t)(xv.x & 0xffffu), (int)xv.x >> 16,
                                      (int)(int16_t)(xv.y & 0xffffu), (int)xv.y >> 16};
#pragma unroll
                    for (int j = 0; j < 4; j++) {
                        const int v = (int)(int8_t)(ey >> (8 * j));
                        const int e2 = tb[j * kTab2P + v];   // E_2(0) = 0
                        cb[j] += v;
                        cg[j] += v * x[j];
                        ce[j] += e2;
                        p2[j] += e2 * x[j];
                    }
                }
#pragma unroll
                for (int j = 0; j < 4; j++) sx[j] += p2[j];
            }
#pragma unroll
            for (int j = 0; j < 4; j++) { sb[j] += cb[j]; sg[j] += cg[j]; se[j] += ce[j]; }
        });
    if (!ok) return;
    constexpr int NQ = 4;
    long long* sq = reinterpret_cast<long long*>(smem);             // [NQ][32][64]
#pragma unroll
    for (int j = 0; j < 4; j++) {
        const int i = rl * kTileC + 4 * g + j;
        sq[0 * 32 * kTileC + i] = sb[j];
        sq[1 * 32 * kTileC + i] = sg[j];
        sq[2 * 32 * kTileC + i] = se[j];
        sq[3 * 32 * kTileC + i] = sx[j];
    }
    __syncthreads();
    const int col = threadIdx.x;
    if (col < kTileC) {
        long long t[NQ] = {0, 0, 0, 0};
        for (int i = 0; i < 32; i++)
#pragma unroll
            for (int q = 0; q < NQ; q++) t[q] += sq[q * 32 * kTileC + i * kTileC + col];
        const int c = c_base + col;
        atomicAdd(&w.sb[c], (unsigned long long)t[0]);
        atomicAdd(&w.sg[c], (unsigned long long)t[1]);
        atomicAdd(&w.se[c], (unsigned long long)t[2]);
        atomicAdd(&w.sex[c], (unsigned long long)t[3]);
    }
}

__global__ void __launch_bounds__(kStreamThreads, 1)
    k_bnb_out_t(const __grid_constant__ CUtensorMap me, const __grid_constant__ CUtensorMap ma,
                const __grid_constant__ CUtensorMap mxh, int64_t m, int32_t C, BnBwd w,
                int8_t* __restrict__ out, uint2* __restrict__ out16, int* __restrict__ err) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = align1k(smem_raw);
    uint8_t* tab = smem + kTileStages * kTileStage + 2 * kTileStages * 8;   // [64][kTab3P]
    if (__syncthreads_or(threadIdx.x == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    const int c_base = blockIdx.x * kTileC;
    {
        const uint32_t* src = reinterpret_cast<const uint32_t*>(w.t3 + (int64_t)c_base * kTab3);
        for (int i = threadIdx.x; i < kTileC * (kTab3 / 4); i += blockDim.x) {
            const int ch = i / (kTab3 / 4), k = i - ch * (kTab3 / 4);
            reinterpret_cast<uint32_t*>(tab + ch * kTab3P)[k] = src[i];
        }
    }
    __syncthreads();
    const int g = threadIdx.x & 15, rl = threadIdx.x >> 4;
    const int8_t* tb = reinterpret_cast<const int8_t*>(tab) + 4 * g * kTab3P + 256 + 128;
    const int64_t nchunk = (m + kTileR - 1) / kTileR;
    pipe_chunks<kTileStages>(
        nchunk, kTileR, m, kTileStage, smem, err,
        [&](uint8_t* st, uint64_t* bar, int64_t k) { tile_issue(&me, &ma, &mxh, st, bar, k); },
        [&](const uint8_t* st, int rows, int64_t r0) {
            const uint32_t* e4 = reinterpret_cast<const uint32_t*>(st);
            const uint32_t* a4 = reinterpret_cast<const uint32_t*>(st + kTileR * kTileC);
            const uint2* x4 = reinterpret_cast<const uint2*>(st + 2 * kTileR * kTileC);
#pragma unroll
            for (int u = 0; u < kTileR / 32; u++) {
                const int r = rl + 32 * u;
                if (r >= rows) break;
                const int i = r * 16 + g;
                const uint32_t ey = e4[i] & __vcmpgts4(a4[i], 0u);
                const uint2 xv = x4[i];
                const int x[4] = {(int)(int16_t)(xv.x & 0xffffu), (int)xv.x >> 16,
                                  (int)(int16_t)(xv.y & 0xffffu), (int)xv.y >> 16};
                uint32_t o = 0;
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    const int v = (int)(int8_t)(ey >> (8 * j));
                    const int sg = (x[j] > 0) - (x[j] < 0);
                    o |= ((uint32_t)(uint8_t)tb[j * kTab3P + sg * 256 + v]) << (8 * j);
                }
                const int64_t oi = (r0 + r) * C + c_base + 4 * g;
                *reinterpret_cast<uint32_t*>(out + oi) = o;
                if (out16) {          // the fp16 copy of the 4 error codes
                    uint2 hv;
                    tc::i8x4_to_f16x4(o, hv.x, hv.y);
                    out16[oi >> 2] = hv;
                }
            }
        });
}

// e = the output code of (sign X, e_y) per element, from the block's tables in shared memory
__global__ void __launch_bounds__(kThreads) k_bnb_pass3(const int8_t* __restrict__ ea,
                                                        const int8_t* __restrict__ a,
                                                        const int16_t* __restrict__ X,
                                                        int64_t m, int32_t C, int CG, BnBwd w,
                                                        int8_t* __restrict__ out) {
    __shared__ __align__(16) int8_t tab[4 * kTabCG * kTab3];
    const int C4 = C >> 2;
    const int cg = threadIdx.x % CG, rl = threadIdx.x / CG, RL = blockDim.x / CG;
    const int g = blockIdx.x * CG + cg;
    {
        const int64_t c0 = 4 * (int64_t)blockIdx.x * CG;
        const int nch = (int)min((int64_t)4 * CG, (int64_t)C - c0);
        load_tables(w.t3, c0, nch, kTab3, reinterpret_cast<uint8_t*>(tab));
    }
    __syncthreads();
    if (g >= C4) return;
    const int8_t* tb = tab + 4 * cg * kTab3;
    const int64_t step = (int64_t)gridDim.y * RL;
    auto code4 = [&](const int (&e)[4], const int (&am)[4], const int (&x)[4]) {
        uint32_t o = 0;
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const int ey = am[j] > 0 ? e[j] : 0;
            const int sg = (x[j] > 0) - (x[j] < 0);
            o |= ((uint32_t)(uint8_t)tb[j * kTab3 + (sg + 1) * 256 + ey + 128]) << (8 * j);
        }
        return o;
    };
    int64_t r = (int64_t)blockIdx.y * RL + rl;
    // four rows per iteration: all their loads in flight together
    for (; r + 3 * step < m; r += 4 * step) {
        int e[4][4], am[4][4], x[4][4];
#pragma unroll
        for (int u = 0; u < 4; u++) load4_e_a_x((r + u * step) * C4 + g, ea, a, X, e[u], am[u], x[u]);
#pragma unroll
        for (int u = 0; u < 4; u++)
            reinterpret_cast<uint32_t*>(out)[(r + u * step) * C4 + g] = code4(e[u], am[u], x[u]);
    }
    for (; r < m; r += step) {
        int e[4], am[4], x[4];
        load4_e_a_x(r * C4 + g, ea, a, X, e, am, x);
        reinterpret_cast<uint32_t*>(out)[r * C4 + g] = code4(e, am, x);
    }
}

// int8 / int16 code j of a packed row segment
__device__ __forceinline__ int code8(const uint32_t* o, int j) {
    return (int)(int8_t)((o[j >> 2] >> (8 * (j & 3))) & 0xffu);
}
__device__ __forceinline__ int code16(const uint32_t* o, int j) {
    const uint32_t v = o[j >> 1];
    return (j & 1) ? (int)v >> 16 : (int)(int16_t)(v & 0xffffu);
}

// Pass 3 with 16 channels per thread (C % 16 == 0): 16-byte loads of the errors and
// activation codes, two of the X codes, one 16-byte store.  A block is 4 channel groups
// (64 channels) x 64 row lanes; the 64 channels' tables sit in shared memory in rows of
// 772 bytes (the 768-byte rows padded by one word, so that the rows of neighbouring
// channels start in different banks).

__global__ void __launch_bounds__(kThreads, 4) k_bnb_p3w(const int8_t* __restrict__ ea,
                                                         const int8_t* __restrict__ a,
                                                         const int16_t* __restrict__ X,
                                                         int64_t m, int32_t C, BnBwd w,
                                                         int8_t* __restrict__ out) {
    extern __shared__ __align__(16) uint32_t tab3w[];   // [64][kTab3P / 4]
    const int64_t cb = 64 * (int64_t)blockIdx.x;
    const int nch = (int)min((int64_t)64, (int64_t)C - cb);
    {
        const uint32_t* src = reinterpret_cast<const uint32_t*>(w.t3 + cb * kTab3);
        for (int i = threadIdx.x; i < nch * (kTab3 / 4); i += blockDim.x) {
            const int ch = i / (kTab3 / 4), k = i - ch * (kTab3 / 4);
            tab3w[ch * (kTab3P / 4) + k] = src[i];
        }
    }
    __syncthreads();
    const int cg = threadIdx.x & 3, rl = threadIdx.x >> 2;
    if (16 * cg >= nch) return;
    const int64_t c0 = cb + 16 * cg;
    const int8_t* tb = reinterpret_cast<const int8_t*>(tab3w) + 16 * cg * kTab3P;
    const int64_t step = (int64_t)gridDim.y * 64;
    auto code16x = [&](const int4 e, const int4 am, const int4 x0, const int4 x1) {
        const uint32_t ev[4] = {(uint32_t)e.x, (uint32_t)e.y, (uint32_t)e.z, (uint32_t)e.w};
        const uint32_t av[4] = {(uint32_t)am.x, (uint32_t)am.y, (uint32_t)am.z, (uint32_t)am.w};
        const uint32_t xv[8] = {(uint32_t)x0.x, (uint32_t)x0.y, (uint32_t)x0.z, (uint32_t)x0.w,
                                (uint32_t)x1.x, (uint32_t)x1.y, (uint32_t)x1.z, (uint32_t)x1.w};
        uint32_t o[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int j = 0; j < 16; j++) {
            const int ey = code8(av, j) > 0 ? code8(ev, j) : 0;
            const int xx = code16(xv, j);
            const int sg = (xx > 0) - (xx < 0);
            o[j >> 2] |= ((uint32_t)(uint8_t)tb[j * kTab3P + (sg + 1) * 256 + ey + 128])
                         << (8 * (j & 3));
        }
        return make_uint4(o[0], o[1], o[2], o[3]);
    };
    int64_t r = (int64_t)blockIdx.y * 64 + rl;
    // two rows per iteration: all their loads in flight together
    for (; r + step < m; r += 2 * step) {
        const int64_t o0 = r * C + c0, o1 = (r + step) * C + c0;
        const int4 e0 = __ldg(reinterpret_cast<const int4*>(ea + o0));
        const int4 a0 = __ldg(reinterpret_cast<const int4*>(a + o0));
        const int4 x00 = __ldg(reinterpret_cast<const int4*>(X + o0));
        const int4 x01 = __ldg(reinterpret_cast<const int4*>(X + o0 + 8));
        const int4 e1 = __ldg(reinterpret_cast<const int4*>(ea + o1));
        const int4 a1 = __ldg(reinterpret_cast<const int4*>(a + o1));
        const int4 x10 = __ldg(reinterpret_cast<const int4*>(X + o1));
        const int4 x11 = __ldg(reinterpret_cast<const int4*>(X + o1 + 8));
        *reinterpret_cast<uint4*>(out + o0) = code16x(e0, a0, x00, x01);
        *reinterpret_cast<uint4*>(out + o1) = code16x(e1, a1, x10, x11);
    }
    if (r < m) {
        const int64_t o0 = r * C + c0;
        *reinterpret_cast<uint4*>(out + o0) =
            code16x(__ldg(reinterpret_cast<const int4*>(ea + o0)),
                    __ldg(reinterpret_cast<const int4*>(a + o0)),
                    __ldg(reinterpret_cast<const int4*>(X + o0)),
                    __ldg(reinterpret_cast<const int4*>(X + o0 + 8)));
    }
}

size_t bn_bwd_ws_bytes(int64_t m, int32_t C) {
    WsCursor c(nullptr, 0);
    bnb_carve(c, m, C);
    return c.off + 256;
}

}  // namespace iq

using namespace iq;

// ==================================================================== C ABI

extern "C" iq_status iq_bn_int_workspace_size(int64_t m, int32_t c, size_t* bytes) {
    if (!bytes || m < 0 || c <= 0) return IQ_ERR_INVALID_ARG;
    size_t f = bn_fwd_ws_bytes(c), b = bn_bwd_ws_bytes(m, c);
    *bytes = f > b ? f : b;
    return IQ_OK;
}

static bool bn_shape_ok(int64_t m, int32_t c) {
    return m > 0 && c > 0 && (c % 4) == 0 && c <= 65536 && m < (int64_t(1) << 40);
}

extern "C" iq_status iq_bn_int_fwd(const int32_t* acc, int64_t m, int32_t c, const double* s_acc,
                                   const int32_t* gamma, const int32_t* beta,
                                   const iq_bn_bits* bits, int16_t* xhat, int8_t* a, double* s_a,
                                   int32_t* bn_codes, double* bn_scales, int64_t* bn_fixed,
                                   void* ws, size_t ws_bytes, iq_stream stream) {
    if (!acc || !s_acc || !gamma || !beta || !a || !s_a) return IQ_ERR_INVALID_ARG;
    if (!bn_shape_ok(m, c)) return (m > 0 && c > 0) ? IQ_ERR_UNSUPPORTED : IQ_ERR_INVALID_ARG;
    iq_bn_bits b = bn_bits_or_default(bits);
    if (!bn_bits_valid(b)) return IQ_ERR_INVALID_ARG;
    if (((uintptr_t)acc | (uintptr_t)a | (uintptr_t)xhat) & 15) return IQ_ERR_INVALID_ARG;
    size_t need = bn_fwd_ws_bytes(c);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    WsCursor cur(ws, ws_bytes);
    BnStats s = bn_stats_carve(cur, c);
    iq_status r = bn_stats_init(s, c, st);
    if (r != IQ_OK) return r;
    r = bn_stats_pass(acc, m, c, s, st);
    if (r != IQ_OK) return r;
    return bn_fwd_after_stats(acc, m, c, s_acc, gamma, beta, b, s, xhat, a, s_a, bn_codes,
                              bn_scales, bn_fixed, st);
}

extern "C" iq_status iq_bn_int_bwd(const int8_t* e_a, const double* s_e, const int8_t* a,
                                   const int16_t* xhat, int64_t m, int32_t c,
                                   const int32_t* gamma, const int32_t* bn_codes,
                                   const double* bn_scales, const iq_bn_bits* bits, int k_e2,
                                   int8_t* e, double* s_e_out, int64_t* dgamma, int64_t* dbeta,
                                   void* e_f16, void* ws, size_t ws_bytes, iq_stream stream) {
    if (!e_a || !s_e || !a || !xhat || !gamma || !bn_codes || !bn_scales || !e || !s_e_out)
        return IQ_ERR_INVALID_ARG;
    if (e_f16 && !f16_copy_ok(e, e_f16, m * (int64_t)c)) return IQ_ERR_INVALID_ARG;
    if (!bn_shape_ok(m, c)) return (m > 0 && c > 0) ? IQ_ERR_UNSUPPORTED : IQ_ERR_INVALID_ARG;
    iq_bn_bits b = bn_bits_or_default(bits);
    if (!bn_bits_valid(b) || k_e2 < 2 || k_e2 > 16) return IQ_ERR_INVALID_ARG;
    if (((uintptr_t)e_a | (uintptr_t)a | (uintptr_t)xhat | (uintptr_t)e) & 15)
        return IQ_ERR_INVALID_ARG;
    if (m > (int64_t)65535 * kHistRows) return IQ_ERR_UNSUPPORTED;
    size_t need = bn_bwd_ws_bytes(m, c);
    if (!ws || ws_bytes < need) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    WsCursor cur(ws, ws_bytes);
    BnBwd w = bnb_carve(cur, m, c);
    k_bnb_init<<<(c + 255) / 256, 256, 0, st>>>(w, c);
    IQ_LAUNCH_CHECK();
    int* err = device_status_ptr();
    if (!err) return IQ_ERR_CUDA;
    const bool streamed = bnb_fast(c) && m < (int64_t(1) << 31);
    const int fb = (c + kFinThreads - 1) / kFinThreads;
    if (streamed) {
        CUtensorMap me, ma, mxh;
        iq_status r = encode_rows_2d(e_a, 1, m, c, kTileC, kTileR, &me);
        if (r == IQ_OK) r = encode_rows_2d(a, 1, m, c, kTileC, kTileR, &ma);
        if (r == IQ_OK) r = encode_rows_2d(xhat, 2, m, c, kTileC, kTileR, &mxh);
        if (r != IQ_OK) return r;
        static bool attr_a = false, attr_b = false, attr_o = false;
        const int smem_a = kTileSmem, smem_b = kTileSmem + kTileC * kTab2P * 2,
                  smem_o = kTileSmem + kTileC * kTab3P;
        if (!attr_a) {
            IQ_CUDA_CHECK(cudaFuncSetAttribute(k_bnb_a_t,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, smem_a));
            attr_a = true;
        }
        if (!attr_b) {
            IQ_CUDA_CHECK(cudaFuncSetAttribute(k_bnb_b_t,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, smem_b));
            attr_b = true;
        }
        if (!attr_o) {
            IQ_CUDA_CHECK(cudaFuncSetAttribute(k_bnb_out_t,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, smem_o));
            attr_o = true;
        }
        const int sms = device_sms();
        const int slabs = c / kTileC;
        int64_t gy = sms / slabs;               // one block per SM: no second wave
        if (gy < 1) gy = 1;
        const int64_t nchunk = (m + kTileR - 1) / kTileR;
        if (gy > nchunk) gy = nchunk;
        if (gy > 65535) gy = 65535;
        const dim3 tgrid((unsigned)slabs, (unsigned)gy);
        kt_pre(st);
        k_bnb_a_t<<<tgrid, kStreamThreads, smem_a, st>>>(me, ma, mxh, m, c, gamma, w, err);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_BNB_PASS1, 4.0 * (double)m * c);
        k_bnb_fin1<<<1, 1, 0, st>>>(w, s_e, b.k_gamma, k_e2);
        IQ_LAUNCH_CHECK();
        const int tb2 = (int)(((int64_t)c * 256 + kThreads - 1) / kThreads);
        k_bnb_tab2<<<tb2 < 152 * 4 ? tb2 : 152 * 4, kThreads, 0, st>>>(gamma, c, k_e2, w);
        IQ_LAUNCH_CHECK();
        k_bnb_ext<<<(3 * c + kThreads - 1) / kThreads, kThreads, 0, st>>>(c, w);
        IQ_LAUNCH_CHECK();
        kt_pre(st);
        k_bnb_b_t<<<tgrid, kStreamThreads, smem_b, st>>>(me, ma, mxh, m, c, w, err);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_BNB_PASS2, 4.0 * (double)m * c);
        k_bnb_fin2a<<<fb, kFinThreads, 0, st>>>(w, m, c, bn_codes + c, bn_scales, b.k_sigma);
        IQ_LAUNCH_CHECK();
        k_bnb_fin2b<<<fb, kFinThreads, 0, st>>>(w, c, k_e2, 8);
        IQ_LAUNCH_CHECK();
        k_bnb_fin2c<<<fb, kFinThreads, 0, st>>>(w, c, 8, s_e_out);
        IQ_LAUNCH_CHECK();
        const int tb3 = (int)(((int64_t)c * kTab3 + kThreads - 1) / kThreads);
        k_bnb_tab3<<<tb3 < 152 * 4 ? tb3 : 152 * 4, kThreads, 0, st>>>(gamma, c, k_e2, 8, w);
        IQ_LAUNCH_CHECK();
        kt_pre(st);
        k_bnb_out_t<<<tgrid, kStreamThreads, smem_o, st>>>(me, ma, mxh, m, c, w, e,
                                                           (uint2*)e_f16, err);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_BNB_PASS3, (e_f16 ? 7.0 : 5.0) * (double)m * c);
    } else {
        const int gy = hist_tiles(m, c);
        static bool hist_attr = false;
        if (!hist_attr) {
            IQ_CUDA_CHECK(cudaFuncSetAttribute(k_bnb_hist, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               kHistSmem));
            hist_attr = true;
        }
        kt_pre(st);
        k_bnb_hist<<<dim3((unsigned)((c + kHistCh - 1) / kHistCh), (unsigned)gy), kThreads, kHistSmem,
                     st>>>(e_a, a, xhat, gamma, m, c, w);
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_BNB_PASS1, 4.0 * (double)m * c);
        k_bnb_fin1<<<1, 1, 0, st>>>(w, s_e, b.k_gamma, k_e2);
        IQ_LAUNCH_CHECK();
        k_bnb_hfin<<<(unsigned)(((int64_t)c * 32 + kThreads - 1) / kThreads), kThreads, 0, st>>>(
            gamma, m, c, gy, k_e2, w);
        IQ_LAUNCH_CHECK();
        k_bnb_fin2a<<<fb, kFinThreads, 0, st>>>(w, m, c, bn_codes + c, bn_scales, b.k_sigma);
        IQ_LAUNCH_CHECK();
        k_bnb_fin2b<<<fb, kFinThreads, 0, st>>>(w, c, k_e2, 8);
        IQ_LAUNCH_CHECK();
        k_bnb_fin2c<<<fb, kFinThreads, 0, st>>>(w, c, 8, s_e_out);
        IQ_LAUNCH_CHECK();
        const int tb3 = (int)(((int64_t)c * kTab3 + kThreads - 1) / kThreads);
        k_bnb_tab3<<<tb3 < 152 * 4 ? tb3 : 152 * 4, kThreads, 0, st>>>(gamma, c, k_e2, 8, w);
        IQ_LAUNCH_CHECK();
        kt_pre(st);
        if (c % 16 == 0) {
            static bool attr = false;
            const int smem = 64 * kTab3P;
            if (!attr) {
                IQ_CUDA_CHECK(cudaFuncSetAttribute(k_bnb_p3w, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   smem));
                attr = true;
            }
            const int bx = (c + 63) / 64;
            int64_t by3 = (m + 63) / 64;
            const int64_t cap3 = (152 * 8 + bx - 1) / bx;
            if (by3 > cap3) by3 = cap3;
            if (by3 > 65535) by3 = 65535;
            k_bnb_p3w<<<dim3((unsigned)bx, (unsigned)by3), kThreads, smem, st>>>(e_a, a, xhat, m, c,
                                                                                 w, e);
        } else {
            RowGrid rt = row_grid(m, c / 4, 152 * 8, kTabCG);
            k_bnb_pass3<<<rt.grid, kThreads, 0, st>>>(e_a, a, xhat, m, c, rt.cg, w, e);
        }
        IQ_LAUNCH_CHECK();
        kt_post_bytes(st, IQ_KERNEL_BNB_PASS3, 5.0 * (double)m * c);
        if (e_f16) {
            iq_status r = codes_to_f16(e, (__half*)e_f16, m * (int64_t)c, st);
            if (r != IQ_OK) return r;
        }
    }
    if (dgamma)
        IQ_CUDA_CHECK(cudaMemcpyAsync(dgamma, w.sg, sizeof(int64_t) * c, cudaMemcpyDeviceToDevice, st));
    if (dbeta)
        IQ_CUDA_CHECK(cudaMemcpyAsync(dbeta, w.sb, sizeof(int64_t) * c, cudaMemcpyDeviceToDevice, st));
    return IQ_OK;
}

// ==================================================================== no-allocation variant
// For callers that may not allocate device memory themselves -- for example a plugin
// running inside a host application that owns every device allocation, or a real-time
// loop that must not allocate once it has started.  The scratch space lives in a
// fixed-size file-scope device array instead of a caller-provided workspace.

namespace {

constexpr int32_t kBnNoAllocMaxC = 4096;          // largest channel count it accepts
constexpr size_t kBnNoAllocBytes = 320 * 1024;    // scratch for up to kBnNoAllocMaxC channels

static __device__ __align__(256) unsigned char g_bn_noalloc_scratch[kBnNoAllocBytes];

}  // namespace

extern "C" iq_status iq_bn_int_fwd_noalloc(const int32_t* acc, int64_t m, int32_t c,
                                           const double* s_acc, const int32_t* gamma,
                                           const int32_t* beta, const iq_bn_bits* bits,
                                           int16_t* xhat, int8_t* a, double* s_a,
                                           int32_t* bn_codes, double* bn_scales,
                                           int64_t* bn_fixed, iq_stream stream) {
    if (c > kBnNoAllocMaxC || bn_fwd_ws_bytes(c > 0 ? c : 1) > kBnNoAllocBytes)
        return IQ_ERR_UNSUPPORTED;
    // The host-side name of the array is not a device address.  Its device address belongs
    // to the CUDA context that is current now (the primary context of the current device for
    // runtime-API callers, or a context the host application made current itself), and it
    // changes when that context is destroyed and another one created.  So it is looked up on
    // every call, in the current context -- a host-side table lookup, no device work.
    void* ws = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ws, g_bn_noalloc_scratch);
    if (e != cudaSuccess || !ws) return IQ_ERR_CUDA;
    // the statistics in the scratch are re-initialised by every call (zero sums,
    // min/max sentinels) before they are accumulated
    return iq_bn_int_fwd(acc, m, c, s_acc, gamma, beta, bits, xhat, a, s_a, bn_codes, bn_scales,
                         bn_fixed, ws, kBnNoAllocBytes, stream);
}

// ---------------------------------------------------------------- parameter update

namespace iq {
namespace {

// The whole parameter update of one L1BN layer in one launch: block 0 updates gamma (gradient
// scale s_e s_X, Philox tag 1), block 1 beta (scale s_e, tag 2).  Each block takes M = max |d|
// of its c sums, quantizes them by RQ to 8 bits with GQ1's scale (s M) 2^-7, then updates
// the x2-grid masters and codes; the same steps as requantize + update, one element per
// thread (c <= 4096).
__global__ void __launch_bounds__(1024) k_bn_update_fused(int32_t* __restrict__ gmaster,
                                                          int32_t* __restrict__ bmaster,
                                                          int32_t* __restrict__ gcodes,
                                                          int32_t* __restrict__ bcodes,
                                                          const int64_t* __restrict__ dgam,
                                                          const int64_t* __restrict__ dbet,
                                                          const double* __restrict__ s_e,
                                                          const double* __restrict__ bn_scales,
                                                          int32_t c, int sh, int k_u, int kg,
                                                          int kb, uint64_t seed, uint64_t layer,
                                                          uint64_t step,
                                                          const unsigned long long* __restrict__ epoch) {
    __shared__ unsigned long long red[32];
    const int b = blockIdx.x;
    const int64_t* d = b ? dbet : dgam;
    int32_t* master = b ? bmaster : gmaster;
    int32_t* codes = b ? bcodes : gcodes;
    const int kw = b ? kb : kg;
    const uint64_t tag = (uint64_t)b + 1;
    uint64_t m = 0;
    for (int i = threadIdx.x; i < c; i += blockDim.x) {
        const int64_t v = d[i];
        const uint64_t a = (uint64_t)(v < 0 ? -v : v);
        m = a > m ? a : m;
    }
    m = warp_max_u64(m);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x < 32) {
        uint64_t r = threadIdx.x < (blockDim.x + 31) / 32 ? red[threadIdx.x] : 0;
        r = warp_max_u64(r);
        if (threadIdx.x == 0) red[0] = r;
    }
    __syncthreads();
    const uint64_t M = red[0];
    const double s_in = b ? *s_e : __dmul_rn(*s_e, bn_scales[IQ_BN_S_XHAT]);
    // GQ1 scale (s M) 2^(1-k), k = 8
    const double s_g = M ? ldexp(__dmul_rn(s_in, (double)M), -7) : ldexp(s_in, -7);
    const UDiv div = make_udiv(M ? M : 1);
    const double p2 = ldexp(1.0, sh);
    const int64_t lu = qmax(k_u), lw = qmax(kw);
    const int dsh = k_u - kw;
    for (int i = threadIdx.x; i < c; i += blockDim.x) {
        int64_t q = 0;
        if (M) {
            uint64_t w[4];
            philox4x64_10((uint64_t)(i / 8), step, tag, *epoch, seed, layer, w);
            const int j = i & 7;
            const uint32_t u = (j & 1) ? (uint32_t)(w[j >> 1] >> 32) : (uint32_t)w[j >> 1];
            q = rq_code(d[i], M, div, 8, u);
        }
        const int64_t du = code_of(__dmul_rn(__dmul_rn((double)q, s_g), p2), k_u);
        const int64_t nm = clamp64((int64_t)master[i] - du, -lu, lu);
        master[i] = (int32_t)nm;
        codes[i] = (int32_t)clamp64((nm + (int64_t(1) << (dsh - 1))) >> dsh, -lw, lw);
    }
}

}  // namespace
}  // namespace iq

extern "C" iq_status iq_bn_update(int32_t* gamma_master, int32_t* beta_master, int32_t* gamma,
                                  int32_t* beta, const int64_t* dgamma, const int64_t* dbeta,
                                  const double* s_e, const double* bn_scales, int32_t c,
                                  const iq_bn_bits* bits, int lr_log2, int k_u, uint64_t seed,
                                  uint64_t layer, uint64_t step, void* ws, size_t ws_bytes,
                                  iq_stream stream) {
    using namespace iq;
    if (!gamma_master || !beta_master || !gamma || !beta || !dgamma || !dbeta || !s_e ||
        !bn_scales || c < 1)
        return IQ_ERR_INVALID_ARG;
    const iq_bn_bits b = bn_bits_or_default(bits);
    if (!bn_bits_valid(b) || k_u <= b.k_gamma || k_u <= b.k_beta || k_u > 31) return IQ_ERR_INVALID_ARG;
    if (lr_log2 < 0 || lr_log2 > 60) return IQ_ERR_INVALID_ARG;
    (void)ws;        // reserved: the update needs no scratch (NULL and any size accepted)
    (void)ws_bytes;
    if (c > 4096) return IQ_ERR_UNSUPPORTED;
    cudaStream_t st = (cudaStream_t)stream;
    const int sh = (k_u - 2) - lr_log2;
    const unsigned long long* ep = rq_epoch_ptr();
    if (!ep) return IQ_ERR_CUDA;
    k_bn_update_fused<<<2, 1024, 0, st>>>(gamma_master, beta_master, gamma, beta, dgamma, dbeta,
                                          s_e, bn_scales, c, sh, k_u, b.k_gamma, b.k_beta, seed,
                                          layer, step, ep);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}
