// iq_conv_tc.cu -- the 8-bit convolutions on the 5th-generation tensor cores (tcgen05).
//
// sm_103a has no integer UMMA (`tcgen05.mma .kind::i8` is rejected for this target), so
// the codes travel as fp16 "carriers": every int8 code is exact in fp16, every product
// |a b| <= 127^2 is exact, and fp32 accumulation of at most 1024 such products stays
// below 2^24 and is therefore exact.  The K loop is cut into chunks of 16 k-blocks
// (1024 products); the epilogue folds every fp32 chunk into an int32 running sum (in TMEM
// or in registers), so the result is the exact integer convolution.
//
// GEMM views of the three convolutions:
//   FWD   (forward, and the stride-1 data gradient as a forward pass over the errors with
//          flipped, transposed weights): D[M x N] = A[M x K] B[N x K]^T, M = output pixels,
//          N = output channels, K = taps x channels, both operands K-major.
//   WGRAD (weight gradient): D[Kout x RSC] = sum over pixels of E^T X, both operands
//          MN-major (channels contiguous), the pixel sum split across CTAs.
// Four persistent kernels (one CTA per SM, tiles 128 x BN x 64, BN in {64, 128, 256}):
//   k_conv_tct  all operands by TMA from fp16 carrier copies (a pre-pass widens the codes
//               once per call): 4-D boxes of the input per tap for FWD, error rectangles
//               and im2col boxes for WGRAD.  The default whenever the shape allows it; its
//               FWD epilogue writes the int32 output through TMA stores.
//   k_conv_tcc  FWD with at most 128 output channels, channel-major (M = output channels,
//               N = 256 pixels), the same TMA loads.
//   k_conv_tcq  FWD with whole 64-channel k-blocks when no TMA tile rectangle fits well:
//               producer threads copy int8 rows with cp.async and widen them in shared memory.
//   k_conv_tcp  everything else (channel counts that are multiples of 8 or 16): producer
//               warps gather int8 rows into registers and widen them on the way to shared
//               memory.
// In all of them one thread (in k_conv_tct / k_conv_tcc: one lane elected in a converged
// warp) issues tcgen05.mma (M=128, K=16) into TMEM, and epilogue warps fold the fp32 chunks
// into int32 and write either int32 outputs plus per-channel statistics (FWD; which ones
// the caller reads, TcP::st_mask), int32 split partials or int64 atomic adds (WGRAD).
// Every mbarrier wait is bounded (about one second); on expiry the CTA records a code in
// the device's sticky status word, drains what it issued and returns, and every later
// launch exits at once until the host reads the status (iq_device_status).
#include "iq_conv_tc.cuh"

#include <algorithm>
#include "iq_tc_ptx.cuh"

#include <climits>
#include <cstring>
#include <cudaTypedefs.h>
#include <mutex>

namespace iq {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;                    // fp16 elements per k-block = 128 bytes
constexpr int STAGES = 4;
constexpr int CHUNK_KB = 16;              // 1024 products per fp32 chunk
constexpr int A_BYTES = BM * 128;         // 16 KB

// Per N-tile width: B tile bytes, stage bytes, TMEM columns (fp32 chunk + int32 running
// sum), dynamic shared memory, epilogue tile pitch.
template <int BN>
struct Cfg {
    static constexpr int B_BYTES = BN * 128;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int TMEM_COLS = 2 * BN;
    static constexpr int SMEM = STAGES * STAGE_BYTES + 1024 + 256;
};

enum { MODE_FWD = 0, MODE_WGRAD = 1 };
enum { OUT_STATS = 0, OUT_ATOMIC64 = 1, OUT_PART32 = 2 };
// the column sums of 32 rows fit one 32-bit warp reduction (R S C <= 4095: 32 4095 128^2 < 2^31)
constexpr int ST_SUM32 = 4;
// only the extremes over the whole output are read (SQ without batch norm): the kernel keeps
// per-thread extremes and writes them to channel 0 once per warp
constexpr int ST_GMAX = 8;
// no extremes at all (TC_STATS_NOEXT: batch norm's deviation pass takes them)
constexpr int ST_NOEXT = (int)TC_STATS_NOEXT;

struct TcP {
    int mode, out;
    int st_mask;     // OUT_STATS: TC_STATS_SUM / TC_STATS_LO wanted, ST_SUM32, ST_GMAX
    int tma_out;     // all-TMA forward: the int32 output leaves through TMA stores (map omap)
    // geometry of the convolution whose operands are gathered
    int N, H, W, C, K, R, S, sh, sw, ph, pw, dh, dw, P, Q;
    int cstride;     // FWD: channel stride of x (>= C) and channel offset of the slice
    int cofs;
    int64_t M;       // GEMM rows
    int ncols;       // GEMM columns
    int kdim, kpad;  // FWD: R*S*C and rounded to 64
    int tap_mode;    // FWD: C % 64 == 0
    int nkb_total;   // k-blocks of the whole reduction
    int kb_per_split;
    int64_t npq;     // WGRAD: reduction length N*P*Q
    int slices;      // FWD on the all-TMA kernel: reduction slices (channel ranges of C
    int slice_rows;  // channels each) run as separate tiles; weight rows per slice
    int skip_taps;   // rectangle kernels: a tile skips the taps whose input box lies wholly
                     // outside the image (their A tiles would be all zero fill): the row taps
    uint32_t band_r[64];   // that meet the image for tile row band pt (bit r), the column
    uint32_t band_s[64];   // taps for column band qt (bit s)
};

// ---------------------------------------------------------------- FWD gather (K-major A)

__device__ __forceinline__ void gather_fwd(const TcP& p, const int8_t* __restrict__ x, bool valid,
                                           int n, int pp, int qq, int kb, uint32_t (&w)[16]) {
#pragma unroll
    for (int i = 0; i < 16; i++) w[i] = 0;
    if (!valid || kb >= p.nkb_total) return;
    const int kpos = kb * BK;
    if (p.tap_mode) {
        const int tap = kpos / p.C;
        const int c0 = kpos - tap * p.C;
        const int r = tap / p.S, s = tap - r * p.S;
        const int hh = pp * p.sh + r * p.dh - p.ph;
        const int ww = qq * p.sw + s * p.dw - p.pw;
        if (hh < 0 || hh >= p.H || ww < 0 || ww >= p.W) return;
        const uint4* src = reinterpret_cast<const uint4*>(
            x + (((int64_t)n * p.H + hh) * p.W + ww) * p.cstride + p.cofs + c0);
#pragma unroll
        for (int i = 0; i < 4; i++) {
            uint4 v = __ldg(src + i);
            w[4 * i + 0] = v.x; w[4 * i + 1] = v.y; w[4 * i + 2] = v.z; w[4 * i + 3] = v.w;
        }
    } else {
        int tap = kpos / p.C;
        int c = kpos - tap * p.C;
#pragma unroll
        for (int i = 0; i < 16; i++) {
            if (kpos + 4 * i < p.kdim) {
                const int r = tap / p.S, s = tap - (tap / p.S) * p.S;
                const int hh = pp * p.sh + r * p.dh - p.ph;
                const int ww = qq * p.sw + s * p.dw - p.pw;
                if (hh >= 0 && hh < p.H && ww >= 0 && ww < p.W)
                    w[i] = __ldg(reinterpret_cast<const uint32_t*>(
                        x + (((int64_t)n * p.H + hh) * p.W + ww) * p.cstride + p.cofs + c));
            }
            c += 4;
            if (c == p.C) { c = 0; tap++; }
        }
    }
}

// K-major 128-byte-swizzled row store of 64 fp16 (from 64 int8 codes)
__device__ __forceinline__ void store_kmajor_row(uint8_t* tile, int row, const uint32_t (&w)[16]) {
    uint8_t* dst = tile + row * 128;
#pragma unroll
    for (int j = 0; j < 8; j++) {
        uint32_t o0, o1, o2, o3;
        tc::i8x4_to_f16x4(w[2 * j], o0, o1);
        tc::i8x4_to_f16x4(w[2 * j + 1], o2, o3);
        *reinterpret_cast<uint4*>(dst + ((j ^ (row & 7)) << 4)) = make_uint4(o0, o1, o2, o3);
    }
}

// ---------------------------------------------------------------- WGRAD gather (MN-major)
// Thread t of the producers owns reduction row j = t/2 of the k-block and half h = t%2:
// A chunks (16 channels each) 4h..4h+3 of E[npq][m0 + 0..127] and B blocks 2h, 2h+1
// (64 consecutive RSC columns each, inside one tap since C % 64 == 0).

struct WgRow {
    bool valid;
    int n, pp, qq;
};

__device__ __forceinline__ WgRow wg_row(const TcP& p, int64_t j) {
    WgRow r;
    r.valid = j < p.npq;
    r.n = r.pp = r.qq = 0;
    if (r.valid) {
        const int64_t pq = (int64_t)p.P * p.Q;
        r.n = (int)(j / pq);
        const int64_t rem = j - (int64_t)r.n * pq;
        r.pp = (int)(rem / p.Q);
        r.qq = (int)(rem - (int64_t)r.pp * p.Q);
    }
    return r;
}

template <int BN>
__device__ __forceinline__ void gather_wgrad(const TcP& p, const int8_t* __restrict__ e,
                                             const int8_t* __restrict__ x, int64_t m0, int n0,
                                             const WgRow& rw, int h, uint4 (&a)[4],
                                             uint4 (&b)[BN / 32]) {
#pragma unroll
    for (int i = 0; i < 4; i++) a[i] = make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int i = 0; i < BN / 32; i++) b[i] = make_uint4(0, 0, 0, 0);
    if (!rw.valid) return;
    const int64_t pix = ((int64_t)rw.n * p.P + rw.pp) * p.Q + rw.qq;
    // A: E[pix][m0 + 64h .. m0 + 64h + 63]; K_out % 16 == 0 so a chunk is all in or all out
    const int8_t* erow = e + pix * p.K;
#pragma unroll
    for (int i = 0; i < 4; i++) {
        const int64_t m = m0 + 64 * h + 16 * i;
        if (m < p.M) a[i] = __ldg(reinterpret_cast<const uint4*>(erow + m));
    }
    // B: 16-column chunks h*BN/32 .. (h+1)*BN/32 - 1 of the RSC columns.  With C % 64 == 0
    // a run of 4 chunks (64 columns) lies inside one tap and is decoded once; otherwise
    // (C % 16 == 0) every chunk is decoded on its own.
    if (p.C % 64 == 0) {
#pragma unroll
        for (int i0 = 0; i0 < BN / 32; i0 += 4) {
            const int col = n0 + 16 * (h * (BN / 32) + i0);
            if (col >= p.ncols) continue;
            const int tap = col / p.C;
            const int c0 = col - tap * p.C;
            const int r = tap / p.S, s = tap - r * p.S;
            const int hh = rw.pp * p.sh + r * p.dh - p.ph;
            const int ww = rw.qq * p.sw + s * p.dw - p.pw;
            if (hh < 0 || hh >= p.H || ww < 0 || ww >= p.W) continue;
            const uint4* src = reinterpret_cast<const uint4*>(
                x + (((int64_t)rw.n * p.H + hh) * p.W + ww) * p.C + c0);
#pragma unroll
            for (int i = 0; i < 4 && i0 + i < BN / 32; i++) b[i0 + i] = __ldg(src + i);
        }
        return;
    }
#pragma unroll
    for (int i = 0; i < BN / 32; i++) {
        const int col = n0 + 16 * (h * (BN / 32) + i);
        if (col >= p.ncols) continue;
        const int tap = col / p.C;
        const int c0 = col - tap * p.C;
        const int r = tap / p.S, s = tap - r * p.S;
        const int hh = rw.pp * p.sh + r * p.dh - p.ph;
        const int ww = rw.qq * p.sw + s * p.dw - p.pw;
        if (hh < 0 || hh >= p.H || ww < 0 || ww >= p.W) continue;
        b[i] = __ldg(reinterpret_cast<const uint4*>(
            x + (((int64_t)rw.n * p.H + hh) * p.W + ww) * p.C + c0));
    }
}

// MN-major 128-byte-swizzled layout: atoms of 8 K-rows x 64 MN-elements (1024 bytes);
// K-groups of 8 rows at stride 1024 (SBO), 64-wide MN blocks at stride 8192 (LBO).
__device__ __forceinline__ void store_mnmajor_chunk(uint8_t* tile, int j, int mchunk,
                                                    uint32_t w0, uint32_t w1, uint32_t w2,
                                                    uint32_t w3) {
    // mchunk indexes 16-element groups along MN; 16 int8 -> 2 x 16-byte fp16 chunks
    const int mb = mchunk >> 2;                 // 64-element block
    const int c8 = (mchunk & 3) * 2;            // first 8-element chunk within the 128-byte row
    uint8_t* atom = tile + mb * 8192 + (j >> 3) * 1024 + (j & 7) * 128;
    uint32_t o0, o1, o2, o3, o4, o5, o6, o7;
    tc::i8x4_to_f16x4(w0, o0, o1);
    tc::i8x4_to_f16x4(w1, o2, o3);
    tc::i8x4_to_f16x4(w2, o4, o5);
    tc::i8x4_to_f16x4(w3, o6, o7);
    *reinterpret_cast<uint4*>(atom + ((c8 ^ (j & 7)) << 4)) = make_uint4(o0, o1, o2, o3);
    *reinterpret_cast<uint4*>(atom + (((c8 + 1) ^ (j & 7)) << 4)) = make_uint4(o4, o5, o6, o7);
}

__device__ __forceinline__ uint64_t sdesc_mnmajor_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFF);
    d |= (uint64_t)(8192 >> 4) << 16;   // LBO: stride between 64-element MN blocks
    d |= (uint64_t)(1024 >> 4) << 32;   // SBO: stride between 8-row K groups
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

__host__ __device__ constexpr uint32_t idesc_f16(int M, int N, bool mn_major) {
    return (1u << 4) | ((mn_major ? 1u : 0u) << 15) | ((mn_major ? 1u : 0u) << 16) |
           ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// ---------------------------------------------------------------- persistent kernel
// One CTA per SM walks a strided list of output tiles (m-tile fastest, then n-tile, then
// K split) as one flat stream of k-blocks, so the producers run ahead across tile
// boundaries.  Warps 0-3 gather A (and for WGRAD B), thread 0 issues the B TMA loads;
// warp 12 issues the MMAs into one fp32 accumulator (TMEM columns [0, BN)); warps 4-11
// fold every finished fp32 chunk into the int32 running sum (columns [BN, 2 BN)), each
// warpgroup one half of the columns, and release the accumulator at once.  After a tile's
// last fold they read the int32 sums back and write the output while the MMAs of the next
// tile already run; the next tile's first fold overwrites the sums in the same threads'
// program order, so no further handshake is needed.

constexpr int THREADS_P = 416;

struct BarsP {
    uint64_t full_a[STAGES];
    uint64_t full_b[STAGES];
    uint64_t empty[STAGES];
    uint64_t accf;
    uint64_t acce;
    uint64_t done;
    uint32_t tmem_base;
    int abort;
    int never;
};

struct TileGrid {
    int mt, nt, ns;      // m-tiles, n-tiles, splits
    int total;
};

// k-block position in a CTA's stream of (tile, kb) pairs
struct Pos {
    int tile;            // linear tile index, >= total when past the end
    int kb;              // k-block within the tile
    int nkb;             // k-blocks of this tile
    int64_t m0;
    int n0, kb0;
};

__device__ __forceinline__ void pos_set_tile(Pos& q, int tile, const TcP& p, const TileGrid& g,
                                             int BN) {
    q.tile = tile;
    q.kb = 0;
    q.nkb = 0;
    if (tile >= g.total) return;
    const int mt = tile % g.mt;
    const int rest = tile / g.mt;
    const int nt = rest % g.nt;
    const int sp = rest / g.nt;
    q.m0 = (int64_t)mt * BM;
    q.n0 = nt * BN;
    q.kb0 = sp * p.kb_per_split;
    int n = p.nkb_total - q.kb0;
    q.nkb = n > p.kb_per_split ? p.kb_per_split : n;
}

__device__ __forceinline__ void pos_next(Pos& q, const TcP& p, const TileGrid& g, int BN) {
    if (q.tile >= g.total) return;
    if (++q.kb >= q.nkb) pos_set_tile(q, q.tile + gridDim.x, p, g, BN);
}

// output-pixel coordinates of one producer row, recomputed only when the tile changes
struct RowCache {
    int tile;
    bool valid;
    int n, pp, qq;
};

__device__ __forceinline__ void gather_fwd_pos(const TcP& p, const int8_t* __restrict__ x,
                                               const Pos& q, int row, RowCache& rc,
                                               uint32_t (&w)[16]) {
    if (rc.tile != q.tile) {
        rc.tile = q.tile;
        const int64_t m = q.m0 + row;
        rc.valid = q.nkb > 0 && m < p.M;
        rc.n = rc.pp = rc.qq = 0;
        if (rc.valid) {
            const int64_t pq = (int64_t)p.P * p.Q;
            rc.n = (int)(m / pq);
            const int64_t rem = m - (int64_t)rc.n * pq;
            rc.pp = (int)(rem / p.Q);
            rc.qq = (int)(rem - (int64_t)rc.pp * p.Q);
        }
    }
    gather_fwd(p, x, rc.valid, rc.n, rc.pp, rc.qq, q.kb0 + q.kb, w);
}

// fold the fp32 chunk into the int32 sums of this warpgroup's BN/2 columns
template <int BN>
__device__ __forceinline__ void fold_half(uint32_t tD, uint32_t tR, bool has_prev) {
#pragma unroll 1
    for (int cb = 0; cb < BN / 2; cb += 32) {
        uint32_t d0[32], r0[32];
        tc::tmem_ld_32x32b_x32(tD + cb, d0);
        if (has_prev) tc::tmem_ld_32x32b_x32(tR + cb, r0);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; i++)
            r0[i] = (uint32_t)((has_prev ? (int)r0[i] : 0) + __float2int_rn(__uint_as_float(d0[i])));
        tc::tmem_st_32x32b_x32(tR + cb, r0);
    }
    tc::tmem_st_wait();
}

template <int BN>
__device__ __forceinline__ void write_half(const TcP& p, uint32_t tR, int64_t m0, int n0, int row,
                                           int lane, int32_t* __restrict__ out32,
                                           long long* __restrict__ out64,
                                           unsigned long long* __restrict__ s1,
                                           int* __restrict__ hi_c, int* __restrict__ lo_c) {
    const int64_t m = m0 + row;
    const bool valid = m < p.M;
    const bool any = __any_sync(0xffffffffu, valid);
#pragma unroll 1
    for (int cb = 0; cb < BN / 2; cb += 32) {
        uint32_t r[32];
        tc::tmem_ld_32x32b_x32(tR + cb, r);
        tc::tmem_ld_wait();
        if (!any) continue;
        const int gc0 = n0 + cb;          // first global column of this block
        if (p.out == OUT_STATS) {
            if (valid) {
                int32_t* dst = out32 + m * p.ncols + gc0;
#pragma unroll
                for (int i = 0; i < 8; i++)
                    if (gc0 + 4 * i < p.ncols)
                        reinterpret_cast<int4*>(dst)[i] =
                            make_int4((int)r[4 * i], (int)r[4 * i + 1], (int)r[4 * i + 2],
                                      (int)r[4 * i + 3]);
            }
            long long my_sum = 0;
            int my_hi = INT_MIN, my_lo = INT_MAX;
#pragma unroll
            for (int j = 0; j < 32; j++) {
                const int v = (int)r[j];
                const int vh = valid ? v : INT_MIN, vl = valid ? v : INT_MAX;
                const unsigned lo16 = valid ? ((unsigned)v & 0xffffu) : 0u;
                const int hi16 = valid ? (v >> 16) : 0;
                const int mx = __reduce_max_sync(0xffffffffu, vh);
                const int mn = __reduce_min_sync(0xffffffffu, vl);
                const unsigned sl = __reduce_add_sync(0xffffffffu, lo16);
                const int sh = __reduce_add_sync(0xffffffffu, hi16);
                if (lane == j) {
                    my_hi = mx;
                    my_lo = mn;
                    my_sum = (long long)sh * 65536 + (long long)sl;
                }
            }
            const int gcol = gc0 + lane;
            if (gcol < p.ncols) {
                atomicAdd(&s1[gcol], (unsigned long long)my_sum);
                atomicMax(&hi_c[gcol], my_hi);
                atomicMin(&lo_c[gcol], my_lo);
            }
        } else if (valid) {
            long long* dst = out64 + m * p.ncols + gc0;
#pragma unroll
            for (int j = 0; j < 32; j++)
                if ((int)r[j] != 0 && gc0 + j < p.ncols)
                    atomicAdd(reinterpret_cast<unsigned long long*>(dst + j),
                              (unsigned long long)(long long)(int)r[j]);
        }
    }
}

template <int BN>
__global__ void __launch_bounds__(THREADS_P, 1)
    k_conv_tcp(const __grid_constant__ CUtensorMap wmap, TcP p, TileGrid g,
               const int8_t* __restrict__ xa, const int8_t* __restrict__ xb,
               int32_t* __restrict__ out32, long long* __restrict__ out64,
               unsigned long long* __restrict__ s1, int* __restrict__ hi_c,
               int* __restrict__ lo_c, int* __restrict__ err) {
    constexpr int STAGE_BYTES = Cfg<BN>::STAGE_BYTES;
    constexpr int B_BYTES = Cfg<BN>::B_BYTES;
    constexpr int TMEM_COLS = Cfg<BN>::TMEM_COLS;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    BarsP* bars = reinterpret_cast<BarsP*>(smem + STAGES * STAGE_BYTES);

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    if (__syncthreads_or(tid == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    if ((int)blockIdx.x >= g.total) return;
    const bool wg = p.mode == MODE_WGRAD;

    if (tid == 0) {
        for (int s = 0; s < STAGES; s++) {
            tc::mbar_init(&bars->full_a[s], 128);
            tc::mbar_init(&bars->full_b[s], 1);
            tc::mbar_init(&bars->empty[s], 1);
        }
        tc::mbar_init(&bars->accf, 1);
        tc::mbar_init(&bars->acce, 256);
        tc::mbar_init(&bars->done, 1);
        bars->abort = 0;
        bars->never = 0;
        tc::mbar_fence_init();
        if (!wg) tc::tma_prefetch_desc(&wmap);
    }
    if (warp == 12) {
        tc::tmem_alloc(&bars->tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort_flag = &bars->abort;

    if (warp < 4) {
        // ================================================ producers
        Pos cur, p1, p2;
        pos_set_tile(cur, blockIdx.x, p, g, BN);
        p1 = cur;
        pos_next(p1, p, g, BN);
        p2 = p1;
        pos_next(p2, p, g, BN);
        int issued_b = 0;
        uint32_t kbc = 0;
        if (!wg) {
            const int row = tid;
            uint32_t c0[16], c1[16], c2[16];
            RowCache rc;
            rc.tile = -1;
            gather_fwd_pos(p, xa, cur, row, rc, c0);
            gather_fwd_pos(p, xa, p1, row, rc, c1);
            while (cur.tile < g.total) {
                const int s = kbc % STAGES;
                const uint32_t it = kbc / STAGES;
                if (!tc::mbar_wait(&bars->empty[s], (it & 1) ^ 1, abort_flag)) {
                    bars->abort = 1;
                    atomicExch(err, 1);
                    break;
                }
                uint8_t* a_tile = smem + s * STAGE_BYTES;
                if (tid == 0) {
                    tc::mbar_expect_tx(&bars->full_b[s], B_BYTES);
                    tc::tma_load_2d(a_tile + A_BYTES, &wmap, &bars->full_b[s],
                                    (cur.kb0 + cur.kb) * BK, cur.n0);
                    tc::mbar_arrive(&bars->full_b[s]);
                    issued_b = (int)kbc + 1;
                }
                if (p2.tile < g.total) gather_fwd_pos(p, xa, p2, row, rc, c2);
                store_kmajor_row(a_tile, row, c0);
                tc::fence_proxy_async_smem();
                tc::mbar_arrive(&bars->full_a[s]);
#pragma unroll
                for (int i = 0; i < 16; i++) { c0[i] = c1[i]; c1[i] = c2[i]; }
                cur = p1;
                p1 = p2;
                pos_next(p2, p, g, BN);
                kbc++;
            }
        } else {
            const int j = tid >> 1, h = tid & 1;
            uint4 a0[4], b0[BN / 32], a1[4], b1[BN / 32];
            {
                WgRow r0 = wg_row(p, (int64_t)(cur.kb0 + cur.kb) * BK + j);
                gather_wgrad<BN>(p, xa, xb, cur.m0, cur.n0, r0, h, a0, b0);
            }
            while (cur.tile < g.total) {
                const int s = kbc % STAGES;
                const uint32_t it = kbc / STAGES;
                if (p1.tile < g.total) {
                    WgRow r1 = wg_row(p, (int64_t)(p1.kb0 + p1.kb) * BK + j);
                    gather_wgrad<BN>(p, xa, xb, p1.m0, p1.n0, r1, h, a1, b1);
                }
                if (!tc::mbar_wait(&bars->empty[s], (it & 1) ^ 1, abort_flag)) {
                    bars->abort = 1;
                    atomicExch(err, 1);
                    break;
                }
                uint8_t* a_tile = smem + s * STAGE_BYTES;
                uint8_t* b_tile = a_tile + A_BYTES;
#pragma unroll
                for (int i = 0; i < 4; i++)
                    store_mnmajor_chunk(a_tile, j, 4 * h + i, a0[i].x, a0[i].y, a0[i].z, a0[i].w);
#pragma unroll
                for (int i = 0; i < BN / 32; i++)
                    store_mnmajor_chunk(b_tile, j, h * (BN / 32) + i, b0[i].x, b0[i].y, b0[i].z,
                                        b0[i].w);
                tc::fence_proxy_async_smem();
                tc::mbar_arrive(&bars->full_a[s]);
                if (tid == 0) tc::mbar_arrive(&bars->full_b[s]);
#pragma unroll
                for (int i = 0; i < 4; i++) a0[i] = a1[i];
#pragma unroll
                for (int i = 0; i < BN / 32; i++) b0[i] = b1[i];
                cur = p1;
                pos_next(p1, p, g, BN);
                kbc++;
            }
        }
        if (!wg && tid == 0 && *abort_flag) {
            for (int kb = (issued_b > STAGES ? issued_b - STAGES : 0); kb < issued_b; kb++)
                tc::mbar_wait(&bars->full_b[kb % STAGES], (uint32_t)(kb / STAGES) & 1,
                              &bars->never);
        }
    } else if (warp == 12) {
        // ================================================ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16(BM, BN, wg);
            bool ok = true;
            uint32_t kbc = 0, cc = 0;
            Pos q;
            pos_set_tile(q, blockIdx.x, p, g, BN);
            while (ok && q.tile < g.total) {
                const int s = kbc % STAGES;
                const uint32_t it = kbc / STAGES;
                const bool first = (q.kb % CHUNK_KB) == 0;
                const bool last = ((q.kb % CHUNK_KB) == CHUNK_KB - 1) || q.kb == q.nkb - 1;
                if (first && cc > 0 &&
                    !tc::mbar_wait(&bars->acce, (cc - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                if (!tc::mbar_wait(&bars->full_b[s], it & 1, abort_flag) ||
                    !tc::mbar_wait(&bars->full_a[s], it & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t a_addr = tc::smem_u32(smem + s * STAGE_BYTES);
                const uint32_t b_addr = a_addr + A_BYTES;
#pragma unroll
                for (int k = 0; k < BK / 16; k++) {
                    uint64_t ad, bd;
                    if (wg) {
                        ad = sdesc_mnmajor_sw128(a_addr + 2 * 1024 * k);
                        bd = sdesc_mnmajor_sw128(b_addr + 2 * 1024 * k);
                    } else {
                        ad = tc::sdesc_kmajor_sw128(a_addr + 32 * k);
                        bd = tc::sdesc_kmajor_sw128(b_addr + 32 * k);
                    }
                    tc::umma_f16(tmem, ad, bd, idesc, (first && k == 0) ? 0u : 1u);
                }
                tc::umma_commit(&bars->empty[s]);
                if (last) {
                    tc::umma_commit(&bars->accf);
                    cc++;
                }
                kbc++;
                pos_next(q, p, g, BN);
            }
            if (!ok) {
                bars->abort = 1;
                atomicExch(err, 2);
            }
            tc::umma_commit(&bars->done);
            tc::mbar_wait(&bars->done, 0, &bars->never);
        }
        __syncwarp();
    } else {
        // ================================================ epilogue (warps 4..11)
        const int half = (warp - 4) >> 2;                 // column half
        const int row = ((warp & 3) << 5) + lane;         // TMEM lane = tile row
        const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
        const uint32_t tD = tmem + lane_base + half * (BN / 2);
        const uint32_t tR = tmem + lane_base + BN + half * (BN / 2);
        uint32_t cc = 0;
        bool ok = true;
        Pos q;
        pos_set_tile(q, blockIdx.x, p, g, BN);
        while (ok && q.tile < g.total) {
            const int nch = (q.nkb + CHUNK_KB - 1) / CHUNK_KB;
            for (int c = 0; c < nch; c++) {
                if (!tc::mbar_wait(&bars->accf, cc & 1, abort_flag)) {
                    ok = false;
                    bars->abort = 1;
                    atomicExch(err, 3);
                    break;
                }
                tc::tc_fence_after();
                fold_half<BN>(tD, tR, c > 0);
                tc::tc_fence_before();
                tc::mbar_arrive(&bars->acce);
                cc++;
            }
            if (!ok || *abort_flag) break;
            write_half<BN>(p, tR, q.m0, q.n0 + half * (BN / 2), row, lane, out32, out64, s1, hi_c,
                           lo_c);
            pos_set_tile(q, q.tile + gridDim.x, p, g, BN);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 12) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, TMEM_COLS);
    }
}

// ---------------------------------------------------------------- persistent forward kernel
// The forward (and stride-1 data-gradient) GEMM for whole 64-channel k-blocks, persistent
// like k_conv_tcp, with the fold spread over 16 epilogue warps (4 warpgroups, each a quarter
// of the columns; warp w reads TMEM lanes 32 (w % 4) ..) so that the MMA warp waits only
// briefly per 16 k-blocks, and the epilogue sleeping between its barrier probes.  Each
// producer thread owns one A row: it copies its 64 int8 codes per k-block with cp.async
// (zero fill for padding and rows past the end) into a private slot of a ring NST_Q
// k-blocks deep, walks the taps with incremental counters (no divisions per k-block), and
// widens the k-block NST_Q - 1 behind into the fp16 stage.

constexpr int THREADS_Q = 672;       // warps 0-3 producers, 4-19 epilogue, 20 MMA
constexpr int EPI_Q = 512;
constexpr int STAGES_Q = 3;          // fp16 A + B stages
constexpr int NST_Q = 6;             // int8 staging ring depth (k-blocks)
constexpr int STG_PITCH = 80;        // bytes per staged row: 64 + 16 (conflict-free 16-B accesses)
constexpr int STG_SLOT = BM * STG_PITCH;

template <int BN>
struct CfgQ {
    static constexpr int STAGE_BYTES = Cfg<BN>::STAGE_BYTES;
    static constexpr int STG_OFF = STAGES_Q * STAGE_BYTES;
    static constexpr int BAR_OFF = STG_OFF + NST_Q * STG_SLOT;
    static constexpr int SMEM = BAR_OFF + 1024 + 256;
    static_assert(SMEM <= 232448, "shared memory");
};

struct BarsQ {
    uint64_t full_a[STAGES_Q];
    uint64_t full_b[STAGES_Q];
    uint64_t empty[STAGES_Q];
    uint64_t accf;
    uint64_t acce;
    uint64_t done;
    uint32_t tmem_base;
    int abort;
    int never;
};

// a producer row's position in its k-block stream, with the tap counters of the k-block
struct FwdCur {
    Pos q;
    bool valid;
    int n, pp, qq;
    int r, s, c0;      // tap mode: tap (r, s) and first channel of the k-block
};

__device__ __forceinline__ void fcur_tile(FwdCur& f, int tile, const TcP& p, const TileGrid& g,
                                          int BN, int row) {
    pos_set_tile(f.q, tile, p, g, BN);
    f.valid = false;
    f.n = f.pp = f.qq = 0;
    f.r = f.s = f.c0 = 0;
    if (f.q.tile >= g.total) return;
    const int64_t m = f.q.m0 + row;
    f.valid = m < p.M;
    if (f.valid) {
        const int64_t pq = (int64_t)p.P * p.Q;
        f.n = (int)(m / pq);
        const int64_t rem = m - (int64_t)f.n * pq;
        f.pp = (int)(rem / p.Q);
        f.qq = (int)(rem - (int64_t)f.pp * p.Q);
    }
    if (p.tap_mode) {
        const int kpos = f.q.kb0 * BK;
        const int tap = kpos / p.C;
        f.c0 = kpos - tap * p.C;
        f.r = tap / p.S;
        f.s = tap - f.r * p.S;
    }
}

__device__ __forceinline__ void fcur_next(FwdCur& f, const TcP& p, const TileGrid& g, int BN,
                                          int row) {
    if (f.q.tile >= g.total) return;
    if (++f.q.kb >= f.q.nkb) {
        fcur_tile(f, f.q.tile + gridDim.x, p, g, BN, row);
        return;
    }
    if (p.tap_mode) {
        f.c0 += BK;
        if (f.c0 >= p.C) {
            f.c0 = 0;
            if (++f.s == p.S) {
                f.s = 0;
                f.r++;
            }
        }
    }
}

// cp.async of this row's 64 codes of the cursor's k-block into a staging slot (tap mode)
__device__ __forceinline__ void fcur_copy(const TcP& p, const int8_t* __restrict__ x,
                                          const FwdCur& f, uint32_t dst) {
    const int hh = f.pp * p.sh + f.r * p.dh - p.ph;
    const int ww = f.qq * p.sw + f.s * p.dw - p.pw;
    const bool in = f.valid && f.q.nkb > 0 && hh >= 0 && hh < p.H && ww >= 0 && ww < p.W;
    const int8_t* src = in ? x + (((int64_t)f.n * p.H + hh) * p.W + ww) * p.cstride + p.cofs + f.c0
                           : x;
    const uint32_t nb = in ? 16u : 0u;
#pragma unroll
    for (int i = 0; i < 4; i++) tc::cp_async16(dst + 16 * i, src + 16 * i, nb);
}

// the output of 32 columns of one warpgroup's quarter: int32 stores and per-channel
// statistics (OUT_STATS) or int64 atomic adds
template <int CW>
__device__ __forceinline__ void write_quarter(const TcP& p, const int (&sum)[CW], int64_t m0,
                                              int c0, int row, int lane,
                                              int32_t* __restrict__ out32,
                                              long long* __restrict__ out64,
                                              unsigned long long* __restrict__ s1,
                                              int* __restrict__ hi_c, int* __restrict__ lo_c) {
    const int64_t m = m0 + row;
    const bool valid = m < p.M;
    if (p.out == OUT_STATS) {
        if (valid) {
            int32_t* dst = out32 + m * p.ncols + c0;
#pragma unroll
            for (int i = 0; i < CW / 4; i++)
                if (c0 + 4 * i < p.ncols)
                    reinterpret_cast<int4*>(dst)[i] =
                        make_int4(sum[4 * i], sum[4 * i + 1], sum[4 * i + 2], sum[4 * i + 3]);
        }
#pragma unroll
        for (int cb = 0; cb < CW; cb += 32) {
            long long my_sum = 0;
            int my_hi = INT_MIN, my_lo = INT_MAX;
#pragma unroll
            for (int j = 0; j < 32 && cb + j < CW; j++) {
                const int v = sum[cb + j];
                const int mx = __reduce_max_sync(0xffffffffu, valid ? v : INT_MIN);
                const int mn = __reduce_min_sync(0xffffffffu, valid ? v : INT_MAX);
                const unsigned sl = __reduce_add_sync(0xffffffffu, valid ? ((unsigned)v & 0xffffu) : 0u);
                const int sh = __reduce_add_sync(0xffffffffu, valid ? (v >> 16) : 0);
                if (lane == j) {
                    my_hi = mx;
                    my_lo = mn;
                    my_sum = (long long)sh * 65536 + (long long)sl;
                }
            }
            const int gcol = c0 + cb + lane;
            if (lane < CW - cb && gcol < p.ncols) {
                atomicAdd(&s1[gcol], (unsigned long long)my_sum);
                atomicMax(&hi_c[gcol], my_hi);
                atomicMin(&lo_c[gcol], my_lo);
            }
        }
    } else if (valid) {
        long long* dst = out64 + m * p.ncols + c0;
#pragma unroll
        for (int j = 0; j < CW; j++)
            if (sum[j] != 0 && c0 + j < p.ncols)
                atomicAdd(reinterpret_cast<unsigned long long*>(dst + j),
                          (unsigned long long)(long long)sum[j]);
    }
}

// TMEM loads / stores of 16 or 32 columns
template <int W>
__device__ __forceinline__ void tmem_ld_w(uint32_t a, uint32_t (&r)[W]) {
    if constexpr (W == 32) tc::tmem_ld_32x32b_x32(a, r);
    else tc::tmem_ld_32x32b_x16(a, r);
}
template <int W>
__device__ __forceinline__ void tmem_st_w(uint32_t a, const uint32_t (&r)[W]) {
    if constexpr (W == 32) tc::tmem_st_32x32b_x32(a, r);
    else tc::tmem_st_32x32b_x16(a, r);
}

template <int BN>
__global__ void __launch_bounds__(THREADS_Q, 1)
    k_conv_tcq(const __grid_constant__ CUtensorMap wmap, TcP p, TileGrid g,
               const int8_t* __restrict__ xa, int32_t* __restrict__ out32,
               long long* __restrict__ out64, unsigned long long* __restrict__ s1,
               int* __restrict__ hi_c, int* __restrict__ lo_c, int* __restrict__ err) {
    constexpr int STAGE_BYTES = CfgQ<BN>::STAGE_BYTES;
    constexpr int B_BYTES = Cfg<BN>::B_BYTES;
    constexpr int TMEM_COLS = Cfg<BN>::TMEM_COLS;     // fp32 chunk + int32 running sum
    constexpr int CW = BN / 4;                         // columns per epilogue warpgroup
    constexpr int LDW = 16;                            // columns per TMEM access
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    BarsQ* bars = reinterpret_cast<BarsQ*>(smem + CfgQ<BN>::BAR_OFF);
    uint8_t* stg = smem + CfgQ<BN>::STG_OFF;

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    if (__syncthreads_or(tid == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    if ((int)blockIdx.x >= g.total) return;

    if (tid == 0) {
        for (int s = 0; s < STAGES_Q; s++) {
            tc::mbar_init(&bars->full_a[s], 128);
            tc::mbar_init(&bars->full_b[s], 1);
            tc::mbar_init(&bars->empty[s], 1);
        }
        tc::mbar_init(&bars->accf, 1);
        tc::mbar_init(&bars->acce, EPI_Q);
        tc::mbar_init(&bars->done, 1);
        bars->abort = 0;
        bars->never = 0;
        tc::mbar_fence_init();
        tc::tma_prefetch_desc(&wmap);
    }
    if (warp == 20) {
        tc::tmem_alloc(&bars->tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort_flag = &bars->abort;

    if (warp < 4) {
        // ================================================ producers
        const int row = tid;
        const uint32_t my_stg = tc::smem_u32(stg) + row * STG_PITCH;
        FwdCur cs, cg;
        fcur_tile(cs, blockIdx.x, p, g, BN, row);
        cg = cs;
        // prologue: copies of the first NST_Q - 1 k-blocks in flight
#pragma unroll 1
        for (int i = 0; i < NST_Q - 1; i++) {
            if (cg.q.tile < g.total) fcur_copy(p, xa, cg, my_stg + i * STG_SLOT);
            tc::cp_async_commit();
            fcur_next(cg, p, g, BN, row);
        }
        uint32_t kbc = 0;
        int issued_b = 0;
        while (cs.q.tile < g.total) {
            // copy k-block kbc + NST_Q - 1, then wait until k-block kbc has landed
            if (cg.q.tile < g.total)
                fcur_copy(p, xa, cg, my_stg + ((kbc + NST_Q - 1) % NST_Q) * STG_SLOT);
            tc::cp_async_commit();
            fcur_next(cg, p, g, BN, row);
            tc::cp_async_wait<NST_Q - 1>();
            const uint8_t* src = stg + (kbc % NST_Q) * STG_SLOT + row * STG_PITCH;
            uint32_t w[16];
#pragma unroll
            for (int i = 0; i < 4; i++) {
                const uint4 v = *reinterpret_cast<const uint4*>(src + 16 * i);
                w[4 * i] = v.x; w[4 * i + 1] = v.y; w[4 * i + 2] = v.z; w[4 * i + 3] = v.w;
            }
            const int s = kbc % STAGES_Q;
            const uint32_t it = kbc / STAGES_Q;
            if (!tc::mbar_wait(&bars->empty[s], (it & 1) ^ 1, abort_flag)) {
                bars->abort = 1;
                atomicExch(err, 1);
                break;
            }
            uint8_t* a_tile = smem + s * STAGE_BYTES;
            if (tid == 0) {
                tc::mbar_expect_tx(&bars->full_b[s], B_BYTES);
                tc::tma_load_2d(a_tile + A_BYTES, &wmap, &bars->full_b[s],
                                (cs.q.kb0 + cs.q.kb) * BK, cs.q.n0);
                tc::mbar_arrive(&bars->full_b[s]);
                issued_b = (int)kbc + 1;
            }
            store_kmajor_row(a_tile, row, w);
            tc::fence_proxy_async_smem();
            tc::mbar_arrive(&bars->full_a[s]);
            fcur_next(cs, p, g, BN, row);
            kbc++;
        }
        tc::cp_async_wait<0>();
        if (tid == 0 && *abort_flag) {
            for (int kb = (issued_b > STAGES_Q ? issued_b - STAGES_Q : 0); kb < issued_b; kb++)
                tc::mbar_wait(&bars->full_b[kb % STAGES_Q], (uint32_t)(kb / STAGES_Q) & 1,
                              &bars->never);
        }
    } else if (warp == 20) {
        // ================================================ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16(BM, BN, false);
            bool ok = true;
            uint32_t kbc = 0, cc = 0;
            Pos q;
            pos_set_tile(q, blockIdx.x, p, g, BN);
            while (ok && q.tile < g.total) {
                const int s = kbc % STAGES_Q;
                const uint32_t it = kbc / STAGES_Q;
                const bool first = (q.kb % CHUNK_KB) == 0;
                const bool last = ((q.kb % CHUNK_KB) == CHUNK_KB - 1) || q.kb == q.nkb - 1;
                // the fp32 accumulator is free once the epilogue folded the previous chunk
                if (first && cc > 0 && !tc::mbar_wait(&bars->acce, (cc - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                if (!tc::mbar_wait(&bars->full_b[s], it & 1, abort_flag) ||
                    !tc::mbar_wait(&bars->full_a[s], it & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t a_addr = tc::smem_u32(smem + s * STAGE_BYTES);
                const uint32_t b_addr = a_addr + A_BYTES;
#pragma unroll
                for (int k = 0; k < BK / 16; k++)
                    tc::umma_f16(tmem, tc::sdesc_kmajor_sw128(a_addr + 32 * k),
                                 tc::sdesc_kmajor_sw128(b_addr + 32 * k), idesc,
                                 (first && k == 0) ? 0u : 1u);
                tc::umma_commit(&bars->empty[s]);
                if (last) {
                    tc::umma_commit(&bars->accf);
                    cc++;
                }
                kbc++;
                pos_next(q, p, g, BN);
            }
            if (!ok) {
                bars->abort = 1;
                atomicExch(err, 2);
            }
            tc::umma_commit(&bars->done);
            tc::mbar_wait(&bars->done, 0, &bars->never);
        }
        __syncwarp();
    } else {
        // ================================================ epilogue (warps 4..19)
        const int quarter = (warp - 4) >> 2;
        const int row = ((warp & 3) << 5) + lane;
        const uint32_t lb = (uint32_t)((warp & 3) * 32) << 16;
        const uint32_t tD = tmem + lb + quarter * CW;          // fp32 chunk
        const uint32_t tR = tmem + lb + BN + quarter * CW;     // int32 running sum
        uint32_t cc = 0;
        bool ok = true;
        Pos q;
        pos_set_tile(q, blockIdx.x, p, g, BN);
        while (ok && q.tile < g.total) {
            const int nch = (q.nkb + CHUNK_KB - 1) / CHUNK_KB;
            for (int c = 0; c < nch; c++) {
                if (!tc::mbar_wait_sleep(&bars->accf, cc & 1, abort_flag)) {
                    ok = false;
                    bars->abort = 1;
                    atomicExch(err, 3);
                    break;
                }
                tc::tc_fence_after();
#pragma unroll
                for (int cb = 0; cb < CW; cb += LDW) {
                    uint32_t d[LDW], r[LDW];
                    tmem_ld_w<LDW>(tD + cb, d);
                    if (c > 0) tmem_ld_w<LDW>(tR + cb, r);
                    tc::tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < LDW; i++)
                        r[i] = (uint32_t)((c > 0 ? (int)r[i] : 0) +
                                          __float2int_rn(__uint_as_float(d[i])));
                    tmem_st_w<LDW>(tR + cb, r);
                }
                tc::tmem_st_wait();
                tc::tc_fence_before();
                tc::mbar_arrive(&bars->acce);
                cc++;
            }
            if (!ok || *abort_flag) break;
            const int64_t m = q.m0 + row;
            if (__any_sync(0xffffffffu, m < p.M)) {
#pragma unroll
                for (int cb = 0; cb < CW; cb += LDW) {
                    uint32_t r[LDW];
                    tmem_ld_w<LDW>(tR + cb, r);
                    tc::tmem_ld_wait();
                    write_quarter<LDW>(p, reinterpret_cast<const int(&)[LDW]>(r), q.m0,
                                       q.n0 + quarter * CW + cb, row, lane, out32, out64, s1, hi_c,
                                       lo_c);
                }
            }
            pos_set_tile(q, q.tile + gridDim.x, p, g, BN);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 20) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, TMEM_COLS);
    }
}

// s[i] += 0x4B400000 + the exact integer held in the fp32 value d[i] (|d| <= 1024 127^2 <
// 2^24), modulo 2^32; the caller subtracts 0x4B400000 per folded chunk at the end.  When
// every |d| < 2^22, d + 1.5 2^23 is exact and its bit pattern is that sum, one add and one
// integer add per value; otherwise the conversion instruction and the constant.  (The
// kernels start each tile's sums at -nch FOLD_BIAS.)
constexpr uint32_t FOLD_BIAS = 0x4B400000u;

template <int W>
__device__ __forceinline__ void fold_f32(int* s, const uint32_t (&d)[W]) {
    float mx = 0.0f;
#pragma unroll
    for (int i = 0; i < W; i++) mx = fmaxf(mx, fabsf(__uint_as_float(d[i])));
    if (mx < 4194304.0f) {
#pragma unroll
        for (int i = 0; i < W; i++)
            s[i] = (int)((uint32_t)s[i] + __float_as_uint(__uint_as_float(d[i]) + 12582912.0f));
    } else {
#pragma unroll
        for (int i = 0; i < W; i++)
            s[i] = (int)((uint32_t)s[i] + (uint32_t)__float2int_rn(__uint_as_float(d[i])) +
                         FOLD_BIAS);
    }
}

// ---------------------------------------------------------------- all-TMA forward kernel
// Stride-1/2 convolutions with whole 64-channel k-blocks, over fp16 carriers of the codes
// (a pre-pass widens the input once per call).  The M tile is a BH x BW rectangle of one
// image's output pixels; for k-block (tap r,s; channels c0..c0+63) its A rows are the input
// box of that tap -- one 4-D TMA load (element strides = the conv strides, zero fill
// outside the image = the padding) lands them directly in the K-major 128-byte-swizzled
// UMMA layout, next to the B tile (fp16 weights, 2-D TMA).  Warps 0 and 2 issue the A and
// the B loads, warp 1 the MMAs into two fp32 accumulators (chunk c in accumulator c % 2), and 16 epilogue
// warps (4 warpgroups, a quarter of the columns each) fold every finished chunk into int32
// sums held in registers, so neither the loads nor the folds stall the tensor pipe; a
// tile's output is written while the next tile's MMAs run.  Persistent over the tiles.

constexpr int THREADS_T = 640;       // warps 0, 2 TMA, warp 1 MMA, warps 4-19 epilogue
constexpr int EPI_T = 512;
constexpr int STAGES_MAX = 8;

template <int BN>
struct CfgT {
    static constexpr int STAGE_BYTES = A_BYTES + BN * 128;
    // as many stages as 192 KB hold: 4 at BN = 256, 6 at 128, 8 at 64 (the k-blocks in
    // flight are what hide the load -> MMA -> release round trip)
    static constexpr int STAGES =
        196608 / STAGE_BYTES < STAGES_MAX ? 196608 / STAGE_BYTES : STAGES_MAX;
    static constexpr int BAR_OFF = STAGES * STAGE_BYTES;
    // per epilogue warp a 2 KB box (32 rows x 16 int32, 64-byte swizzle) staging the TMA
    // stores of the int32 output
    static constexpr int OUT_OFF = BAR_OFF + 1024;
    static constexpr int SMEM = OUT_OFF + 16 * 2048 + 1024;
    static constexpr int TMEM_COLS = 2 * BN;
    static_assert(SMEM <= 232448, "shared memory");
};

struct BarsT {
    uint64_t full[STAGES_MAX];      // count 2: the A and the B issuer
    uint64_t empty[STAGES_MAX];
    uint64_t accf[2];
    uint64_t acce[2];
    uint64_t done;
    uint32_t tmem_base;
    int abort;
    int never;
};

struct RectGrid {
    int PT, QT, BW, BH;   // rectangles per image (rows x columns) and their size
    int mt, nt, total;    // m-tiles (N * PT * QT), n-tiles, tiles
    int nb;               // weight gradient: 64-channel blocks per im2col box
};

struct RectPos {
    int tile, kb;
    int n, p0, q0, n0;
    int slice;            // reduction slice (tiles beyond mt nt)
    int e, ne;            // k-block kb is the tile's e-th of ne
    int r, s, c0;         // its tap and first channel
    uint32_t rm, sm;      // the tile's taps (bits r of rm, s of sm) in k-block order
};

// whether an output index o in [o_lo, o_hi] reads an input index o stride + off in [0, extent)
// (stride 1 or 2, as the rectangle kernels take)
__host__ __device__ __forceinline__ bool tap_meets(int extent, int o_lo, int o_hi, int stride,
                                                   int off) {
    const int sh = stride - 1;
    const int lo = off >= 0 ? 0 : (-off + sh) >> sh;
    const int top = extent - 1 - off;
    if (top < 0) return false;
    const int hi = top >> sh;
    return (lo > o_lo ? lo : o_lo) <= (hi < o_hi ? hi : o_hi);
}

// Tile `tile` and its first k-block.  k-blocks run over taps (r, s) in row-major order, 64
// channels at a time; with skip_taps a tile keeps only the rows r and columns s of taps that
// read inside the image for some of its output pixels (all of them if that leaves none).
__device__ __forceinline__ void rpos_set(RectPos& q, int tile, const TcP& p, const RectGrid& g,
                                         int BN) {
    q.tile = tile;
    q.kb = 0;
    q.e = 0;
    q.ne = 0;
    if (tile >= g.total) return;
    const int mt = tile % g.mt;
    const int rest = tile / g.mt;
    q.n0 = (rest % g.nt) * BN;
    q.slice = rest / g.nt;
    const int qt = mt % g.QT;
    const int pt = (mt / g.QT) % g.PT;
    q.n = mt / (g.QT * g.PT);
    q.p0 = pt * g.BH;
    q.q0 = qt * g.BW;
    if (!p.skip_taps) {
        q.rm = (1u << p.R) - 1u;
        q.sm = (1u << p.S) - 1u;
        q.r = q.s = q.c0 = 0;
        q.ne = p.nkb_total;
        return;
    }
    uint32_t rm = (1u << p.R) - 1u, sm = (1u << p.S) - 1u;
    {
        const uint32_t a = p.band_r[pt], b = p.band_s[qt];
        if (a && b) { rm = a; sm = b; }
    }
    q.rm = rm;
    q.sm = sm;
    q.r = __ffs(rm) - 1;
    q.s = __ffs(sm) - 1;
    q.c0 = 0;
    q.ne = __popc(rm) * __popc(sm) * (p.C / BK);
    q.kb = (q.r * p.S + q.s) * (p.C / BK);
}

__device__ __forceinline__ void rpos_next(RectPos& q, const TcP& p, const RectGrid& g, int BN) {
    if (q.tile >= g.total) return;
    if (++q.e >= q.ne) {
        rpos_set(q, q.tile + gridDim.x, p, g, BN);
        return;
    }
    q.c0 += BK;
    if (!p.skip_taps) {          // every tap: k-blocks in plain order
        q.kb++;
        if (q.c0 >= p.C) {
            q.c0 = 0;
            if (++q.s == p.S) { q.s = 0; q.r++; }
        }
        return;
    }
    if (q.c0 >= p.C) {
        q.c0 = 0;
        const uint32_t sn = q.sm & (0xfffffffeu << q.s);      // the tile's taps after s
        if (sn) {
            q.s = __ffs(sn) - 1;
        } else {
            q.s = __ffs(q.sm) - 1;
            q.r = __ffs(q.rm & (0xfffffffeu << q.r)) - 1;
        }
    }
    q.kb = (q.r * p.S + q.s) * (p.C / BK) + q.c0 / BK;
}

// per-channel statistics of LDW columns over the warp's 32 rows (OUT_STATS): the maximum,
// and the minimum and the sum when st_mask asks for them (the sum as one signed 32-bit
// reduction under ST_SUM32, else as two 16-bit halves)
template <int LDW>
__device__ __forceinline__ void col_stats(const TcP& p, const int* r, bool valid, int c0,
                                          int lane, unsigned long long* __restrict__ s1,
                                          int* __restrict__ hi_c, int* __restrict__ lo_c) {
    long long my_sum = 0;
    int my_hi = INT_MIN, my_lo = INT_MAX;
    const bool want_hi = !(p.st_mask & ST_NOEXT);
    const bool want_lo = want_hi && (p.st_mask & TC_STATS_LO);
    const bool want_sum = p.st_mask & TC_STATS_SUM, sum32 = p.st_mask & ST_SUM32;
#pragma unroll
    for (int j = 0; j < LDW; j++) {
        const int v = r[j];
        if (want_hi) {
            const int mx = __reduce_max_sync(0xffffffffu, valid ? v : INT_MIN);
            if (lane == j) my_hi = mx;
        }
        if (want_lo) {
            const int mn = __reduce_min_sync(0xffffffffu, valid ? v : INT_MAX);
            if (lane == j) my_lo = mn;
        }
        if (want_sum) {
            if (sum32) {
                const int sm = __reduce_add_sync(0xffffffffu, valid ? v : 0);
                if (lane == j) my_sum = sm;
            } else {
                const unsigned sl =
                    __reduce_add_sync(0xffffffffu, valid ? ((unsigned)v & 0xffffu) : 0u);
                const int sh = __reduce_add_sync(0xffffffffu, valid ? (v >> 16) : 0);
                if (lane == j) my_sum = (long long)sh * 65536 + (long long)sl;
            }
        }
    }
    const int gcol = c0 + lane;
    if (lane < LDW && gcol < p.ncols) {
        if (want_hi && my_hi != INT_MIN) atomicMax(&hi_c[gcol], my_hi);
        if (want_lo && my_lo != INT_MAX) atomicMin(&lo_c[gcol], my_lo);
        if (want_sum && my_sum) atomicAdd(&s1[gcol], (unsigned long long)my_sum);
    }
}

// int32 stores and per-channel statistics (OUT_STATS) or int64 atomic adds of LDW columns
// of one output row m (valid: the row exists)
template <int LDW>
__device__ __forceinline__ void write_row(const TcP& p, const uint32_t (&r)[LDW], int64_t m,
                                          bool valid, int c0, int lane,
                                          int32_t* __restrict__ out32,
                                          long long* __restrict__ out64,
                                          unsigned long long* __restrict__ s1,
                                          int* __restrict__ hi_c, int* __restrict__ lo_c) {
    if (p.out == OUT_PART32) {
        if (valid) {
            int32_t* dst = out32 + m * p.ncols + c0;
#pragma unroll
            for (int i = 0; i < LDW / 4; i++)
                if (c0 + 4 * i < p.ncols)
                    reinterpret_cast<int4*>(dst)[i] = make_int4((int)r[4 * i], (int)r[4 * i + 1],
                                                                (int)r[4 * i + 2], (int)r[4 * i + 3]);
        }
        return;
    }
    if (p.out == OUT_STATS) {
        if (valid) {
            int32_t* dst = out32 + m * p.ncols + c0;
#pragma unroll
            for (int i = 0; i < LDW / 4; i++)
                if (c0 + 4 * i < p.ncols)
                    reinterpret_cast<int4*>(dst)[i] = make_int4((int)r[4 * i], (int)r[4 * i + 1],
                                                                (int)r[4 * i + 2], (int)r[4 * i + 3]);
        }
        col_stats<LDW>(p, reinterpret_cast<const int*>(r), valid, c0, lane, s1, hi_c, lo_c);
    } else if (valid) {
        long long* dst = out64 + m * p.ncols + c0;
#pragma unroll
        for (int j = 0; j < LDW; j++)
            if ((int)r[j] != 0 && c0 + j < p.ncols)
                atomicAdd(reinterpret_cast<unsigned long long*>(dst + j),
                          (unsigned long long)(long long)(int)r[j]);
    }
}

// The warp's 32 output rows (tile rows 32 (warp % 4) .. + 31) are a box of pixels, min(BW,
// 32) wide and 32 / min(BW, 32) high, starting at output pixel (pp0, qq0) of image n.  Per
// 16 columns the lanes write their 64-byte rows into the warp's 2 KB staging box in the
// 64-byte-swizzled layout of map `omap` (16-byte chunk i of row l at chunk i ^ ((l >> 1) & 3):
// eight lanes of a store phase hit eight distinct bank groups) and lane 0 issues one TMA
// store, which writes only the part inside the tensor.  The box is reused once the previous
// store has read it.
template <int CW>
__device__ __forceinline__ void tile_store(const CUtensorMap* omap, const int (&sum)[CW],
                                           uint8_t* stg, int c0, int pp0, int qq0, int n,
                                           const TcP& p, int lane) {
    const bool box_in = pp0 < p.P && qq0 < p.Q;
    const uint32_t sw = (uint32_t)((lane >> 1) & 3);
#pragma unroll
    for (int cb = 0; cb < CW; cb += 16) {
        if (lane == 0) tc::bulk_wait_read_all();
        __syncwarp();
        uint8_t* row = stg + lane * 64;
#pragma unroll
        for (int i = 0; i < 4; i++)
            *reinterpret_cast<int4*>(row + (((uint32_t)i ^ sw) << 4)) =
                make_int4(sum[cb + 4 * i], sum[cb + 4 * i + 1], sum[cb + 4 * i + 2],
                          sum[cb + 4 * i + 3]);
        tc::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0 && box_in && c0 + cb < p.ncols) {
            tc::tma_store_4d(omap, stg, c0 + cb, qq0, pp0, n);
            tc::bulk_commit();
        }
    }
}

// weight-gradient tile position: (channel tile, column tile, K split) and k-block
struct WgPos {
    int tile, kb, nkb, kb0;
    int64_t m0;
    int n0;
};

__device__ __forceinline__ void wpos_set(WgPos& q, int tile, const TcP& p, const RectGrid& g,
                                         int BN) {
    q.tile = tile;
    q.kb = 0;
    q.nkb = 0;
    if (tile >= g.total) return;
    const int mt = tile % g.mt;
    const int rest = tile / g.mt;
    const int nt = rest % g.nt;
    const int sp = rest / g.nt;
    q.m0 = (int64_t)mt * BM;
    q.n0 = nt * BN;
    q.kb0 = sp * p.kb_per_split;
    const int n = p.nkb_total - q.kb0;
    q.nkb = n > p.kb_per_split ? p.kb_per_split : n;
}

__device__ __forceinline__ void wpos_next(WgPos& q, const TcP& p, const RectGrid& g, int BN) {
    if (q.tile >= g.total) return;
    if (++q.kb >= q.nkb) wpos_set(q, q.tile + gridDim.x, p, g, BN);
}

template <bool WG>
struct TPos;

// idx(): the k-block's place in its tile, cnt(): the tile's k-blocks
// (the MMA issuer and the epilogue only count a tile's k-blocks: next() does not track taps)
template <>
struct TPos<false> : RectPos {
    __device__ void set(int t, const TcP& p, const RectGrid& g, int BN) {
        rpos_set(*this, t, p, g, BN);
    }
    __device__ void next(const TcP& p, const RectGrid& g, int BN) {
        if (tile < g.total && ++e >= ne) rpos_set(*this, tile + gridDim.x, p, g, BN);
    }
    __device__ int idx() const { return e; }
    __device__ int cnt() const { return ne; }
};

template <>
struct TPos<true> : WgPos {
    __device__ void set(int t, const TcP& p, const RectGrid& g, int BN) { wpos_set(*this, t, p, g, BN); }
    __device__ void next(const TcP& p, const RectGrid& g, int BN) { wpos_next(*this, p, g, BN); }
    __device__ int idx() const { return kb; }
    __device__ int cnt() const { return nkb; }
};

// WG: the weight gradient.  A k-block is a BW x BH rectangle of 64 output pixels of one
// image (the rectangles tile every image; pixels outside it read zero errors).  A = E^T
// (one 5-D box: 64 channels x the rectangle x 2 channel blocks of the fp16 errors, map
// `wmap`) and B = the im2col of x (per tap, one 5-D box of 64 channels x the rectangle at
// the conv strides x g.nb channel blocks, map `amap`), both MN-major: a box lands as
// g.nb blocks of 64 rows of 128 bytes, the 8192-byte MN-block stride of the UMMA layout.
// Tiles are (channel tile, column tile, K split); the epilogue writes each split's int32
// sums to its own slab (OUT_PART32).
template <int BN, bool WG>
__global__ void __launch_bounds__(THREADS_T, 1)
    k_conv_tct(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap amap,
               const __grid_constant__ CUtensorMap omap,
               TcP p, RectGrid g, int32_t* __restrict__ out32, long long* __restrict__ out64,
               unsigned long long* __restrict__ s1, int* __restrict__ hi_c,
               int* __restrict__ lo_c, int* __restrict__ err) {
    constexpr int STAGE_BYTES = CfgT<BN>::STAGE_BYTES;
    constexpr int NST = CfgT<BN>::STAGES;
    constexpr int TMEM_COLS = CfgT<BN>::TMEM_COLS;
    constexpr int CW = BN / 4;                 // columns per epilogue warpgroup
    constexpr int LDW = CW < 16 ? CW : 16;     // columns per TMEM load
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    BarsT* bars = reinterpret_cast<BarsT*>(smem + CfgT<BN>::BAR_OFF);

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    if (__syncthreads_or(tid == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    if ((int)blockIdx.x >= g.total) return;

    if (tid == 0) {
        for (int s = 0; s < NST; s++) {
            tc::mbar_init(&bars->full[s], 2);
            tc::mbar_init(&bars->empty[s], 1);
        }
        for (int b = 0; b < 2; b++) {
            tc::mbar_init(&bars->accf[b], 1);
            tc::mbar_init(&bars->acce[b], EPI_T);
        }
        tc::mbar_init(&bars->done, 1);
        bars->abort = 0;
        bars->never = 0;
        tc::mbar_fence_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&bars->tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort_flag = &bars->abort;

    if (warp == 0 || warp == 2) {
        // ================================================ TMA issuers
        // Warp 0 loads the A tiles and warp 2 the B tiles of the same k-blocks; each adds
        // its bytes to the stage's full barrier and arrives once (count 2), so the two
        // issue chains run side by side.
        const bool side_a = warp == 0;
        if (lane == 0) tc::tma_prefetch_desc(side_a == WG ? &wmap : &amap);
        const uint32_t tx = side_a ? (uint32_t)A_BYTES : (uint32_t)(STAGE_BYTES - A_BYTES);
        int s = 0;
        uint32_t ph = 0;
        uint32_t kbc = 0;
        int issued = 0;
        if constexpr (WG) {
            WgPos q;
            wpos_set(q, blockIdx.x, p, g, BN);
            // per tile: the box coordinates of the B column runs (x and y offsets of the tap,
            // first channel block); per k-block: the rectangle, advanced without divisions
            int bx[4], by[4], bc[4];
            int tile_seen = -1, nimg = 0, pt = 0, qt = 0;
            while (q.tile < g.total) {
                if (q.tile != tile_seen) {
                    tile_seen = q.tile;
#pragma unroll
                    for (int j = 0; j < 4; j++) {
                        const int col = q.n0 + 64 * g.nb * j;
                        const int tap = col / p.C;
                        const int r = tap / p.S, ss = tap - r * p.S;
                        bx[j] = ss * p.dw - p.pw;
                        by[j] = r * p.dh - p.ph;
                        bc[j] = (col - tap * p.C) >> 6;
                    }
                    const int kr = q.kb0;
                    nimg = kr / (g.PT * g.QT);
                    const int rr = kr - nimg * (g.PT * g.QT);
                    pt = rr / g.QT;
                    qt = rr - pt * g.QT;
                }
                if (!tc::mbar_wait_warp(&bars->empty[s], ph ^ 1, abort_flag)) {
                    bars->abort = 1;
                    atomicExch(err, 4);
                    break;
                }
                uint8_t* st = smem + s * STAGE_BYTES;
                tc::mbar_expect_tx_e(&bars->full[s], tx);
                // the k-block's pixels: rectangle (pt, qt) of image nimg
                const int pp = pt * g.BH, qq = qt * g.BW;
                if (side_a) {
                    // A: E[rectangle][m0 .. m0+127], both 64-channel blocks in one box (zero
                    // outside P x Q and past the last channel block)
                    tc::tma_load_5d_e(st, &wmap, &bars->full[s], 0, qq, pp, (int)(q.m0 >> 6),
                                      nimg);
                } else {
                    // B: per run of g.nb 64-column blocks (one tap, 64 g.nb channels) the
                    // input box of the pixels
#pragma unroll
                    for (int j = 0; j < 4; j++) {
                        if (j * g.nb >= BN / 64) break;
                        tc::tma_load_5d_e(st + A_BYTES + 8192 * g.nb * j, &amap, &bars->full[s],
                                          0, qq * p.sw + bx[j], pp * p.sh + by[j], bc[j], nimg);
                    }
                }
                if (++qt == g.QT) {
                    qt = 0;
                    if (++pt == g.PT) { pt = 0; nimg++; }
                }
                tc::mbar_arrive_e(&bars->full[s]);
                issued = (int)kbc + 1;
                kbc++;
                if (++s == NST) { s = 0; ph ^= 1; }
                wpos_next(q, p, g, BN);
            }
        } else {
            RectPos q;
            rpos_set(q, blockIdx.x, p, g, BN);
            while (q.tile < g.total) {
                if (!tc::mbar_wait_warp(&bars->empty[s], ph ^ 1, abort_flag)) {
                    bars->abort = 1;
                    atomicExch(err, 4);
                    break;
                }
                uint8_t* st = smem + s * STAGE_BYTES;
                tc::mbar_expect_tx_e(&bars->full[s], tx);
                if (side_a)
                    tc::tma_load_4d_e(st, &amap, &bars->full[s], p.cofs + q.slice * p.C + q.c0,
                                      q.q0 * p.sw + q.s * p.dw - p.pw,
                                      q.p0 * p.sh + q.r * p.dh - p.ph, q.n);
                else
                    tc::tma_load_2d_e(st + A_BYTES, &wmap, &bars->full[s], q.kb * BK,
                                      q.slice * p.slice_rows + q.n0);
                tc::mbar_arrive_e(&bars->full[s]);
                issued = (int)kbc + 1;
                kbc++;
                if (++s == NST) { s = 0; ph ^= 1; }
                rpos_next(q, p, g, BN);
            }
        }
        if (*abort_flag) {
            // let this warp's copies in flight land before the CTA leaves
            for (int kb = (issued > NST ? issued - NST : 0); kb < issued; kb++)
                tc::mbar_wait(&bars->full[kb % NST], (uint32_t)(kb / NST) & 1, &bars->never);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ================================================ MMA issuer
        {
            const uint32_t idesc = idesc_f16(BM, BN, WG);
            bool ok = true;
            uint32_t kbc = 0, cc = 0;
            int s = 0;
            uint32_t ph = 0;
            TPos<WG> q;
            q.set(blockIdx.x, p, g, BN);
            while (ok && q.tile < g.total) {
                const bool first = (q.idx() % CHUNK_KB) == 0;
                const bool last = ((q.idx() % CHUNK_KB) == CHUNK_KB - 1) || q.idx() == q.cnt() - 1;
                const uint32_t buf = cc & 1;
                if (first && cc >= 2 &&
                    !tc::mbar_wait_warp(&bars->acce[buf], ((cc >> 1) - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                if (!tc::mbar_wait_warp(&bars->full[s], ph, abort_flag)) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t a_addr = tc::smem_u32(smem + s * STAGE_BYTES);
                const uint32_t b_addr = a_addr + A_BYTES;
#pragma unroll
                for (int k = 0; k < BK / 16; k++) {
                    uint64_t ad, bd;
                    if (WG) {
                        ad = sdesc_mnmajor_sw128(a_addr + 2 * 1024 * k);
                        bd = sdesc_mnmajor_sw128(b_addr + 2 * 1024 * k);
                    } else {
                        ad = tc::sdesc_kmajor_sw128(a_addr + 32 * k);
                        bd = tc::sdesc_kmajor_sw128(b_addr + 32 * k);
                    }
                    tc::umma_f16_e(tmem + buf * BN, ad, bd, idesc, (first && k == 0) ? 0u : 1u);
                }
                tc::umma_commit_e(&bars->empty[s]);
                if (last) {
                    tc::umma_commit_e(&bars->accf[buf]);
                    cc++;
                }
                kbc++;
                if (++s == NST) { s = 0; ph ^= 1; }
                q.next(p, g, BN);
            }
            if (!ok) {
                bars->abort = 1;
                atomicExch(err, 2);
            }
            tc::umma_commit_e(&bars->done);
            tc::mbar_wait(&bars->done, 0, &bars->never);
        }
        __syncwarp();
    } else if (warp >= 4) {
        // ================================================ epilogue (warps 4..19)
        const int quarter = (warp - 4) >> 2;
        const int row = ((warp & 3) << 5) + lane;
        const uint32_t taddr = tmem + ((uint32_t)((warp & 3) * 32) << 16) + quarter * CW;
        const int dp = row / g.BW, dq = row - (row / g.BW) * g.BW;
        uint32_t cc = 0;
        bool ok = true;
        TPos<WG> q;
        q.set(blockIdx.x, p, g, BN);
        int sum[CW];
        uint32_t amax_t = 0;      // WG with a single split: max |G| of this thread's outputs
        int gmx = INT_MIN, gmn = INT_MAX;     // ST_GMAX: this thread's extremes
        const int wr0 = (warp & 3) << 5;      // first tile row (pixel) of the warp
        uint8_t* stg = smem + CfgT<BN>::OUT_OFF + (warp - 4) * 2048;
        while (ok && q.tile < g.total) {
            const int nch = (q.cnt() + CHUNK_KB - 1) / CHUNK_KB;
            // the sums start at minus the FOLD_BIAS of the tile's nch chunks
            const int sum0 = (int)(0u - (uint32_t)nch * FOLD_BIAS);
#pragma unroll
            for (int i = 0; i < CW; i++) sum[i] = sum0;
            for (int c = 0; c < nch; c++) {
                const uint32_t buf = cc & 1;
                if (!tc::mbar_wait_sleep(&bars->accf[buf], (cc >> 1) & 1, abort_flag)) {
                    ok = false;
                    bars->abort = 1;
                    atomicExch(err, 3);
                    break;
                }
                tc::tc_fence_after();
#pragma unroll
                for (int cb = 0; cb < CW; cb += LDW) {
                    uint32_t d[LDW];
                    tmem_ld_w<LDW>(taddr + buf * BN + cb, d);
                    tc::tmem_ld_wait();
                    fold_f32<LDW>(sum + cb, d);
                }
                tc::tc_fence_before();
                tc::mbar_arrive(&bars->acce[buf]);
                cc++;
            }
            if (!ok || *abort_flag) break;
            bool valid;
            int64_t m;
            if constexpr (WG) {
                m = q.m0 + row;
                valid = m < p.M;
            } else {
                const int pp = q.p0 + dp, qq = q.q0 + dq;
                valid = pp < p.P && qq < p.Q;
                m = ((int64_t)q.n * p.P + pp) * p.Q + qq;
            }
            int32_t* o32 = out32;
            if constexpr (WG) {
                // the split's own int32 slab (OUT_PART32): no atomics
                if (p.out == OUT_PART32)
                    o32 = out32 + (int64_t)(q.kb0 / p.kb_per_split) * p.M * p.ncols;
                // a single split: its slab is the result, and s1 collects max |G|
                if (s1 && valid) {
#pragma unroll
                    for (int i = 0; i < CW; i++)
                        if (q.n0 + quarter * CW + i < p.ncols)
                            amax_t = max(amax_t, (uint32_t)abs(sum[i]));
                }
            }
            if (!WG && p.tma_out) {
                if constexpr (!WG) {
                    if (p.st_mask & ST_GMAX) {
                        // columns past ncols hold zeros (zero-filled weight rows): harmless
                        if (valid) {
#pragma unroll
                            for (int i = 0; i < CW; i++) {
                                gmx = max(gmx, sum[i]);
                                gmn = min(gmn, sum[i]);
                            }
                        }
                    } else if ((p.st_mask & (TC_STATS_SUM | TC_STATS_LO)) ||
                               !(p.st_mask & ST_NOEXT)) {
#pragma unroll
                        for (int cb = 0; cb < CW; cb += LDW)
                            col_stats<LDW>(p, sum + cb, valid, q.n0 + quarter * CW + cb, lane, s1,
                                           hi_c, lo_c);
                    }
                    tile_store<CW>(&omap, sum, stg, q.n0 + quarter * CW, q.p0 + wr0 / g.BW,
                                   q.q0 + wr0 % g.BW, q.n, p, lane);
                }
            } else if (__any_sync(0xffffffffu, valid)) {
#pragma unroll
                for (int cb = 0; cb < CW; cb += LDW) {
                    uint32_t v[LDW];
#pragma unroll
                    for (int i = 0; i < LDW; i++) v[i] = (uint32_t)sum[cb + i];
                    write_row<LDW>(p, v, m, valid, q.n0 + quarter * CW + cb, lane, o32, out64,
                                   s1, hi_c, lo_c);
                }
            }
            q.set(q.tile + gridDim.x, p, g, BN);
        }
        if (!WG && p.tma_out) {
            // the last stores leave the staging box before the CTA does; the global extremes
            if (lane == 0) tc::bulk_wait_all();
            __syncwarp();
            if (p.st_mask & ST_GMAX) {
                gmx = __reduce_max_sync(0xffffffffu, gmx);
                gmn = __reduce_min_sync(0xffffffffu, gmn);
                if (lane == 0 && gmx >= gmn) {
                    atomicMax(&hi_c[0], gmx);
                    if (p.st_mask & TC_STATS_LO) atomicMin(&lo_c[0], gmn);
                }
            }
        }
        if constexpr (WG) {
            if (s1) {
                amax_t = warp_max_u32(amax_t);
                if (lane == 0 && amax_t) atomicMax(s1, (unsigned long long)amax_t);
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, TMEM_COLS);
    }
}

// ---------------------------------------------------------------- channel-major forward
// The forward (and stride-1 data-gradient) GEMM transposed, for layers with at most 128
// output channels: D^T[channels x pixels] = W X^T with M = 128 output channels (weight rows
// past the last channel are TMA zero fill) and N = 256 pixels (a BW x BH rectangle of one
// image).  tcgen05 reaches its full rate only at N = 256; the pixel-major kernel would run
// these layers at N = 64 or 128, a quarter or half of it.  TMEM lane = output channel,
// column = pixel of the rectangle.  Each epilogue thread owns one channel and 64 pixels, so
// a warp's int32 stores cover 32 consecutive channels of one pixel and the per-channel
// statistics are per-thread sums (one atomic triple per thread and tile).  Loads, MMA
// issue, accumulator handshake and bounded waits are those of k_conv_tct.
constexpr int CM_PIX = 256;        // pixels per tile (GEMM N)
constexpr int CM_CH = 128;         // output channels per tile (GEMM M)

__global__ void __launch_bounds__(THREADS_T, 1)
    k_conv_tcc(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap amap,
               TcP p, RectGrid g, int bw_log2, int32_t* __restrict__ out32,
               unsigned long long* __restrict__ s1, int* __restrict__ hi_c,
               int* __restrict__ lo_c, int* __restrict__ err) {
    constexpr int STAGE_BYTES = A_BYTES + CM_PIX * 128;
    constexpr int NST = CfgT<256>::STAGES;
    constexpr int TMEM_COLS = 2 * CM_PIX;
    constexpr int CW = CM_PIX / 4;             // pixels per epilogue warpgroup
    constexpr int LDW = 16;                    // columns per TMEM load
    static_assert(STAGE_BYTES == CfgT<256>::STAGE_BYTES, "stage layout of CfgT<256>");
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    BarsT* bars = reinterpret_cast<BarsT*>(smem + CfgT<256>::BAR_OFF);

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    if (__syncthreads_or(tid == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    if ((int)blockIdx.x >= g.total) return;

    if (tid == 0) {
        for (int s = 0; s < NST; s++) {
            tc::mbar_init(&bars->full[s], 2);
            tc::mbar_init(&bars->empty[s], 1);
        }
        for (int b = 0; b < 2; b++) {
            tc::mbar_init(&bars->accf[b], 1);
            tc::mbar_init(&bars->acce[b], EPI_T);
        }
        tc::mbar_init(&bars->done, 1);
        bars->abort = 0;
        bars->never = 0;
        tc::mbar_fence_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&bars->tmem_base, TMEM_COLS);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort_flag = &bars->abort;

    if (warp == 0 || warp == 2) {
        // ================================================ TMA issuers
        // warp 0 the weight tiles (A), warp 2 the pixel tiles (B); full barriers count 2
        const bool side_a = warp == 0;
        if (lane == 0) tc::tma_prefetch_desc(side_a ? &wmap : &amap);
        const uint32_t tx = side_a ? (uint32_t)A_BYTES : (uint32_t)(STAGE_BYTES - A_BYTES);
        int s = 0;
        uint32_t ph = 0;
        RectPos q;
        rpos_set(q, blockIdx.x, p, g, CM_CH);
        uint32_t kbc = 0;
        int issued = 0;
        while (q.tile < g.total) {
            if (!tc::mbar_wait_warp(&bars->empty[s], ph ^ 1, abort_flag)) {
                bars->abort = 1;
                atomicExch(err, 4);
                break;
            }
            uint8_t* st = smem + s * STAGE_BYTES;
            tc::mbar_expect_tx_e(&bars->full[s], tx);
            if (side_a)     // A: weight rows n0 .. n0 + 127 (zero past the last channel)
                tc::tma_load_2d_e(st, &wmap, &bars->full[s], q.kb * BK, q.n0);
            else            // B: the 256 input pixels of tap (r, s), channels c0 .. c0 + 63
                tc::tma_load_4d_e(st + A_BYTES, &amap, &bars->full[s], p.cofs + q.c0,
                                  q.q0 * p.sw + q.s * p.dw - p.pw,
                                  q.p0 * p.sh + q.r * p.dh - p.ph, q.n);
            tc::mbar_arrive_e(&bars->full[s]);
            issued = (int)kbc + 1;
            kbc++;
            if (++s == NST) { s = 0; ph ^= 1; }
            rpos_next(q, p, g, CM_CH);
        }
        if (*abort_flag) {
            for (int kb = (issued > NST ? issued - NST : 0); kb < issued; kb++)
                tc::mbar_wait(&bars->full[kb % NST], (uint32_t)(kb / NST) & 1, &bars->never);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ================================================ MMA issuer
        {
            const uint32_t idesc = idesc_f16(CM_CH, CM_PIX, false);
            bool ok = true;
            uint32_t kbc = 0, cc = 0;
            int s = 0;
            uint32_t ph = 0;
            TPos<false> q;
            q.set(blockIdx.x, p, g, CM_CH);
            while (ok && q.tile < g.total) {
                const bool first = (q.idx() % CHUNK_KB) == 0;
                const bool last = ((q.idx() % CHUNK_KB) == CHUNK_KB - 1) || q.idx() == q.cnt() - 1;
                const uint32_t buf = cc & 1;
                if (first && cc >= 2 &&
                    !tc::mbar_wait_warp(&bars->acce[buf], ((cc >> 1) - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                if (!tc::mbar_wait_warp(&bars->full[s], ph, abort_flag)) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t a_addr = tc::smem_u32(smem + s * STAGE_BYTES);
                const uint32_t b_addr = a_addr + A_BYTES;
#pragma unroll
                for (int k = 0; k < BK / 16; k++)
                    tc::umma_f16_e(tmem + buf * CM_PIX, tc::sdesc_kmajor_sw128(a_addr + 32 * k),
                                 tc::sdesc_kmajor_sw128(b_addr + 32 * k), idesc,
                                 (first && k == 0) ? 0u : 1u);
                tc::umma_commit_e(&bars->empty[s]);
                if (last) {
                    tc::umma_commit_e(&bars->accf[buf]);
                    cc++;
                }
                kbc++;
                if (++s == NST) { s = 0; ph ^= 1; }
                q.next(p, g, CM_CH);
            }
            if (!ok) {
                bars->abort = 1;
                atomicExch(err, 2);
            }
            tc::umma_commit_e(&bars->done);
            tc::mbar_wait(&bars->done, 0, &bars->never);
        }
        __syncwarp();
    } else if (warp >= 4) {
        // ================================================ epilogue (warps 4..19)
        const int quarter = (warp - 4) >> 2;          // pixels [64 quarter, 64 quarter + 64)
        const int lq = warp & 3;                      // TMEM lanes (channels) 32 lq ..
        const uint32_t taddr = tmem + ((uint32_t)(lq * 32) << 16) + quarter * CW;
        const int bw_mask = g.BW - 1;
        uint32_t cc = 0;
        bool ok = true;
        TPos<false> q;
        q.set(blockIdx.x, p, g, CM_CH);
        int sum[CW];
        while (ok && q.tile < g.total) {
            const int nch = (q.cnt() + CHUNK_KB - 1) / CHUNK_KB;
            // the sums start at minus the FOLD_BIAS of the tile's nch chunks
            const int sum0 = (int)(0u - (uint32_t)nch * FOLD_BIAS);
#pragma unroll
            for (int i = 0; i < CW; i++) sum[i] = sum0;
            for (int c = 0; c < nch; c++) {
                const uint32_t buf = cc & 1;
                if (!tc::mbar_wait_sleep(&bars->accf[buf], (cc >> 1) & 1, abort_flag)) {
                    ok = false;
                    bars->abort = 1;
                    atomicExch(err, 3);
                    break;
                }
                tc::tc_fence_after();
#pragma unroll
                for (int cb = 0; cb < CW; cb += LDW) {
                    uint32_t d[LDW];
                    tc::tmem_ld_32x32b_x16(taddr + buf * CM_PIX + cb, d);
                    tc::tmem_ld_wait();
                    fold_f32<LDW>(sum + cb, d);
                }
                tc::tc_fence_before();
                tc::mbar_arrive(&bars->acce[buf]);
                cc++;
            }
            if (!ok || *abort_flag) break;
            const int ch = q.n0 + lq * 32 + lane;
            const bool chv = ch < p.ncols;
            long long my_sum = 0;
            int my_hi = INT_MIN, my_lo = INT_MAX;
            if (g.BW >= CW) {
                // the quarter's pixels are one run of one output row: pixel j at dst + j ncols
                const int rr0 = quarter * CW;
                const int pp = q.p0 + (rr0 >> bw_log2), qq0 = q.q0 + (rr0 & bw_mask);
                int jlim = pp < p.P ? p.Q - qq0 : 0;
                jlim = jlim < CW ? jlim : CW;
                if (jlim > 0) {
                    int32_t* dst = out32 + (((int64_t)q.n * p.P + pp) * p.Q + qq0) * p.ncols + ch;
#pragma unroll
                    for (int j = 0; j < CW; j++) {
                        if (j < jlim) {               // the same pixel for the whole warp
                            if (chv) dst[j * p.ncols] = sum[j];
                            my_sum += sum[j];
                            my_hi = max(my_hi, sum[j]);
                            my_lo = min(my_lo, sum[j]);
                        }
                    }
                }
            } else {
#pragma unroll
                for (int j = 0; j < CW; j++) {
                    const int rr = quarter * CW + j;
                    const int pp = q.p0 + (rr >> bw_log2), qq = q.q0 + (rr & bw_mask);
                    if (pp < p.P && qq < p.Q) {      // the same pixel for the whole warp
                        const int64_t m = ((int64_t)q.n * p.P + pp) * p.Q + qq;
                        if (chv) out32[m * p.ncols + ch] = sum[j];
                        my_sum += sum[j];
                        my_hi = max(my_hi, sum[j]);
                        my_lo = min(my_lo, sum[j]);
                    }
                }
            }
            if (chv && my_hi != INT_MIN) {
                atomicAdd(&s1[ch], (unsigned long long)my_sum);
                atomicMax(&hi_c[ch], my_hi);
                atomicMin(&lo_c[ch], my_lo);
            }
            q.set(q.tile + gridDim.x, p, g, CM_CH);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, TMEM_COLS);
    }
}

// G[k ncols_out + j] = sum over the splits of the partial sums [k][j] of rows of ncols_in
// columns, j < ncols_out (the weight gradient computed over an im2col with padded columns),
// and max |G| into *amax (zeroed by the caller)
__global__ void k_split_sum_cols(const int32_t* __restrict__ part, int ns, int64_t rows,
                                 int ncols_in, int ncols_out, long long* __restrict__ G,
                                 unsigned long long* __restrict__ amax) {
    const int64_t total = rows * ncols_out, slab = rows * ncols_in;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    uint64_t m = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        const int64_t k = i / ncols_out;
        const int64_t src = k * ncols_in + (i - k * ncols_out);
        long long a = 0;
        for (int sp = 0; sp < ns; sp++) a += __ldg(part + sp * slab + src);
        G[i] = a;
        const uint64_t b = (uint64_t)(a < 0 ? -a : a);
        m = b > m ? b : m;
    }
    m = warp_max_u64(m);
    if ((threadIdx.x & 31) == 0 && m) atomicMax(amax, (unsigned long long)m);
}

// G[i] = sum over the splits of their int32 partial sums (4 elements per thread), and
// max |G| into *amax (zeroed by the caller)
__global__ void k_split_sum(const int32_t* __restrict__ part, int ns, int64_t total4,
                            long long* __restrict__ G, unsigned long long* __restrict__ amax) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    uint64_t m = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total4; i += stride) {
        long long a0 = 0, a1 = 0, a2 = 0, a3 = 0;
        for (int sp = 0; sp < ns; sp++) {
            const int4 v = __ldg(reinterpret_cast<const int4*>(part) + (int64_t)sp * total4 + i);
            a0 += v.x; a1 += v.y; a2 += v.z; a3 += v.w;
        }
        longlong2* g2 = reinterpret_cast<longlong2*>(G) + 2 * i;
        g2[0] = make_longlong2(a0, a1);
        g2[1] = make_longlong2(a2, a3);
        const uint64_t b0 = (uint64_t)(a0 < 0 ? -a0 : a0), b1 = (uint64_t)(a1 < 0 ? -a1 : a1);
        const uint64_t b2 = (uint64_t)(a2 < 0 ? -a2 : a2), b3 = (uint64_t)(a3 < 0 ? -a3 : a3);
        const uint64_t c0 = b0 > b1 ? b0 : b1, c1 = b2 > b3 ? b2 : b3;
        const uint64_t c = c0 > c1 ? c0 : c1;
        m = c > m ? c : m;
    }
    m = warp_max_u64(m);
    if ((threadIdx.x & 31) == 0 && m) atomicMax(amax, (unsigned long long)m);
}

__global__ void k_codes_to_f16_pad(const int8_t* __restrict__ x, __half* __restrict__ xf,
                                   int64_t npix, int K, int Kp) {
    const int kg = Kp / 8;
    const int64_t total = npix * kg;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        const int64_t pix = i / kg;
        const int c0 = (int)(i - pix * kg) * 8;
        uint32_t b[2] = {0u, 0u};
#pragma unroll
        for (int j = 0; j < 8; j++)
            if (c0 + j < K) b[j >> 2] |= ((uint32_t)(uint8_t)x[pix * K + c0 + j]) << (8 * (j & 3));
        uint32_t o[4];
        tc::i8x4_to_f16x4(b[0], o[0], o[1]);
        tc::i8x4_to_f16x4(b[1], o[2], o[3]);
        *reinterpret_cast<uint4*>(xf + pix * Kp + c0) = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

// the im2col of a forward problem with few channels (C % 4 == 0) as fp16 [N P Q][kpad]:
// column j = (r S + s) C + c (the widened weights' order), zeros for padding and
// j >= R S C.  Blocks (pixel range, output row pp, image n); a thread writes 4 columns (one
// tap, 4 channels: one 4-byte load, one 8-byte store) of several output pixels.
__global__ void k_im2col_f16(const int8_t* __restrict__ x, TcP p, __half* __restrict__ A) {
    // thread (g, y): columns 4g .. 4g + 3 (one tap, 4 channels) of the pixels q = y, y +
    // blockDim.y, ... of output row blockIdx.y of image blockIdx.z; the tap is decoded once
    const int j = 4 * threadIdx.x;
    const int pp = blockIdx.y, n = blockIdx.z;
    bool ok = j < p.kdim;
    int dx = 0, c = 0, hh = 0;
    if (ok) {
        const int tap = j / p.C;
        c = j - tap * p.C;
        const int r = tap / p.S, sx = tap - r * p.S;
        hh = pp * p.sh + r * p.dh - p.ph;
        dx = sx * p.dw - p.pw;
        ok = hh >= 0 && hh < p.H;
    }
    const int8_t* xrow = x + (((int64_t)n * p.H + (ok ? hh : 0)) * p.W) * p.cstride + p.cofs + c;
    __half* arow = A + ((int64_t)n * p.P + pp) * p.Q * p.kpad + j;
    for (int qq = blockIdx.x * blockDim.y + threadIdx.y; qq < p.Q; qq += gridDim.x * blockDim.y) {
        const int ww = qq * p.sw + dx;
        uint32_t v = 0;
        if (ok && ww >= 0 && ww < p.W)
            v = __ldg(reinterpret_cast<const uint32_t*>(xrow + (int64_t)ww * p.cstride));
        uint32_t o0, o1;
        tc::i8x4_to_f16x4(v, o0, o1);
        *reinterpret_cast<uint2*>(arow + (int64_t)qq * p.kpad) = make_uint2(o0, o1);
    }
}

// int8 codes [npix][cstride] -> exact fp16 carriers, 16 codes per thread
// launch k_im2col_f16 for the geometry in p (kpad / 4 <= 128 column groups per pixel)
void launch_im2col(const int8_t* x, const TcP& p, __half* A, cudaStream_t st) {
    const int g4 = p.kpad / 4;
    const int by = 256 / g4 > 0 ? 256 / g4 : 1;
    dim3 block((unsigned)g4, (unsigned)by);
    // about 8 pixels per thread: long-lived blocks rather than one pixel each
    dim3 grid((unsigned)((p.Q + 8 * by - 1) / (8 * by)), (unsigned)p.P, (unsigned)p.N);
    k_im2col_f16<<<grid, block, 0, st>>>(x, p, A);
}

__global__ void k_codes_to_f16(const int8_t* __restrict__ x, __half* __restrict__ xf, int64_t n16) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += stride) {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(x) + i);
        uint32_t o[8];
        tc::i8x4_to_f16x4(v.x, o[0], o[1]);
        tc::i8x4_to_f16x4(v.y, o[2], o[3]);
        tc::i8x4_to_f16x4(v.z, o[4], o[5]);
        tc::i8x4_to_f16x4(v.w, o[6], o[7]);
        uint4* dst = reinterpret_cast<uint4*>(xf) + 2 * i;
        dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
        dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
    }
}

// Tile rectangle of the TMA-fed kernels: BW x BH output pixels of one image.
struct TmaTile {
    int BW, BH, PT, QT;
};

// Sticky status of the tensor-core kernels on each device: 0, or the code of the first
// bounded wait that gave up (1: operand loads, 2: MMA issue, 3: epilogue, 4: a TMA-fed
// producer).  Set by the kernels, read and cleared by iq_device_status; while it is set,
// every later launch of these kernels returns at once.
__device__ int g_tc_status;


// int8 KRSC weights -> fp16 [K][kpad] (zero beyond R*S*C)
// int8 KRSC weights -> fp16 [K][kpad] (zero beyond R*S*C): blocks (x, rows y, y + gridDim.y,
// ...), each thread 8 consecutive columns (one 16-byte store)
__global__ void k_widen_weights(const int8_t* __restrict__ w, __half* __restrict__ wf, int K,
                                int kdim, int kpad) {
    const int j0 = (blockIdx.x * blockDim.x + threadIdx.x) * 8;
    if (j0 >= kpad) return;
    for (int k = blockIdx.y; k < K; k += gridDim.y) {
        const int8_t* src = w + (int64_t)k * kdim;
        uint32_t b[2] = {0u, 0u};
#pragma unroll
        for (int t = 0; t < 8; t++)
            if (j0 + t < kdim) b[t >> 2] |= (uint32_t)(uint8_t)src[j0 + t] << (8 * (t & 3));
        uint32_t o[4];
        tc::i8x4_to_f16x4(b[0], o[0], o[1]);
        tc::i8x4_to_f16x4(b[1], o[2], o[3]);
        *reinterpret_cast<uint4*>(wf + (int64_t)k * kpad + j0) = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

// data-gradient weights: wf[c][(r s) kc + k] = w[kofs + k][R-1-r][S-1-s][c] (zero for the
// padding columns j >= R S kc), one 32 x 32 (k, c) transpose through shared memory per block
// and tap: block (c tile, k tile, tap), 32 x 8 threads
__global__ void k_widen_weights_dgrad(const int8_t* __restrict__ w, __half* __restrict__ wf, int K,
                                      int R, int S, int C, int kofs, int kc, int kpad) {
    __shared__ int8_t tile[32][33];
    const int c0 = blockIdx.x * 32, k0 = blockIdx.y * 32, tap = blockIdx.z;
    const int r = tap / S, s = tap - r * S;
    const int tx = threadIdx.x, ty = threadIdx.y;
#pragma unroll
    for (int i = 0; i < 32; i += 8) {
        const int k = k0 + ty + i, c = c0 + tx;
        tile[ty + i][tx] = (k < kc && c < C)
            ? w[(((int64_t)(kofs + k) * R + (R - 1 - r)) * S + (S - 1 - s)) * C + c] : (int8_t)0;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 32; i += 8) {
        const int c = c0 + ty + i, k = k0 + tx;
        if (c < C && k < kc) wf[(int64_t)c * kpad + (int64_t)tap * kc + k] = __int2half_rn(tile[tx][ty + i]);
    }
    // the padding columns of row c (written by the first tap's blocks of the first k tile)
    if (tap == 0 && blockIdx.y == 0) {
        const int kdim = R * S * kc;
#pragma unroll
        for (int i = 0; i < 32; i += 8) {
            const int c = c0 + ty + i;
            if (c < C)
                for (int j = kdim + tx; j < kpad; j += 32) wf[(int64_t)c * kpad + j] = __float2half(0.0f);
        }
    }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// device address of g_tc_status in the CUDA context current at the call (an address that
// belongs to a context, not to a device ordinal: looked up on every call)
int* tc_status_ptr() {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_tc_status) != cudaSuccess || !p) return nullptr;
    return static_cast<int*>(p);
}

bool tc_env_disabled() {
    const char* e = getenv("IQ_DISABLE_TC");
    return e && e[0] == '1';
}

iq_status encode_weights(const __half* wf, int rows, int kpad, int box_rows, CUtensorMap* map) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
    if (!enc) return IQ_ERR_UNSUPPORTED;
    cuuint64_t gdim[2] = {(cuuint64_t)kpad, (cuuint64_t)rows};
    cuuint64_t gstride[1] = {(cuuint64_t)kpad * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, (void*)wf, gdim, gstride, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? IQ_OK : IQ_ERR_CUDA;
}

// N-tile width for a GEMM with `ncols` columns: the smallest of 64 / 128 / 256 covering it
int pick_bn(int ncols) { return ncols <= 64 ? 64 : (ncols <= 128 ? 128 : 256); }

int num_sms() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
            n = 152;
    }
    return n;
}

template <int BN>
iq_status launch_p(const CUtensorMap& map, const TcP& p, int nsplit, const int8_t* xa,
                   const int8_t* xb, int32_t* out32, long long* out64, unsigned long long* s1,
                   int* hi, int* lo, int* err, cudaStream_t st) {
    IQ_CUDA_CHECK(cudaFuncSetAttribute(k_conv_tcp<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg<BN>::SMEM));
    TileGrid g;
    g.mt = (int)((p.M + BM - 1) / BM);
    g.nt = (p.ncols + BN - 1) / BN;
    g.ns = nsplit;
    g.total = g.mt * g.nt * g.ns;
    const int grid = g.total < num_sms() ? g.total : num_sms();
    kt_pre(st);
    k_conv_tcp<BN><<<grid, THREADS_P, Cfg<BN>::SMEM, st>>>(map, p, g, xa, xb, out32, out64, s1, hi,
                                                          lo, err);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_CONV_GATHER);
    return IQ_OK;
}

template <int BN>
iq_status launch_q(const CUtensorMap& map, const TcP& p, const int8_t* xa, int32_t* out32,
                   long long* out64, unsigned long long* s1, int* hi, int* lo, int* err,
                   cudaStream_t st) {
    IQ_CUDA_CHECK(cudaFuncSetAttribute(k_conv_tcq<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       CfgQ<BN>::SMEM));
    TileGrid g;
    g.mt = (int)((p.M + BM - 1) / BM);
    g.nt = (p.ncols + BN - 1) / BN;
    g.ns = 1;
    g.total = g.mt * g.nt;
    const int grid = g.total < num_sms() ? g.total : num_sms();
    kt_pre(st);
    k_conv_tcq<BN><<<grid, THREADS_Q, CfgQ<BN>::SMEM, st>>>(map, p, g, xa, out32, out64, s1, hi, lo,
                                                           err);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_CONV_CPASYNC);
    return IQ_OK;
}

iq_status launch(const CUtensorMap& map, const TcP& p, int nsplit, const int8_t* xa,
                 const int8_t* xb, int32_t* out32, long long* out64, unsigned long long* s1,
                 int* hi, int* lo, int* err, cudaStream_t st) {
    if (p.mode == MODE_FWD && nsplit == 1 && p.tap_mode && p.cstride % 16 == 0 &&
        p.cofs % 16 == 0 && ((uintptr_t)xa & 15) == 0) {
        switch (pick_bn(p.ncols)) {
            case 64: return launch_q<64>(map, p, xa, out32, out64, s1, hi, lo, err, st);
            case 128: return launch_q<128>(map, p, xa, out32, out64, s1, hi, lo, err, st);
            default: return launch_q<256>(map, p, xa, out32, out64, s1, hi, lo, err, st);
        }
    }
    switch (pick_bn(p.ncols)) {
        case 64: return launch_p<64>(map, p, nsplit, xa, xb, out32, out64, s1, hi, lo, err, st);
        case 128: return launch_p<128>(map, p, nsplit, xa, xb, out32, out64, s1, hi, lo, err, st);
        default: return launch_p<256>(map, p, nsplit, xa, xb, out32, out64, s1, hi, lo, err, st);
    }
}

// Tile rectangle for the TMA-fed kernels: BW x BH = npix output pixels; the shape with the
// least padding waste, if that waste is small.
bool pick_tma_tile(int P, int Q, TmaTile* t, double min_util = 0.8, int npix = 128) {
    double best = 0.0;
    for (int BW = npix; BW >= 16; BW /= 2) {
        const int BH = npix / BW;
        const int PT = (P + BH - 1) / BH, QT = (Q + BW - 1) / BW;
        const double util = (double)P * Q / ((double)PT * BH * QT * BW);
        if (util > best + 1e-9) {
            best = util;
            t->BW = BW; t->BH = BH; t->PT = PT; t->QT = QT;
        }
    }
    return best >= min_util;
}

// 4-D map over the fp16 carriers [N][H][W][cstride]: box 64 channels x BW x BH pixels at
// the conv strides (element strides), 128-byte swizzle, zero fill outside the tensor
iq_status encode_acts16(const __half* xf, int N, int H, int W, int cstride, const TmaTile& t,
                        int sh, int sw, CUtensorMap* map) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
    if (!enc) return IQ_ERR_UNSUPPORTED;
    cuuint64_t gdim[4] = {(cuuint64_t)cstride, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t gstride[3] = {(cuuint64_t)cstride * 2, (cuuint64_t)W * cstride * 2,
                             (cuuint64_t)H * W * cstride * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)(t.BW * sw), (cuuint32_t)(t.BH * sh), 1};
    cuuint32_t estr[4] = {1, (cuuint32_t)sw, (cuuint32_t)sh, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, (void*)xf, gdim, gstride, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? IQ_OK : IQ_ERR_CUDA;
}

// 4-D map over the int32 output [N][P][Q][ncols] for the epilogue's TMA stores: box 16
// channels x min(BW, 32) x 32 / min(BW, 32) pixels (one warp's 32 tile rows), 64-byte
// swizzle.  Needs ncols % 4 == 0 and a 16-byte-aligned base.
iq_status encode_out32(int32_t* out, int N, int P, int Q, int ncols, const TmaTile& t,
                       CUtensorMap* map) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
    if (!enc || ncols % 4 || ((uintptr_t)out & 15) || t.BW < 16 || 32 % (t.BW < 32 ? t.BW : 32))
        return IQ_ERR_UNSUPPORTED;
    const int bw = t.BW < 32 ? t.BW : 32;
    cuuint64_t gdim[4] = {(cuuint64_t)ncols, (cuuint64_t)Q, (cuuint64_t)P, (cuuint64_t)N};
    cuuint64_t gstride[3] = {(cuuint64_t)ncols * 4, (cuuint64_t)Q * ncols * 4,
                             (cuuint64_t)P * Q * ncols * 4};
    cuuint32_t box[4] = {16, (cuuint32_t)bw, (cuuint32_t)(32 / bw), 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_INT32, 4, (void*)out, gdim, gstride, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                     CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? IQ_OK : IQ_ERR_UNSUPPORTED;
}

// 5-D map over the fp16 carriers [N][H][W][cstride] with the channels split into 64-wide
// blocks: dims (64 channels, W, H, cstride / 64 blocks, N), box 64 x BW x BH pixels (at the
// conv strides) x nb blocks, so one load lands nb MN-major blocks of BW BH rows, 8192 bytes
// apart when BW BH = 64.  cstride % 64 == 0.
iq_status encode_acts16_blocks(const __half* xf, int N, int H, int W, int cstride,
                               const TmaTile& t, int sh, int sw, int nb, CUtensorMap* map) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
    if (!enc || cstride % 64) return IQ_ERR_UNSUPPORTED;
    cuuint64_t gdim[5] = {64, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)(cstride / 64),
                          (cuuint64_t)N};
    cuuint64_t gstride[4] = {(cuuint64_t)cstride * 2, (cuuint64_t)W * cstride * 2, 128,
                             (cuuint64_t)H * W * cstride * 2};
    cuuint32_t box[5] = {64, (cuuint32_t)(t.BW * sw), (cuuint32_t)(t.BH * sh), (cuuint32_t)nb,
                         1};
    cuuint32_t estr[5] = {1, (cuuint32_t)sw, (cuuint32_t)sh, 1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 5, (void*)xf, gdim, gstride, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? IQ_OK : IQ_ERR_CUDA;
}

bool tma16_disabled() {
    const char* e = getenv("IQ_TC_GATHER");
    return e && e[0] == '1';
}

// Whether the all-TMA kernel takes this problem (whole 64-channel k-blocks, strides 1 or
// 2, aligned slices, a rectangle tiling with little waste)
bool tma16_ok(const TcP& p, TmaTile* t) {
    if (tma16_disabled() || !p.tap_mode || p.sh > 2 || p.sw > 2 || (p.cstride % 8) ||
        (p.cofs % 64) || p.R > 16 || p.S > 16)
        return false;
    if (!pick_tma_tile(p.P, p.Q, t, 0.6)) return false;
    return t->BW * p.sw <= 256 && t->BH * p.sh <= 256;
}

template <int BN>
iq_status launch_t(const CUtensorMap& wmap, const CUtensorMap& amap, const CUtensorMap& omap,
                   const TcP& p, const TmaTile& t, int32_t* out32, long long* out64,
                   unsigned long long* s1, int* hi, int* lo, int* err, cudaStream_t st) {
    IQ_CUDA_CHECK(cudaFuncSetAttribute(k_conv_tct<BN, false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, CfgT<BN>::SMEM));
    RectGrid g;
    g.PT = t.PT; g.QT = t.QT; g.BW = t.BW; g.BH = t.BH;
    g.mt = p.N * t.PT * t.QT;
    g.nt = (p.ncols + BN - 1) / BN;
    g.total = g.mt * g.nt * (p.slices > 1 ? p.slices : 1);
    g.nb = 1;
    const int grid = g.total < num_sms() ? g.total : num_sms();
    kt_pre(st);
    k_conv_tct<BN, false><<<grid, THREADS_T, CfgT<BN>::SMEM, st>>>(wmap, amap, omap, p, g, out32,
                                                                  out64, s1, hi, lo, err);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_CONV_PIXEL_MAJOR);
    return IQ_OK;
}

// whether a BH x BW tile of the P x Q output (tiles of the tiling t) can skip a tap: some
// tile row band or column band misses the image for some tap
// (fills the band masks of q; false when no tile can skip, or there are over 64 bands)
bool taps_skippable(TcP& q, const TmaTile& t) {
    if ((q.R <= 1 && q.S <= 1) || t.PT > 64 || t.QT > 64) return false;
    bool any = false;
    for (int pt = 0; pt < t.PT; pt++) {
        const int p0 = pt * t.BH, pe = std::min(p0 + t.BH, q.P) - 1;
        uint32_t m = 0;
        for (int r = 0; r < q.R; r++)
            if (tap_meets(q.H, p0, pe, q.sh, r * q.dh - q.ph)) m |= 1u << r;
        q.band_r[pt] = m;
        any |= m != (1u << q.R) - 1u;
    }
    for (int qt = 0; qt < t.QT; qt++) {
        const int q0 = qt * t.BW, qe = std::min(q0 + t.BW, q.Q) - 1;
        uint32_t m = 0;
        for (int s = 0; s < q.S; s++)
            if (tap_meets(q.W, q0, qe, q.sw, s * q.dw - q.pw)) m |= 1u << s;
        q.band_s[qt] = m;
        any |= m != (1u << q.S) - 1u;
    }
    return any;
}

// widen the input codes into xf and run the all-TMA kernel; *used = false when not taken
iq_status try_launch_t(const CUtensorMap& wmap, const TcP& p, const int8_t* x, __half* xf,
                       bool convert, int32_t* out32, long long* out64, unsigned long long* s1,
                       int* hi, int* lo, int* err, cudaStream_t st, bool* used) {
    *used = false;
    TmaTile t;
    if (!xf || !tma16_ok(p, &t)) return IQ_OK;
    if (convert) {
        const int64_t n16 = (int64_t)p.N * p.H * p.W * p.cstride / 16;
        kt_pre(st);
        k_codes_to_f16<<<grid_for(n16), kThreads, 0, st>>>(x, xf, n16);
        kt_post_bytes(st, IQ_KERNEL_CODES_TO_F16, 48.0 * (double)(n16));
        IQ_LAUNCH_CHECK();
    }
    CUtensorMap amap, omap;
    iq_status r = encode_acts16(xf, p.N, p.H, p.W, p.cstride, t, p.sh, p.sw, &amap);
    if (r != IQ_OK) return r;
    TcP q = p;
    q.skip_taps = taps_skippable(q, t);
    // int32 output with statistics: TMA stores of the warps' pixel boxes
    q.tma_out = p.out == OUT_STATS && out32 && p.slices <= 1 &&
                encode_out32(out32, p.N, p.P, p.Q, p.ncols, t, &omap) == IQ_OK;
    if (!q.tma_out) omap = amap;    // not read
    switch (pick_bn(p.ncols)) {
        case 64: r = launch_t<64>(wmap, amap, omap, q, t, out32, out64, s1, hi, lo, err, st); break;
        case 128: r = launch_t<128>(wmap, amap, omap, q, t, out32, out64, s1, hi, lo, err, st); break;
        default: r = launch_t<256>(wmap, amap, omap, q, t, out32, out64, s1, hi, lo, err, st); break;
    }
    if (r == IQ_OK) *used = true;
    return r;
}

// Whether the channel-major kernel takes this problem (at most 128 output channels, whole
// 64-channel k-blocks, strides 1 or 2, aligned slices, a 256-pixel rectangle tiling with
// little waste)
bool cm_ok(const TcP& p, TmaTile* t) {
    if (p.ncols > CM_CH || tma16_disabled() || !p.tap_mode || p.sh > 2 || p.sw > 2 ||
        (p.cstride % 8) || (p.cofs % 64) || p.R > 16 || p.S > 16)
        return false;
    if (!pick_tma_tile(p.P, p.Q, t, 0.6, CM_PIX)) return false;
    return t->BW * p.sw <= 256 && t->BH * p.sh <= 256;
}

// the channel-major kernel for problems with at most 128 output channels and int32 output
// with statistics (wf: the fp16 weights [rows][kpad]); *used = false when not taken
iq_status try_launch_c(const __half* wf, int rows, const TcP& p, const int8_t* x, __half* xf,
                       bool convert, int32_t* out32, unsigned long long* s1, int* hi, int* lo,
                       int* err, cudaStream_t st, bool* used) {
    *used = false;
    TmaTile t;
    if (!xf || !out32 || !s1 || !cm_ok(p, &t)) return IQ_OK;
    CUtensorMap wmap, amap;
    if (encode_weights(wf, rows, p.kpad, CM_CH, &wmap) != IQ_OK) return IQ_OK;
    if (encode_acts16(xf, p.N, p.H, p.W, p.cstride, t, p.sh, p.sw, &amap) != IQ_OK) return IQ_OK;
    if (convert) {
        const int64_t n16 = (int64_t)p.N * p.H * p.W * p.cstride / 16;
        kt_pre(st);
        k_codes_to_f16<<<grid_for(n16), kThreads, 0, st>>>(x, xf, n16);
        kt_post_bytes(st, IQ_KERNEL_CODES_TO_F16, 48.0 * (double)(n16));
        IQ_LAUNCH_CHECK();
    }
    IQ_CUDA_CHECK(cudaFuncSetAttribute(k_conv_tcc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       CfgT<256>::SMEM));
    RectGrid g;
    g.PT = t.PT; g.QT = t.QT; g.BW = t.BW; g.BH = t.BH;
    g.mt = p.N * t.PT * t.QT;
    g.nt = (p.ncols + CM_CH - 1) / CM_CH;
    g.total = g.mt * g.nt;
    g.nb = 1;
    int bw_log2 = 0;
    while ((1 << bw_log2) < t.BW) bw_log2++;
    const int grid = g.total < num_sms() ? g.total : num_sms();
    TcP pc = p;
    pc.skip_taps = taps_skippable(pc, t);
    kt_pre(st);
    k_conv_tcc<<<grid, THREADS_T, CfgT<256>::SMEM, st>>>(wmap, amap, pc, g, bw_log2, out32, s1,
                                                          hi, lo, err);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_CONV_CHANNEL_MAJOR);
    *used = true;
    return IQ_OK;
}

void fill_geom(TcP& p, const iq_conv_desc* d) {
    p.N = d->n; p.H = d->h; p.W = d->w; p.C = d->c; p.K = d->k; p.R = d->r; p.S = d->s;
    p.sh = d->stride_h; p.sw = d->stride_w; p.ph = d->pad_h; p.pw = d->pad_w;
    p.dh = d->dil_h; p.dw = d->dil_w;
    p.P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    p.Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    p.cstride = d->c;
    p.cofs = 0;
    p.slices = 1;
    p.slice_rows = 0;
    p.st_mask = TC_STATS_SUM | TC_STATS_LO;
    p.tma_out = 0;
    p.skip_taps = 0;
}

// k-blocks per split so that each split's int32 running sum cannot overflow
constexpr int MAX_KB_INT32 = 133120 / 64;   // 2080 k-blocks: 133120 * 127^2 < 2^31

}  // namespace

// the sticky device status word of the current context (iq_device_status reads it)
int* device_status_ptr() { return tc_status_ptr(); }

// streaming multiprocessors of the current device
int device_sms() { return num_sms(); }

// 2-D tensor map of a row-major [m][C] array of 1- or 2-byte elements: box {box_c channels,
// box_r rows}, no swizzle, zero fill outside the array
iq_status encode_rows_2d(const void* base, int esz, int64_t m, int C, int box_c, int box_r,
                         CUtensorMap* map) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
    if (!enc || (esz != 1 && esz != 2)) return IQ_ERR_UNSUPPORTED;
    cuuint64_t gdim[2] = {(cuuint64_t)C, (cuuint64_t)m};
    cuuint64_t gstride[1] = {(cuuint64_t)C * esz};
    cuuint32_t box[2] = {(cuuint32_t)box_c, (cuuint32_t)box_r};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, esz == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_UINT16,
                     2, const_cast<void*>(base), gdim, gstride, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? IQ_OK : IQ_ERR_CUDA;
}

// ================================================================ forward

// fp16 weights, a reserved 256-byte slot, then the fp16 carriers of the input
static size_t acts16_offset(size_t wbytes) { return (wbytes + 256 + 255) / 256 * 256; }

// inputs with few channels (C % 64 != 0, R S C <= 512) go through an fp16 im2col
constexpr int IM2COL_MAX_K = 512;

iq_status codes_to_f16(const int8_t* x, __half* xf, int64_t n, cudaStream_t st) {
    if (n % 16 || (((uintptr_t)x | (uintptr_t)xf) & 15)) return IQ_ERR_INVALID_ARG;
    if (n == 0) return IQ_OK;
    kt_pre(st);
    k_codes_to_f16<<<grid_for(n / 16), kThreads, 0, st>>>(x, xf, n / 16);
    kt_post_bytes(st, IQ_KERNEL_CODES_TO_F16, 48.0 * (double)(n / 16));
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

// A stride-1, unpadded 1 x 1 convolution treats every pixel alike, so its N x H x W pixels
// can run as one image of 1 x (N H W) pixels -- the same memory layout for the input, the
// errors and the output.  The rectangle tilings then take runs of 128 (256, 64) consecutive
// pixels and waste none at the image borders (at 65 x 65, 128-pixel rectangles of one
// image cover 27% padding).  Returns d itself when the convolution is not of that kind.
static const iq_conv_desc* flat_pointwise(const iq_conv_desc* d, iq_conv_desc* tmp) {
    if (d->r != 1 || d->s != 1 || d->stride_h != 1 || d->stride_w != 1 || d->pad_h || d->pad_w)
        return d;
    const int64_t pix = (int64_t)d->n * d->h * d->w;
    if (pix > INT_MAX || (d->n == 1 && d->h == 1)) return d;
    *tmp = *d;
    tmp->n = 1;
    tmp->h = 1;
    tmp->w = (int32_t)pix;
    return tmp;
}

// ---------------------------------------------------------------- channel sums from the input
// With batch norm the forward needs S1[k] = the sum over every output pixel of acc[.][k].  In
// the pixel-major kernel that is a reduction across the lanes of the epilogue, about half the
// time of a 1x1 layer; for a 1x1 convolution without padding it follows exactly from the
// input instead: S1[k] = sum_c W[k][c] S_A[c], S_A[c] the sum of x[n][h][w][c] over the input
// pixels the output pixels read (h = p sh, w = q sw).  Taken where the output has at least
// twice the elements of the input (the expanding 1x1 layers), where reading the int8 input
// costs a small fraction of the epilogue reduction it replaces.

bool input_sums_ok(const iq_conv_desc* d) {
    return d->r == 1 && d->s == 1 && d->pad_h == 0 && d->pad_w == 0 && d->groups == 1 &&
           d->c % 4 == 0 && (int64_t)d->k * ((d->h - 1) / d->stride_h + 1) *
                                    ((d->w - 1) / d->stride_w + 1) >= 2LL * d->c * d->h * d->w;
}

// S_A[c] += the sum of x over the sampled pixels: thread t owns channels 4 (t % C4) and a row
// lane of the pixels; the block's lanes combine in shared memory, then one atomic per channel
__global__ void __launch_bounds__(kThreads) k_input_colsums(const int8_t* __restrict__ x, int N,
                                                            int H, int W, int C, int P, int Q,
                                                            int sh, int sw,
                                                            long long* __restrict__ SA) {
    __shared__ long long sh_s[kThreads * 4];
    const int C4 = C >> 2;
    const int lanes = blockDim.x / C4;                  // blockDim.x % C4 == 0 (host)
    const int g = threadIdx.x % C4, rl = threadIdx.x / C4;
    const int64_t npix = (int64_t)N * P * Q;
    const int64_t step = (int64_t)gridDim.x * lanes;
    int a[4] = {0, 0, 0, 0};
    long long acc[4] = {0, 0, 0, 0};
    int cnt = 0;
    for (int64_t m = (int64_t)blockIdx.x * lanes + rl; m < npix; m += step) {
        const int q = (int)(m % Q);
        const int64_t np = m / Q;
        const int pp = (int)(np % P), n = (int)(np / P);
        const uint32_t v = __ldg(reinterpret_cast<const uint32_t*>(
                                     x + (((int64_t)n * H + (int64_t)pp * sh) * W + (int64_t)q * sw) * C) + g);
        a[0] += (int)(int8_t)v; a[1] += (int)(int8_t)(v >> 8);
        a[2] += (int)(int8_t)(v >> 16); a[3] += (int)(int8_t)(v >> 24);
        if (++cnt == 1 << 20) {                          // |partial| < 2^27
#pragma unroll
            for (int j = 0; j < 4; j++) { acc[j] += a[j]; a[j] = 0; }
            cnt = 0;
        }
    }
#pragma unroll
    for (int j = 0; j < 4; j++) sh_s[rl * C + 4 * g + j] = acc[j] + a[j];
    __syncthreads();
    for (int c = threadIdx.x; c < C; c += blockDim.x) {
        long long t = 0;
        for (int i = 0; i < lanes; i++) t += sh_s[i * C + c];
        if (t) atomicAdd(reinterpret_cast<unsigned long long*>(SA + c), (unsigned long long)t);
    }
}

// S1[k] = sum_c S_A[c] W[k][c] (one warp per output channel)
__global__ void k_input_gemv(const long long* __restrict__ SA, const int8_t* __restrict__ w, int K,
                             int C, unsigned long long* __restrict__ s1) {
    const int k = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (k >= K) return;                              // whole warps leave together
    const int8_t* wk = w + (int64_t)k * C;
    long long a = 0;
    for (int j = lane; j < C; j += 32) a += SA[j] * (long long)wk[j];
#pragma unroll
    for (int o = 16; o; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
    if (lane == 0) s1[k] = (unsigned long long)a;
}

// scratch of the input-side sums (S_A)
size_t input_sums_bytes(const iq_conv_desc* d) { return (size_t)d->c * 8 + 256; }

iq_status input_sums(const iq_conv_desc* d, const int8_t* x, const int8_t* w, char* scratch,
                     unsigned long long* s1, cudaStream_t st) {
    const int P = (d->h - 1) / d->stride_h + 1, Q = (d->w - 1) / d->stride_w + 1;
    long long* SA = reinterpret_cast<long long*>(scratch);
    IQ_CUDA_CHECK(cudaMemsetAsync(SA, 0, (size_t)d->c * sizeof(long long), st));
    const int C4 = d->c / 4;
    // a block is kThreads / C4 pixel lanes of all channels (C4 <= kThreads, dividing it), or
    // for wider rows the general mapping does not apply
    if (C4 > kThreads || kThreads % C4) return IQ_ERR_UNSUPPORTED;
    const int lanes = kThreads / C4;
    int64_t blocks = ((int64_t)d->n * P * Q + lanes * 16 - 1) / (lanes * 16);
    if (blocks > 152 * 8) blocks = 152 * 8;
    if (blocks < 1) blocks = 1;
    k_input_colsums<<<(unsigned)blocks, kThreads, 0, st>>>(x, d->n, d->h, d->w, d->c, P, Q,
                                                           d->stride_h, d->stride_w, SA);
    IQ_LAUNCH_CHECK();
    k_input_gemv<<<(unsigned)(((int64_t)d->k * 32 + kThreads - 1) / kThreads), kThreads, 0, st>>>(
        SA, w, d->k, d->c, s1);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

// bytes of the fp16 copy of the input (or of its im2col) in the forward's workspace
size_t conv_fwd_xf_bytes(const iq_conv_desc* d) {
    int64_t kdim = (int64_t)d->r * d->s * (d->c / d->groups);
    int64_t kpad = (kdim + 63) / 64 * 64;
    size_t xb = (size_t)d->n * d->h * d->w * d->c * 2;
    if (d->c % 64 != 0 && kpad <= IM2COL_MAX_K) {
        const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
        const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
        const size_t ib = (size_t)d->n * P * Q * kpad * 2;
        if (ib > xb) xb = ib;
    }
    return xb;
}

size_t conv_fwd_tc_ws_bytes(const iq_conv_desc* d) {
    int64_t kdim = (int64_t)d->r * d->s * (d->c / d->groups);
    int64_t kpad = (kdim + 63) / 64 * 64;
    const size_t wb = (size_t)(d->k * kpad * 2);
    size_t xb = (size_t)d->n * d->h * d->w * d->c * 2;
    if (d->c % 64 != 0 && kpad <= IM2COL_MAX_K) {
        const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
        const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
        const size_t ib = (size_t)d->n * P * Q * kpad * 2;
        if (ib > xb) xb = ib;
    }
    return (acts16_offset(wb) + xb + 511) / 256 * 256 + input_sums_bytes(d);
}

bool conv_fwd_tc_supported(const iq_conv_desc* d) {
    if (tc_env_disabled()) return false;
    return d->groups == 1 && d->c % 4 == 0 && d->k % 8 == 0;
}

iq_status conv_fwd_tc(const iq_conv_desc* d, const int8_t* x, const int8_t* w, int32_t* acc,
                      unsigned long long* s1, int* hi, int* lo, void* ws, cudaStream_t st,
                      bool* done, const __half* xf_given, unsigned st_mask) {
    *done = false;
    if (!conv_fwd_tc_supported(d) || ((uintptr_t)x & 15) != 0 || !get_encode()) return IQ_OK;
    const iq_conv_desc* d0 = d;
    iq_conv_desc dflat;
    d = flat_pointwise(d, &dflat);
    TcP p;
    fill_geom(p, d);
    p.mode = MODE_FWD;
    p.out = OUT_STATS;
    p.M = (int64_t)p.N * p.P * p.Q;
    p.ncols = p.K;
    p.kdim = d->r * d->s * d->c;
    p.st_mask = (int)(st_mask & (TC_STATS_SUM | TC_STATS_LO | TC_STATS_NOEXT)) |
                (p.kdim <= 4095 ? ST_SUM32 : 0);
    if (!(st_mask & TC_STATS_SUM)) p.st_mask |= ST_GMAX;   // no batch norm: one scale only
    p.kpad = (p.kdim + 63) / 64 * 64;
    p.tap_mode = (d->c % 64) == 0;
    p.nkb_total = p.kpad / 64;
    p.kb_per_split = p.nkb_total;
    p.npq = 0;
    if (p.nkb_total > MAX_KB_INT32) return IQ_OK;   // cannot happen under the CRS bound
    // for an expanding 1x1 layer the pixel-major kernel leaves the channel sums to input_sums
    // (the other kernels, and other layers, take them from their epilogues)
    const bool in_sums = (st_mask & TC_STATS_SUM) != 0 && input_sums_ok(d0) &&
                         d0->c / 4 <= kThreads && kThreads % (d0->c / 4) == 0;
    TcP pt = p;
    if (in_sums) pt.st_mask &= ~(int)TC_STATS_SUM;
    char* wsb = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    __half* wf = reinterpret_cast<__half*>(wsb);
    int* err = tc_status_ptr();
    if (!err) return IQ_ERR_CUDA;
    k_widen_weights<<<dim3((unsigned)((p.kpad / 8 + kThreads - 1) / kThreads),
                           (unsigned)(p.K < 65535 ? p.K : 65535)),
                      kThreads, 0, st>>>(w, wf, p.K, p.kdim, p.kpad);
    IQ_LAUNCH_CHECK();
    CUtensorMap map;
    iq_status r = encode_weights(wf, p.K, p.kpad, pick_bn(p.ncols), &map);
    if (r != IQ_OK) return r;
    __half* xf = reinterpret_cast<__half*>(wsb + acts16_offset((size_t)p.K * p.kpad * 2));
    bool used = false, via_t = false;
    if (!p.tap_mode && p.kpad <= IM2COL_MAX_K && p.C % 4 == 0 && p.cstride % 4 == 0 &&
        p.cofs % 4 == 0 && !tma16_disabled() && p.N <= 65535 && p.P <= 65535) {
        // few input channels: the fp16 im2col, then a 1x1 problem over kpad channels
        TcP q = p;
        q.H = p.P; q.W = p.Q; q.C = p.kpad; q.cstride = p.kpad; q.cofs = 0;
        q.R = q.S = 1; q.sh = q.sw = 1; q.ph = q.pw = 0; q.dh = q.dw = 1;
        q.kdim = p.kpad; q.tap_mode = 1;
        TmaTile tt;
        const bool cm = cm_ok(q, &tt);
        if (cm || tma16_ok(q, &tt)) {
            launch_im2col(x, p, xf, st);
            IQ_LAUNCH_CHECK();
            if (cm) {
                r = try_launch_c(wf, p.K, q, nullptr, xf, false, acc, s1, hi, lo, err, st, &used);
                if (r != IQ_OK) return r;
            }
            if (!used) {
                TcP qt = q;
                qt.st_mask = pt.st_mask;
                r = try_launch_t(map, qt, nullptr, xf, false, acc, nullptr, s1, hi, lo, err, st,
                                 &used);
                if (r != IQ_OK) return r;
                via_t = used;
            }
        }
    }
    if (!used && (p.N * (int64_t)p.H * p.W * p.cstride) % 16 == 0) {
        // the fp16 carrier of x: the caller's copy, or converted into the workspace
        __half* xc = xf_given ? const_cast<__half*>(xf_given) : xf;
        const bool convert = xf_given == nullptr;
        r = try_launch_c(wf, p.K, p, x, xc, convert, acc, s1, hi, lo, err, st, &used);
        if (r != IQ_OK) return r;
        if (!used) {
            r = try_launch_t(map, pt, x, xc, convert, acc, nullptr, s1, hi, lo, err, st, &used);
            via_t = used;
        }
        if (r != IQ_OK) return r;
    }
    if (!used) r = launch(map, p, 1, x, nullptr, acc, nullptr, s1, hi, lo, err, st);
    if (r == IQ_OK && via_t && in_sums) {
        char* scratch = wsb + (acts16_offset((size_t)p.K * p.kpad * 2) +
                               conv_fwd_xf_bytes(d0) + 511) / 256 * 256;
        r = input_sums(d0, x, w, scratch, s1, st);
    }
    if (r == IQ_OK) *done = true;
    return r;
}

// ================================================================ data gradient (stride 1)
// dx = conv(e, w') with w'[c][r][s][k] = w[k][R-1-r][S-1-s][c], pad' = dil (R-1) - pad.
// When (K R S) 127^2 could overflow int32 the reduction is split over channel slices of e
// whose int32 partial results are added in int64.

int conv_dgrad_tc_slices(const iq_conv_desc* d) {
    int nsl = 1;
    while (nsl <= d->k &&
           ((int64_t)(d->k / nsl) * d->r * d->s * 16129 >= (int64_t(1) << 31) || (d->k % nsl) ||
            ((d->k / nsl) % 4)))
        nsl++;
    return nsl <= d->k ? nsl : 0;
}

size_t conv_dgrad_tc_ws_bytes(const iq_conv_desc* d) {
    int nsl = conv_dgrad_tc_slices(d);
    if (nsl < 1) nsl = 1;
    int64_t kpad = ((int64_t)d->r * d->s * (d->k / nsl) + 63) / 64 * 64;
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    const size_t wb = (size_t)nsl * d->c * kpad * 2;    // every slice's widened weights
    return acts16_offset(wb) + (size_t)d->n * P * Q * d->k * 2 + 512;
}

bool conv_dgrad_tc_supported(const iq_conv_desc* d) {
    if (tc_env_disabled()) return false;
    if (d->groups != 1 || d->stride_h != 1 || d->stride_w != 1) return false;
    if (d->k % 4 || d->c % 8) return false;
    if (d->dil_h * (d->r - 1) < d->pad_h || d->dil_w * (d->s - 1) < d->pad_w) return false;
    return conv_dgrad_tc_slices(d) >= 1;
}

iq_status conv_dgrad_tc(const iq_conv_desc* d, const int8_t* e, const int8_t* w, int32_t* out32,
                        long long* out64, unsigned long long* s1, int* hi, int* lo, void* ws,
                        cudaStream_t st, bool* done, const __half* ef_given) {
    *done = false;
    if (!conv_dgrad_tc_supported(d) || ((uintptr_t)e & 15) != 0 || !get_encode()) return IQ_OK;
    iq_conv_desc dflat;
    d = flat_pointwise(d, &dflat);
    const int nsl = conv_dgrad_tc_slices(d);
    if (nsl > 1 && !out64) return IQ_OK;
    if (nsl == 1 && !out32) return IQ_OK;
    iq_conv_desc g = *d;   // the forward problem over the errors
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    g.h = P; g.w = Q; g.c = d->k; g.k = d->c;
    g.pad_h = d->dil_h * (d->r - 1) - d->pad_h;
    g.pad_w = d->dil_w * (d->s - 1) - d->pad_w;
    const int kc = d->k / nsl;
    TcP p;
    fill_geom(p, &g);
    p.C = kc;                 // channels per slice
    p.cstride = d->k;
    p.mode = MODE_FWD;
    p.out = nsl == 1 ? OUT_STATS : OUT_ATOMIC64;
    p.M = (int64_t)d->n * d->h * d->w;
    p.ncols = d->c;
    p.kdim = d->r * d->s * kc;
    p.st_mask = TC_STATS_LO | ST_GMAX;   // the requantizer of dx reads the extremes only
    p.kpad = (p.kdim + 63) / 64 * 64;
    p.tap_mode = (kc % 64) == 0;
    p.nkb_total = p.kpad / 64;
    p.kb_per_split = p.nkb_total;
    p.npq = 0;
    if (p.P != d->h || p.Q != d->w) return IQ_OK;
    char* wsb = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    __half* wf = reinterpret_cast<__half*>(wsb);
    int* err = tc_status_ptr();
    if (!err) return IQ_ERR_CUDA;
    __half* ef = ef_given ? const_cast<__half*>(ef_given)
                          : reinterpret_cast<__half*>(
                                wsb + acts16_offset((size_t)nsl * d->c * p.kpad * 2));
    const bool convert = ef_given == nullptr;
    const bool ef_ok = ((int64_t)p.N * p.H * p.W * p.cstride) % 16 == 0;
    TmaTile tt;
    if (nsl > 1 && ef_ok && tma16_ok(p, &tt)) {
        // every slice in one launch of the all-TMA kernel: slice sl's weights are rows
        // [sl C, (sl + 1) C) of one matrix, its errors channels [sl kc, (sl + 1) kc)
        for (int sl = 0; sl < nsl; sl++) {
            k_widen_weights_dgrad<<<dim3((unsigned)((d->c + 31) / 32), (unsigned)((kc + 31) / 32),
                                         (unsigned)(d->r * d->s)), dim3(32, 8), 0, st>>>(
                w, wf + (size_t)sl * d->c * p.kpad, d->k, d->r, d->s, d->c, sl * kc, kc, p.kpad);
            IQ_LAUNCH_CHECK();
        }
        CUtensorMap map;
        iq_status r = encode_weights(wf, nsl * d->c, p.kpad, pick_bn(p.ncols), &map);
        if (r != IQ_OK) return r;
        TcP ps = p;
        ps.cofs = 0;
        ps.slices = nsl;
        ps.slice_rows = d->c;
        bool used = false;
        r = try_launch_t(map, ps, e, ef, convert, out32, out64, s1, hi, lo, err, st, &used);
        if (r != IQ_OK) return r;
        if (used) {
            *done = true;
            return IQ_OK;
        }
    }
    for (int sl = 0; sl < nsl; sl++) {
        k_widen_weights_dgrad<<<dim3((unsigned)((d->c + 31) / 32), (unsigned)((kc + 31) / 32),
                                     (unsigned)(d->r * d->s)), dim3(32, 8), 0, st>>>(
            w, wf, d->k, d->r, d->s, d->c, sl * kc, kc, p.kpad);
        IQ_LAUNCH_CHECK();
        CUtensorMap map;
        iq_status r = encode_weights(wf, d->c, p.kpad, pick_bn(p.ncols), &map);
        if (r != IQ_OK) return r;
        p.cofs = sl * kc;
        bool used = false;
        if (ef_ok && nsl == 1) {
            r = try_launch_c(wf, d->c, p, e, ef, convert, out32, s1, hi, lo, err, st, &used);
            if (r != IQ_OK) return r;
        }
        if (ef_ok && !used) {
            r = try_launch_t(map, p, e, ef, convert && sl == 0, out32, out64, s1, hi, lo, err, st,
                             &used);
            if (r != IQ_OK) return r;
        }
        if (!used) r = launch(map, p, 1, e, nullptr, out32, out64, s1, hi, lo, err, st);
        if (r != IQ_OK) return r;
    }
    *done = true;
    return IQ_OK;
}

// ================================================================ stride-2 data gradient
//
// With stride 2 the input pixels split into four phases by the parity of their row and
// column.  Input row h = 2i + a takes the taps r with r dil + a + pad even: p = (h + pad -
// r dil) / 2 = i + o_r.  Those taps form an arithmetic progression (every second tap when dil
// is odd; all or none when dil is even), so phase (a, b) is the stride-1 data gradient of a
// sub-kernel -- the taps of the progression, dilation dil' = step dil / 2, padding
// o_{first tap} -- over the same errors, with ceil((h - a) / 2) rows.  Each phase runs on the
// stride-1 tensor-core path into a scratch tensor that one kernel interleaves into dx; a phase
// that no tap reaches is zero.

namespace {

struct Phase1d {
    int n;        // taps of the phase (0: the phase is zero)
    int first;    // first tap
    int step;     // tap step
    int pad;      // padding of the phase's stride-1 problem
    int dil;      // its dilation
    int len;      // input rows (columns) of the phase
};

Phase1d phase_1d(int extent, int taps, int pad, int dil, int a) {
    Phase1d f;
    f.len = (extent - a + 1) / 2;
    f.step = (dil & 1) ? 2 : 1;
    f.first = (dil & 1) ? ((a + pad) & 1) : 0;
    f.n = 0;
    if (!(dil & 1) && ((a + pad) & 1)) return f;   // even dilation: every tap or none
    for (int r = f.first; r < taps; r += f.step) f.n++;
    f.dil = f.step * dil / 2;
    f.pad = (a + pad - f.first * dil) / 2;          // a + pad - first dil is even
    return f;
}

// wsub[k][t][u][c] = w[k][rf + t rs][sf + u ss][c]
__global__ void k_gather_taps(const int8_t* __restrict__ w, int K, int R, int S, int C, int rf,
                              int rs, int nr, int sf, int ss, int ns, int8_t* __restrict__ wsub) {
    const int64_t n = (int64_t)K * nr * ns * C;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % C);
        int64_t t = i / C;
        const int u = (int)(t % ns);
        t /= ns;
        const int tr = (int)(t % nr);
        const int k = (int)(t / nr);
        wsub[i] = w[(((int64_t)k * R + rf + tr * rs) * S + sf + u * ss) * C + c];
    }
}

// dx[n][2i + a][2j + b][c] = src[n][i][j][c] (src NULL: 0)
__global__ void k_phase_scatter(const int32_t* __restrict__ src, int N, int Ha, int Wb, int C,
                                int H, int W, int a, int b, int32_t* __restrict__ dx) {
    const int64_t n4 = (int64_t)N * Ha * Wb * (C / 4);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c4 = (int)(i % (C / 4));
        int64_t t = i / (C / 4);
        const int j = (int)(t % Wb);
        t /= Wb;
        const int ii = (int)(t % Ha);
        const int nn = (int)(t / Ha);
        const int4 v = src ? reinterpret_cast<const int4*>(src)[i] : make_int4(0, 0, 0, 0);
        reinterpret_cast<int4*>(dx)[(((int64_t)nn * H + 2 * ii + a) * W + 2 * j + b) * (C / 4) + c4] = v;
    }
}

}  // namespace

static bool conv_dgrad_tc_stride2_plan(const iq_conv_desc* d, iq_conv_desc sub[4],
                                       Phase1d* ph = nullptr, Phase1d* pw = nullptr) {
    if (tc_env_disabled()) return false;
    if (d->groups != 1 || d->stride_h != 2 || d->stride_w != 2 || d->c % 4) return false;
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / 2 + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / 2 + 1;
    for (int a = 0; a < 2; a++)
        for (int b = 0; b < 2; b++) {
            const Phase1d fr = phase_1d(d->h, d->r, d->pad_h, d->dil_h, a);
            const Phase1d fs = phase_1d(d->w, d->s, d->pad_w, d->dil_w, b);
            if (ph) ph[2 * a + b] = fr;
            if (pw) pw[2 * a + b] = fs;
            iq_conv_desc& g = sub[2 * a + b];
            g = *d;
            g.stride_h = g.stride_w = 1;
            if (fr.n == 0 || fs.n == 0 || fr.len < 1 || fs.len < 1) {
                g.r = 0;                       // a zero phase
                continue;
            }
            g.h = fr.len; g.w = fs.len;
            g.r = fr.n; g.s = fs.n;
            g.pad_h = fr.pad; g.pad_w = fs.pad;
            g.dil_h = fr.dil; g.dil_w = fs.dil;
            if (g.pad_h < 0 || g.pad_w < 0) return false;
            // the phase's stride-1 problem must read exactly the P x Q errors
            if (g.h + 2 * g.pad_h - g.dil_h * (g.r - 1) != P ||
                g.w + 2 * g.pad_w - g.dil_w * (g.s - 1) != Q)
                return false;
            if (!conv_dgrad_tc_supported(&g) || conv_dgrad_tc_slices(&g) != 1) return false;
        }
    return true;
}

size_t conv_dgrad_tc_stride2_ws_bytes(const iq_conv_desc* d) {
    iq_conv_desc sub[4];
    if (!conv_dgrad_tc_stride2_plan(d, sub)) return 0;
    size_t b = 0;
    for (int i = 0; i < 4; i++)
        if (sub[i].r) b = std::max(b, conv_dgrad_tc_ws_bytes(&sub[i]));
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / 2 + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / 2 + 1;
    const size_t ef = ((size_t)d->n * P * Q * d->k * 2 + 255) / 256 * 256;
    const size_t wsub = ((size_t)d->k * d->r * d->s * d->c + 255) / 256 * 256;
    const size_t scr = ((size_t)d->n * ((d->h + 1) / 2) * ((d->w + 1) / 2) * d->c * 4 + 255) / 256 * 256;
    return b + ef + wsub + scr + 1024;
}

iq_status conv_dgrad_tc_stride2(const iq_conv_desc* d, const int8_t* e, const int8_t* w,
                                int32_t* out32, unsigned long long* s1, int* hi, int* lo,
                                void* ws, size_t ws_bytes, cudaStream_t st, bool* done,
                                const __half* ef_given) {
    *done = false;
    iq_conv_desc sub[4];
    Phase1d ph[4], pw[4];
    if (!conv_dgrad_tc_stride2_plan(d, sub, ph, pw) || !out32 || !s1 || !hi || !lo ||
        ((uintptr_t)e & 15) || !get_encode())
        return IQ_OK;
    if (ws_bytes < conv_dgrad_tc_stride2_ws_bytes(d)) return IQ_ERR_WORKSPACE;
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / 2 + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / 2 + 1;
    const int64_t ne = (int64_t)d->n * P * Q * d->k;
    if (ne % 16) return IQ_OK;
    size_t b = 0;
    for (int i = 0; i < 4; i++)
        if (sub[i].r) b = std::max(b, conv_dgrad_tc_ws_bytes(&sub[i]));
    b = (b + 255) / 256 * 256;
    char* base = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    char* tcws = base;
    __half* ef = reinterpret_cast<__half*>(base + b);
    int8_t* wsub = reinterpret_cast<int8_t*>(base + b + ((size_t)ne * 2 + 255) / 256 * 256);
    int32_t* scr = reinterpret_cast<int32_t*>(
        (char*)wsub + ((size_t)d->k * d->r * d->s * d->c + 255) / 256 * 256);
    if (ef_given) {
        ef = const_cast<__half*>(ef_given);
    } else {
        iq_status r = codes_to_f16(e, ef, ne, st);
        if (r != IQ_OK) return r;
    }
    for (int i = 0; i < 4; i++) {
        const int a = i >> 1, bb = i & 1;
        const int Ha = (d->h - a + 1) / 2, Wb = (d->w - bb + 1) / 2;
        if (Ha < 1 || Wb < 1) continue;
        const int64_t n4 = (int64_t)d->n * Ha * Wb * (d->c / 4);
        if (!sub[i].r) {
            k_phase_scatter<<<grid_for(n4), kThreads, 0, st>>>(nullptr, d->n, Ha, Wb, d->c, d->h,
                                                               d->w, a, bb, out32);
            IQ_LAUNCH_CHECK();
            continue;
        }
        const int64_t nw = (int64_t)d->k * sub[i].r * sub[i].s * d->c;
        k_gather_taps<<<grid_for(nw), kThreads, 0, st>>>(w, d->k, d->r, d->s, d->c, ph[i].first,
                                                         ph[i].step, sub[i].r, pw[i].first,
                                                         pw[i].step, sub[i].s, wsub);
        IQ_LAUNCH_CHECK();
        bool pdone = false;
        iq_status r = conv_dgrad_tc(&sub[i], e, wsub, scr, nullptr, s1, hi, lo, tcws, st, &pdone,
                                    ef);
        if (r != IQ_OK) return r;
        if (!pdone) return IQ_ERR_CUDA;   // the plan admitted every phase
        k_phase_scatter<<<grid_for(n4), kThreads, 0, st>>>(scr, d->n, Ha, Wb, d->c, d->h, d->w, a,
                                                           bb, out32);
        IQ_LAUNCH_CHECK();
    }
    *done = true;
    return IQ_OK;
}

// ================================================================ weight gradient

// a reserved 256-byte slot, then the fp16 carriers of the errors and of the input
namespace {

// the split of nkb k-blocks that minimises (tiles per SM) x (k-blocks per tile) on the
// persistent grid, each split within the int32 bound and at least 16 k-blocks long; a split
// count only wins if it beats every smaller one by more than 10% (each extra split costs a
// partial slab and its sum).  Returns the number of splits, *kbs the k-blocks per split.
int choose_split(int64_t nkb, int64_t tiles, int64_t* kbs_out) {
    const int64_t sms = num_sms();
    int64_t best_cost = INT64_MAX, kbs = MAX_KB_INT32;
    for (int64_t ns = 1; ns <= 256; ns++) {
        const int64_t k = (nkb + ns - 1) / ns;
        if (k > MAX_KB_INT32) continue;
        if (k < 16 && ns > 1) break;
        const int64_t nsr = (nkb + k - 1) / k;
        const int64_t cost = ((tiles * nsr + sms - 1) / sms) * k;
        if (best_cost == INT64_MAX || cost * 10 < best_cost * 9) { best_cost = cost; kbs = k; }
    }
    *kbs_out = kbs;
    return (int)((nkb + kbs - 1) / kbs);
}

bool wgrad_rect(const TcP& p, TmaTile* t);

// the all-TMA weight-gradient plan: geometry, k-block rectangles and splits
bool wgrad_tma_plan(const iq_conv_desc* d, TcP* p, TmaTile* t, int* nsplit) {
    fill_geom(*p, d);
    p->mode = MODE_WGRAD;
    p->M = p->K;
    p->ncols = p->R * p->S * p->C;
    p->npq = (int64_t)p->N * p->P * p->Q;
    p->kdim = 0; p->kpad = 0; p->tap_mode = 1;
    if (d->groups != 1 || p->C % 64 || p->sh > 2 || p->sw > 2) return false;
    if (((int64_t)p->N * p->H * p->W * p->C) % 16) return false;
    if (!wgrad_rect(*p, t)) return false;
    const int64_t nkb = (int64_t)p->N * t->PT * t->QT;
    if (nkb > INT_MAX) return false;
    const int bn = pick_bn(p->ncols);
    const int64_t tiles = ((p->M + BM - 1) / BM) * ((p->ncols + bn - 1) / bn);
    int64_t kbs;
    *nsplit = choose_split(nkb, tiles, &kbs);
    p->nkb_total = (int)nkb;
    p->kb_per_split = (int)kbs;
    return true;
}

}  // namespace

// a reserved 256-byte slot, the fp16 carriers of the errors and of the input, and the per-split
// int32 partial sums of the all-TMA path
// The weight gradient of a convolution with few input channels (C % 4 == 0, C < 64) as that
// of a 1 x 1 convolution over its fp16 im2col (kpad = R S C rounded up to 64 channels per
// output pixel, the forward's im2col layout); false when the shape does not qualify.
bool wgrad_im2col_desc(const iq_conv_desc* d, iq_conv_desc* d2) {
    if (d->groups != 1 || d->c % 4 || d->c >= 64) return false;
    const int kpad = (d->r * d->s * d->c + 63) / 64 * 64;
    if (kpad > IM2COL_MAX_K) return false;
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    if (P > 65535 || d->n > 65535) return false;
    *d2 = *d;
    d2->h = P; d2->w = Q; d2->c = kpad;
    d2->r = d2->s = 1;
    d2->stride_h = d2->stride_w = 1;
    d2->pad_h = d2->pad_w = 0;
    d2->dil_h = d2->dil_w = 1;
    return true;
}

size_t conv_wgrad_tc_ws_bytes(const iq_conv_desc* d) {
    iq_conv_desc dflat;
    d = flat_pointwise(d, &dflat);      // the tiling (and split count) conv_wgrad_tc uses
    const int P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    const int Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    const size_t eb = ((size_t)d->n * P * Q * ((d->k + 63) / 64 * 64) * 2 + 255) / 256 * 256;
    size_t xb = ((size_t)d->n * d->h * d->w * d->c * 2 + 255) / 256 * 256;
    size_t parts = 0;
    TcP p;
    TmaTile t;
    int ns = 1;
    iq_conv_desc d2;
    if (d->c > 0 && d->k > 0 && wgrad_tma_plan(d, &p, &t, &ns)) {
        parts = (size_t)ns * d->k * d->r * d->s * d->c * 4;
    } else if (d->c > 0 && d->k > 0 && wgrad_im2col_desc(d, &d2) &&
               wgrad_tma_plan(&d2, &p, &t, &ns)) {
        xb = ((size_t)d->n * P * Q * d2.c * 2 + 255) / 256 * 256;
        parts = (size_t)ns * d->k * d2.c * 4;
    }
    return 256 + eb + xb + parts + 512;
}

namespace {

// the k-block rectangle of 64 output pixels (BW x BH) that wastes the fewest pixels at the
// image borders
bool wgrad_rect(const TcP& p, TmaTile* t) {
    double best = 0.0;
    for (int BW = 64; BW >= 1; BW /= 2) {
        const int BH = 64 / BW;
        if (BW * p.sw > 256 || BH * p.sh > 256) continue;
        const int PT = (p.P + BH - 1) / BH, QT = (p.Q + BW - 1) / BW;
        const double util = (double)p.P * p.Q / ((double)PT * BH * QT * BW);
        if (util > best + 1e-9) {
            best = util;
            t->BW = BW; t->BH = BH; t->PT = PT; t->QT = QT;
        }
    }
    return best >= 0.5;
}

template <int BN>
iq_status launch_tw(const CUtensorMap& emap, const CUtensorMap& xmap, const TcP& p,
                    const TmaTile& t, int nb, int nsplit, int32_t* part, int* err,
                    cudaStream_t st, unsigned long long* amax = nullptr) {
    IQ_CUDA_CHECK(cudaFuncSetAttribute(k_conv_tct<BN, true>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, CfgT<BN>::SMEM));
    RectGrid g;
    g.PT = t.PT; g.QT = t.QT; g.BW = t.BW; g.BH = t.BH;
    g.mt = (int)((p.M + BM - 1) / BM);
    g.nt = (p.ncols + BN - 1) / BN;
    g.total = g.mt * g.nt * nsplit;
    g.nb = nb < BN / 64 ? nb : BN / 64;
    const int grid = g.total < num_sms() ? g.total : num_sms();
    // (the output map is not read: the weight gradient writes its slabs with plain stores)
    kt_pre(st);
    k_conv_tct<BN, true><<<grid, THREADS_T, CfgT<BN>::SMEM, st>>>(emap, xmap, emap, p, g, part,
                                                                 nullptr, amax, nullptr, nullptr,
                                                                 err);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_CONV_WGRAD);
    return IQ_OK;
}

}  // namespace

bool conv_wgrad_tc_supported(const iq_conv_desc* d) {
    if (tc_env_disabled()) return false;
    return d->groups == 1 && d->c % 16 == 0 && d->k % 16 == 0;
}

// G (int64 KRSC, zeroed by the caller) += E^T im2col(x)
iq_status conv_wgrad_tc(const iq_conv_desc* d, const int8_t* e, const int8_t* x, long long* G,
                        void* ws, cudaStream_t st, bool* done, unsigned long long* amax,
                        bool* amax_done, const __half* ef_given, const __half* xf_given,
                        const int32_t** g32_out) {
    *done = false;
    *amax_done = false;
    if (g32_out) *g32_out = nullptr;
    if (tc_env_disabled() || (((uintptr_t)e | (uintptr_t)x) & 15) != 0) return IQ_OK;
    iq_conv_desc dflat;
    d = flat_pointwise(d, &dflat);
    char* wsb = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    int* err = tc_status_ptr();
    if (!err) return IQ_ERR_CUDA;
    TcP p;
    TmaTile t;
    int nsplit = 1;
    CUtensorMap emap, xmap;
    int nb = 1;
    bool maps = false;
    int Kp = 0;
    size_t eb = 0, xb = 0;
    bool use_ef = false, use_xf = false;   // read the caller's carriers instead of converting
    if (!tma16_disabled() && get_encode() && wgrad_tma_plan(d, &p, &t, &nsplit)) {
        Kp = (p.K + 63) / 64 * 64;            // fp16 error rows padded to whole 64-channel blocks
        eb = ((size_t)p.npq * Kp * 2 + 255) / 256 * 256;
        xb = ((size_t)p.N * p.H * p.W * p.C * 2 + 255) / 256 * 256;
        // channel blocks per im2col box: the tile's columns of one tap in as few boxes as
        // the channel count allows
        nb = p.C % 256 == 0 ? 4 : (p.C % 128 == 0 ? 2 : 1);
        if (nb > pick_bn(p.ncols) / 64) nb = pick_bn(p.ncols) / 64;
        use_ef = ef_given && Kp == p.K;
        use_xf = xf_given != nullptr;
        maps = encode_acts16_blocks(use_ef ? ef_given : reinterpret_cast<__half*>(wsb + 256), p.N,
                                    p.P, p.Q, Kp, t, 1, 1, 2, &emap) == IQ_OK &&
               encode_acts16_blocks(use_xf ? xf_given : reinterpret_cast<__half*>(wsb + 256 + eb),
                                    p.N, p.H, p.W, p.C, t, p.sh, p.sw, nb, &xmap) == IQ_OK;
    }
    // few input channels: the 1 x 1 problem over the im2col of x (pc: the conv's own geometry)
    iq_conv_desc d2;
    bool im2col = false;
    TcP pc;
    if (!maps && !tma16_disabled() && get_encode() && wgrad_im2col_desc(d, &d2) &&
        wgrad_tma_plan(&d2, &p, &t, &nsplit)) {
        Kp = (p.K + 63) / 64 * 64;
        eb = ((size_t)p.npq * Kp * 2 + 255) / 256 * 256;
        xb = ((size_t)p.npq * p.C * 2 + 255) / 256 * 256;
        nb = p.C % 256 == 0 ? 4 : (p.C % 128 == 0 ? 2 : 1);
        if (nb > pick_bn(p.ncols) / 64) nb = pick_bn(p.ncols) / 64;
        use_ef = ef_given && Kp == p.K;
        use_xf = false;
        maps = encode_acts16_blocks(use_ef ? ef_given : reinterpret_cast<__half*>(wsb + 256), p.N,
                                    p.P, p.Q, Kp, t, 1, 1, 2, &emap) == IQ_OK &&
               encode_acts16_blocks(reinterpret_cast<__half*>(wsb + 256 + eb), p.N, p.H, p.W,
                                    p.C, t, 1, 1, nb, &xmap) == IQ_OK;
        im2col = maps;
        fill_geom(pc, d);
        pc.kdim = d->r * d->s * d->c;
        pc.kpad = p.C;
    }
    if (maps) {
        // k-blocks: the pixel rectangles of every image; each split writes its own int32
        // partial sums, added into G afterwards
        const int64_t ne = p.npq * Kp, nx = (int64_t)p.N * p.H * p.W * p.C;
        __half* ef = reinterpret_cast<__half*>(wsb + 256);
        __half* xf = reinterpret_cast<__half*>(wsb + 256 + eb);
        int32_t* part = reinterpret_cast<int32_t*>(wsb + 256 + eb + xb);
        p.out = OUT_PART32;
        if (!use_ef) {
            if (Kp == p.K && ne % 16 == 0) {
                kt_pre(st);
                k_codes_to_f16<<<grid_for(ne / 16), kThreads, 0, st>>>(e, ef, ne / 16);
                kt_post_bytes(st, IQ_KERNEL_CODES_TO_F16, 48.0 * (double)(ne / 16));
            } else {
                k_codes_to_f16_pad<<<grid_for(p.npq * (Kp / 8)), kThreads, 0, st>>>(e, ef, p.npq,
                                                                                  p.K, Kp);
            }
            IQ_LAUNCH_CHECK();
        }
        if (im2col) {
            launch_im2col(x, pc, xf, st);
            IQ_LAUNCH_CHECK();
        } else if (!use_xf) {
            kt_pre(st);
            k_codes_to_f16<<<grid_for(nx / 16), kThreads, 0, st>>>(x, xf, nx / 16);
            kt_post_bytes(st, IQ_KERNEL_CODES_TO_F16, 48.0 * (double)(nx / 16));
            IQ_LAUNCH_CHECK();
        }
        iq_status r = IQ_OK;
        // one split and no column compaction: the int32 slab is the result (max |G| from the
        // epilogue), no int64 copy
        const bool direct = g32_out && nsplit == 1 && !im2col;
        unsigned long long* am = direct ? amax : nullptr;
        switch (pick_bn(p.ncols)) {
            case 64: r = launch_tw<64>(emap, xmap, p, t, nb, nsplit, part, err, st, am); break;
            case 128: r = launch_tw<128>(emap, xmap, p, t, nb, nsplit, part, err, st, am); break;
            default: r = launch_tw<256>(emap, xmap, p, t, nb, nsplit, part, err, st, am); break;
        }
        if (r != IQ_OK) return r;
        if (direct) {
            *g32_out = part;
            *done = true;
            *amax_done = true;
            return IQ_OK;
        }
        if (im2col) {
            const int kdim = d->r * d->s * d->c;
            k_split_sum_cols<<<grid_for(p.M * (int64_t)kdim), kThreads, 0, st>>>(
                part, nsplit, p.M, p.ncols, kdim, G, amax);
        } else {
            const int64_t total4 = p.M * (int64_t)p.ncols / 4;
            k_split_sum<<<grid_for(total4), kThreads, 0, st>>>(part, nsplit, total4, G, amax);
        }
        IQ_LAUNCH_CHECK();
        *done = true;
        *amax_done = true;
        return IQ_OK;
    }
    if (!conv_wgrad_tc_supported(d)) return IQ_OK;
    fill_geom(p, d);
    p.mode = MODE_WGRAD;
    p.out = OUT_ATOMIC64;
    p.M = p.K;
    p.ncols = p.R * p.S * p.C;
    p.npq = (int64_t)p.N * p.P * p.Q;
    p.kdim = 0; p.kpad = 0; p.tap_mode = 1;
    const int64_t nkb = (p.npq + BK - 1) / BK;
    if (nkb > INT_MAX) return IQ_OK;
    const int bn = pick_bn(p.ncols);
    const int64_t tiles = ((p.M + BM - 1) / BM) * ((p.ncols + bn - 1) / bn);
    int64_t kbs;
    nsplit = choose_split(nkb, tiles, &kbs);
    p.nkb_total = (int)nkb;
    p.kb_per_split = (int)kbs;
    CUtensorMap dummy;
    memset(&dummy, 0, sizeof(dummy));
    IQ_CUDA_CHECK(cudaMemsetAsync(G, 0, sizeof(long long) * (size_t)p.M * p.ncols, st));
    iq_status r = launch(dummy, p, nsplit, e, x, nullptr, G, nullptr, nullptr, nullptr, err, st);
    if (r == IQ_OK) *done = true;
    return r;
}

}  // namespace iq

namespace iq {
namespace {
// One thread waits, with the bounded wait of the tensor-core kernels and a limit of `limit`
// SM cycles, on an mbarrier that nothing arrives on; when the wait gives up it records code 5
// in the sticky status, as a kernel whose wait expired does.  The thread issues no copies and
// no MMAs, so nothing is in flight when it returns.
__global__ void k_wait_selftest(int* err, long long limit) {
    __shared__ uint64_t bar;
    __shared__ int never;
    if (threadIdx.x == 0) {
        tc::mbar_init(&bar, 1);
        never = 0;
        tc::mbar_fence_init();
        if (!tc::mbar_wait(&bar, 0, &never, limit)) atomicExch(err, 5);
    }
}
}  // namespace
}  // namespace iq

extern "C" iq_status iq_wait_selftest(long long limit_cycles, iq_stream stream) {
    if (limit_cycles < 0 || limit_cycles > (1LL << 31)) return IQ_ERR_INVALID_ARG;
    int* p = iq::tc_status_ptr();
    if (!p) return IQ_ERR_CUDA;
    iq::k_wait_selftest<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(p, limit_cycles);
    IQ_LAUNCH_CHECK();
    return IQ_OK;
}

extern "C" iq_status iq_device_status(int32_t* code, iq_stream stream) {
    if (!code) return IQ_ERR_INVALID_ARG;
    int* p = iq::tc_status_ptr();
    if (!p) return IQ_ERR_CUDA;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int v = 0;
    IQ_CUDA_CHECK(cudaStreamSynchronize(st));
    IQ_CUDA_CHECK(cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost));
    if (v != 0) IQ_CUDA_CHECK(cudaMemset(p, 0, sizeof(int)));
    *code = v;
    return v != 0 ? IQ_ERR_TIMEOUT : IQ_OK;
}
