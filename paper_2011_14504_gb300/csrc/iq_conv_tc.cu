// iq_conv_tc.cu -- the 8-bit convolution on the 5th-generation tensor cores (tcgen05).
//
// sm_103a has no integer UMMA (`tcgen05.mma .kind::i8` is rejected for this target), so
// the codes travel as fp16 "carriers": every int8 code is exactly representable in fp16,
// every product |a b| <= 127^2 is exact, and fp32 accumulation of at most 1024 such
// products stays below 2^24 and is therefore exact.  The K loop is cut into chunks of
// 1024 (16 k-blocks of 64); each chunk accumulates in its own fp32 TMEM buffer and the
// epilogue folds it into int32 registers, so the result is the exact int32 convolution.
//
// Implicit GEMM: D[M x N] = A[M x K] B[N x K]^T with M = N*P*Q output pixels,
// N = output channels, K = R*S*C taps x channels.  One CTA computes a 128 x 128 tile.
//   warps 0-3  producers: thread t gathers A row t (one output pixel) for each k-block
//              (64 int8 codes, 16-byte loads, zero outside the image), widens them to fp16
//              and stores them in the 128-byte-swizzled K-major UMMA layout; thread 0 also
//              issues the TMA load of the weight tile (pre-widened to fp16 once per call).
//   warp 8     allocates TMEM; lane 0 issues tcgen05.mma (M=128, N=128, K=16) and commits.
//   warps 4-7  epilogue: TMEM -> registers (fp32 -> int32 fold per chunk), then the tile
//              goes through shared memory for per-channel sum/max/min and coalesced stores.
// All mbarrier waits are bounded (about one second); on expiry the CTA records an error
// word, drains what it issued and returns.
#include "iq_conv_tc.cuh"
#include "iq_tc_ptx.cuh"

#include <climits>
#include <cudaTypedefs.h>

namespace iq {

namespace {

constexpr int TC_BM = 128;
constexpr int TC_BN = 128;
constexpr int TC_BK = 64;                  // fp16 elements per k-block = 128 bytes
constexpr int TC_STAGES = 4;
constexpr int TC_CHUNK_KB = 16;            // 16 k-blocks = 1024 products per fp32 chunk
constexpr int TC_A_BYTES = TC_BM * 128;    // 16 KB
constexpr int TC_B_BYTES = TC_BN * 128;    // 16 KB
constexpr int TC_STAGE_BYTES = TC_A_BYTES + TC_B_BYTES;
constexpr int TC_THREADS = 288;
constexpr int TC_TMEM_COLS = 2 * TC_BN;    // two fp32 chunk buffers
constexpr int TC_SMEM = TC_STAGES * TC_STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/;
static_assert(TC_BM * (TC_BN + 1) * 4 <= TC_STAGES * TC_STAGE_BYTES, "epilogue tile fits");

struct TcConv {
    int N, H, W, C, K, R, S, sh, sw, ph, pw, dh, dw, P, Q;
    int64_t M;
    int kdim;     // R*S*C
    int kpad;     // kdim rounded up to 64
    int nkb;      // kpad / 64
    int tap_mode; // C % 64 == 0: every k-block lies inside one tap
};

struct Bars {
    uint64_t full_a[TC_STAGES];
    uint64_t full_b[TC_STAGES];
    uint64_t empty[TC_STAGES];
    uint64_t accf[2];
    uint64_t acce[2];
    uint64_t done;
    uint32_t tmem_base;
    int abort;
    int never;   // stays 0: the abort word of the drain waits, which must not short-cut
};

__device__ __forceinline__ void record_abort(Bars* b, int* err, int code) {
    b->abort = 1;
    if (err) atomicExch(err, code);
}

// 64 consecutive K-elements (k-block kb) of A row (n, pp, qq), as 16 words of int8.
__device__ __forceinline__ void gather_a(const TcConv& p, const int8_t* __restrict__ x, bool valid,
                                         int n, int pp, int qq, int kb, uint32_t (&w)[16]) {
#pragma unroll
    for (int i = 0; i < 16; i++) w[i] = 0;
    if (!valid) return;
    const int kpos = kb * TC_BK;
    if (p.tap_mode) {
        const int tap = kpos / p.C;
        const int c0 = kpos - tap * p.C;
        const int r = tap / p.S, s = tap - (tap / p.S) * p.S;
        const int hh = pp * p.sh + r * p.dh - p.ph;
        const int ww = qq * p.sw + s * p.dw - p.pw;
        if (hh < 0 || hh >= p.H || ww < 0 || ww >= p.W) return;
        const uint4* src = reinterpret_cast<const uint4*>(
            x + (((int64_t)n * p.H + hh) * p.W + ww) * p.C + c0);
#pragma unroll
        for (int i = 0; i < 4; i++) {
            uint4 v = __ldg(src + i);
            w[4 * i + 0] = v.x; w[4 * i + 1] = v.y; w[4 * i + 2] = v.z; w[4 * i + 3] = v.w;
        }
    } else {
        // C % 4 == 0: each 4-code word holds 4 channels of one tap
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
                        x + (((int64_t)n * p.H + hh) * p.W + ww) * p.C + c));
            }
            c += 4;
            if (c == p.C) { c = 0; tap++; }
        }
    }
}

__global__ void __launch_bounds__(TC_THREADS, 1)
    k_conv_fwd_tc(const __grid_constant__ CUtensorMap wmap, TcConv p,
                  const int8_t* __restrict__ x, int32_t* __restrict__ acc,
                  unsigned long long* __restrict__ s1, int* __restrict__ hi_c,
                  int* __restrict__ lo_c, int* __restrict__ err) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    Bars* bars = reinterpret_cast<Bars*>(smem + TC_STAGES * TC_STAGE_BYTES);

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    // a CTA that timed out earlier in this launch makes the rest leave at once
    if (*reinterpret_cast<volatile int*>(err) != 0) return;
    const int64_t m0 = (int64_t)blockIdx.x * TC_BM;
    const int n0 = blockIdx.y * TC_BN;
    const int nkb = p.nkb;
    const int nchunks = (nkb + TC_CHUNK_KB - 1) / TC_CHUNK_KB;

    if (tid == 0) {
        for (int s = 0; s < TC_STAGES; s++) {
            tc::mbar_init(&bars->full_a[s], 128);
            tc::mbar_init(&bars->full_b[s], 1);
            tc::mbar_init(&bars->empty[s], 1);
        }
        for (int b = 0; b < 2; b++) {
            tc::mbar_init(&bars->accf[b], 1);
            tc::mbar_init(&bars->acce[b], 128);
        }
        tc::mbar_init(&bars->done, 1);
        bars->abort = 0;
        bars->never = 0;
        tc::mbar_fence_init();
        tc::tma_prefetch_desc(&wmap);
    }
    if (warp == 8) {
        tc::tmem_alloc(&bars->tmem_base, TC_TMEM_COLS);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort_flag = &bars->abort;

    if (warp < 4) {
        // ------------------------------------------------ producers
        const int row = tid;
        const int64_t m = m0 + row;
        const bool valid = m < p.M;
        int n = 0, pp = 0, qq = 0;
        if (valid) {
            const int64_t pq = (int64_t)p.P * p.Q;
            n = (int)(m / pq);
            const int64_t rem = m - (int64_t)n * pq;
            pp = (int)(rem / p.Q);
            qq = (int)(rem - (int64_t)pp * p.Q);
        }
        uint32_t cur[16], nxt[16];
        gather_a(p, x, valid, n, pp, qq, 0, cur);
        int issued_b = 0;
        for (int kb = 0; kb < nkb; kb++) {
            const int s = kb % TC_STAGES;
            const uint32_t it = (uint32_t)(kb / TC_STAGES);
            if (!tc::mbar_wait(&bars->empty[s], (it & 1) ^ 1, abort_flag)) {
                record_abort(bars, err, 1);
                break;
            }
            uint8_t* a_tile = smem + s * TC_STAGE_BYTES;
            uint8_t* b_tile = a_tile + TC_A_BYTES;
            if (tid == 0) {
                tc::mbar_expect_tx(&bars->full_b[s], TC_B_BYTES);
                tc::tma_load_2d(b_tile, &wmap, &bars->full_b[s], kb * TC_BK, n0);
                tc::mbar_arrive(&bars->full_b[s]);
                issued_b = kb + 1;
            }
            if (kb + 1 < nkb) gather_a(p, x, valid, n, pp, qq, kb + 1, nxt);
            uint8_t* dst_row = a_tile + row * 128;
#pragma unroll
            for (int j = 0; j < 8; j++) {
                uint32_t o0, o1, o2, o3;
                tc::i8x4_to_f16x4(cur[2 * j], o0, o1);
                tc::i8x4_to_f16x4(cur[2 * j + 1], o2, o3);
                *reinterpret_cast<uint4*>(dst_row + ((j ^ (row & 7)) << 4)) =
                    make_uint4(o0, o1, o2, o3);
            }
            tc::fence_proxy_async_smem();
            tc::mbar_arrive(&bars->full_a[s]);
#pragma unroll
            for (int i = 0; i < 16; i++) cur[i] = nxt[i];
        }
        if (tid == 0 && *abort_flag) {
            // let the weight tiles already requested land before the CTA leaves
            for (int kb = (issued_b > TC_STAGES ? issued_b - TC_STAGES : 0); kb < issued_b; kb++)
                tc::mbar_wait(&bars->full_b[kb % TC_STAGES], (uint32_t)(kb / TC_STAGES) & 1,
                              &bars->never);
        }
    } else if (warp == 8) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = tc::idesc_f16_f32(TC_BM, TC_BN);
            bool ok = true;
            for (int kb = 0; kb < nkb && ok; kb++) {
                const int s = kb % TC_STAGES;
                const uint32_t it = (uint32_t)(kb / TC_STAGES);
                const int chunk = kb / TC_CHUNK_KB;
                const int buf = chunk & 1;
                const bool first = (kb % TC_CHUNK_KB) == 0;
                const bool last = ((kb % TC_CHUNK_KB) == TC_CHUNK_KB - 1) || kb == nkb - 1;
                if (first && !tc::mbar_wait(&bars->acce[buf], (uint32_t)((chunk >> 1) & 1) ^ 1,
                                            abort_flag)) { ok = false; break; }
                if (!tc::mbar_wait(&bars->full_b[s], it & 1, abort_flag) ||
                    !tc::mbar_wait(&bars->full_a[s], it & 1, abort_flag)) { ok = false; break; }
                tc::tc_fence_after();
                const uint32_t a_addr = tc::smem_u32(smem + s * TC_STAGE_BYTES);
                const uint32_t b_addr = a_addr + TC_A_BYTES;
#pragma unroll
                for (int j = 0; j < TC_BK / 16; j++) {
                    tc::umma_f16(tmem + buf * TC_BN, tc::sdesc_kmajor_sw128(a_addr + 32 * j),
                                 tc::sdesc_kmajor_sw128(b_addr + 32 * j), idesc,
                                 (first && j == 0) ? 0u : 1u);
                }
                tc::umma_commit(&bars->empty[s]);
                if (last) tc::umma_commit(&bars->accf[buf]);
            }
            if (!ok) record_abort(bars, err, 2);
            // every MMA issued must finish before TMEM is released
            tc::umma_commit(&bars->done);
            tc::mbar_wait(&bars->done, 0, &bars->never);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue (warps 4..7)
        const int row = tid - 128;
        const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
        int accv[TC_BN];
#pragma unroll
        for (int j = 0; j < TC_BN; j++) accv[j] = 0;
        bool ok = true;
        for (int c = 0; c < nchunks; c++) {
            const int buf = c & 1;
            if (!tc::mbar_wait(&bars->accf[buf], (uint32_t)(c >> 1) & 1, abort_flag)) {
                ok = false;
                record_abort(bars, err, 3);
                break;
            }
            tc::tc_fence_after();
#pragma unroll
            for (int cb = 0; cb < TC_BN / 32; cb++) {
                uint32_t r[32];
                tc::tmem_ld_32x32b_x32(tmem + lane_base + buf * TC_BN + cb * 32, r);
                tc::tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; i++) accv[cb * 32 + i] += __float2int_rn(__uint_as_float(r[i]));
            }
            tc::tc_fence_before();
            tc::mbar_arrive(&bars->acce[buf]);
        }
        // tile -> shared memory (stage buffers are free: every MMA has completed)
        int* tile = reinterpret_cast<int*>(smem);
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (ok && !*abort_flag) {
#pragma unroll
            for (int j = 0; j < TC_BN; j++) tile[row * (TC_BN + 1) + j] = accv[j];
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (ok && !*abort_flag) {
            const int rows = (int)((p.M - m0) < TC_BM ? (p.M - m0) : TC_BM);
            const int col = row;  // one output channel per thread
            if (n0 + col < p.K) {
                long long sum = 0;
                int h = INT_MIN, l = INT_MAX;
                for (int i = 0; i < rows; i++) {
                    int v = tile[i * (TC_BN + 1) + col];
                    sum += v; h = max(h, v); l = min(l, v);
                }
                atomicAdd(&s1[n0 + col], (unsigned long long)sum);
                atomicMax(&hi_c[n0 + col], h);
                atomicMin(&lo_c[n0 + col], l);
                for (int i = 0; i < rows; i++)
                    acc[(m0 + i) * p.K + n0 + col] = tile[i * (TC_BN + 1) + col];
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 8) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, TC_TMEM_COLS);
    }
}

// int8 KRSC weights -> fp16 [K][kpad] (zero beyond R*S*C)
__global__ void k_widen_weights(const int8_t* __restrict__ w, __half* __restrict__ wf, int K,
                                int kdim, int kpad) {
    int64_t total = (int64_t)K * kpad;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        int k = (int)(i / kpad), j = (int)(i - (int64_t)k * kpad);
        wf[i] = __int2half_rn(j < kdim ? (int)w[(int64_t)k * kdim + j] : 0);
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

bool tc_env_disabled() {
    const char* e = getenv("IQ_DISABLE_TC");
    return e && e[0] == '1';
}

}  // namespace

size_t conv_fwd_tc_ws_bytes(const iq_conv_desc* d) {
    int64_t kdim = (int64_t)d->r * d->s * (d->c / d->groups);
    int64_t kpad = (kdim + 63) / 64 * 64;
    return (size_t)(d->k * kpad * 2) + 256 + 256;
}

bool conv_fwd_tc_supported(const iq_conv_desc* d) {
    if (tc_env_disabled()) return false;
    if (d->groups != 1) return false;
    if (d->c % 4) return false;
    if (d->k % 8) return false;   // TMA row stride of the fp16 weights is 16-byte aligned anyway
    return true;
}

iq_status conv_fwd_tc(const iq_conv_desc* d, const int8_t* x, const int8_t* w, int32_t* acc,
                      unsigned long long* s1, int* hi, int* lo, void* ws, cudaStream_t st,
                      bool* done) {
    *done = false;
    if (!conv_fwd_tc_supported(d)) return IQ_OK;
    if (((uintptr_t)x & 15) != 0) return IQ_OK;
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
    if (!enc) return IQ_OK;
    TcConv p;
    p.N = d->n; p.H = d->h; p.W = d->w; p.C = d->c; p.K = d->k; p.R = d->r; p.S = d->s;
    p.sh = d->stride_h; p.sw = d->stride_w; p.ph = d->pad_h; p.pw = d->pad_w;
    p.dh = d->dil_h; p.dw = d->dil_w;
    p.P = (d->h + 2 * d->pad_h - d->dil_h * (d->r - 1) - 1) / d->stride_h + 1;
    p.Q = (d->w + 2 * d->pad_w - d->dil_w * (d->s - 1) - 1) / d->stride_w + 1;
    p.M = (int64_t)p.N * p.P * p.Q;
    p.kdim = d->r * d->s * d->c;
    p.kpad = (p.kdim + 63) / 64 * 64;
    p.nkb = p.kpad / 64;
    p.tap_mode = (d->c % 64) == 0;

    char* wsb = (char*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    __half* wf = reinterpret_cast<__half*>(wsb);
    int* err = reinterpret_cast<int*>(wsb + (size_t)p.K * p.kpad * 2);
    k_widen_weights<<<grid_for((int64_t)p.K * p.kpad), kThreads, 0, st>>>(w, wf, p.K, p.kdim,
                                                                         p.kpad);
    IQ_LAUNCH_CHECK();
    IQ_CUDA_CHECK(cudaMemsetAsync(err, 0, sizeof(int), st));

    CUtensorMap map;
    cuuint64_t gdim[2] = {(cuuint64_t)p.kpad, (cuuint64_t)p.K};
    cuuint64_t gstride[1] = {(cuuint64_t)p.kpad * 2};
    cuuint32_t box[2] = {64, TC_BN};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, wf, gdim, gstride, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return IQ_ERR_CUDA;

    IQ_CUDA_CHECK(cudaFuncSetAttribute(k_conv_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       TC_SMEM));
    dim3 grid((unsigned)((p.M + TC_BM - 1) / TC_BM), (unsigned)((p.K + TC_BN - 1) / TC_BN), 1);
    k_conv_fwd_tc<<<grid, TC_THREADS, TC_SMEM, st>>>(map, p, x, acc, s1, hi, lo, err);
    IQ_LAUNCH_CHECK();
    *done = true;
    return IQ_OK;
}

}  // namespace iq
