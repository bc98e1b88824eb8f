// iq_gemm.cu -- an exact int8 GEMM on the fp8 tensor-core path, the third exact route to the
// int8 products of Sec. 3.2-3.3 (the library's convolutions carry int8 codes as exact fp16
// operands of tcgen05 kind::f16; sm_103a assembles no kind::i8).  Each int8 value v splits
// into v = 16 h + l with the signed high nibble h = v >> 4 in [-8, 7] and the low nibble
// l = v & 15 in [0, 15], all exact in e4m3.  Then
//     A B^T = 256 (H_A H_B^T) + 16 (H_A L_B^T + L_A H_B^T) + L_A L_B^T,
// four tcgen05 kind::f8f6f4 MMAs per k-step into three fp32 accumulators in TMEM; every
// partial sum is an integer of magnitude at most 240 K < 2^24 for K <= 65536, so the fp32
// sums are exact, and the epilogue combines them in integers.
//
// Layout: A [m][k], B [n][k] row-major int8 (k contiguous), C = A B^T int32 [m][n];
// m, n multiples of 128, k a multiple of 128, k <= 65536.
#include "iq_internal.cuh"
#include "iq_tc_ptx.cuh"

#include <cudaTypedefs.h>

namespace iq {
namespace {

constexpr int GT = 128;                       // tile rows of A and of B, bytes of k per block
constexpr int GT_TILE = GT * GT;              // one operand tile: 16 KB
constexpr int GT_STAGE = 4 * GT_TILE;         // H_A, L_A, H_B, L_B
constexpr int GT_STAGES = 3;
constexpr int GT_SMEM = 1024 + GT_STAGES * GT_STAGE + 256;
constexpr int GT_THREADS = 256;               // warp 0 TMA, warp 1 MMA, warps 4-7 epilogue
constexpr int GT_TMEM = 512;                  // three 128-column accumulators

// e4m3 (exponent bias 7, 3 mantissa bits) byte of an integer of magnitude <= 15
__host__ __device__ constexpr uint32_t e4m3_of_small(int v) {
    const uint32_t s = v < 0 ? 0x80u : 0u;
    const int a = v < 0 ? -v : v;
    if (a == 0) return s;
    int e = 0;
    while ((2 << e) <= a) e++;                // 2^e <= a < 2^(e+1)
    const int m = ((a << 3) >> e) - 8;         // a = 2^e (1 + m / 8), exact for a <= 15
    return s | (uint32_t)((e + 7) << 3) | (uint32_t)m;
}

// the nibble split of 4 codes a thread: hi = e4m3(v >> 4), lo = e4m3(v & 15)
__global__ void k_nibble_split(const uint32_t* __restrict__ x, int64_t n4,
                               uint32_t* __restrict__ hi, uint32_t* __restrict__ lo) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t w = x[i];
        uint32_t h = 0, l = 0;
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const int v = (int)(int8_t)(w >> (8 * j));
            h |= e4m3_of_small(v >> 4) << (8 * j);
            l |= e4m3_of_small(v & 15) << (8 * j);
        }
        hi[i] = h;
        lo[i] = l;
    }
}

__device__ __forceinline__ void umma_f8_e(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                          uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p, e;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "elect.sync _|e, 0xffffffff;\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

struct GemmBars {
    uint64_t full[GT_STAGES];
    uint64_t empty[GT_STAGES];
    uint64_t done;
    uint32_t tmem_base;
    int abort;
    int never;
};

// one 128 x 128 tile of C per CTA
__global__ void __launch_bounds__(GT_THREADS, 1)
    k_gemm_nibble(const __grid_constant__ CUtensorMap mah, const __grid_constant__ CUtensorMap mal,
                  const __grid_constant__ CUtensorMap mbh, const __grid_constant__ CUtensorMap mbl,
                  int n, int k, int32_t* __restrict__ c, int* __restrict__ err) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    GemmBars* bars = reinterpret_cast<GemmBars*>(smem + GT_STAGES * GT_STAGE);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (__syncthreads_or(tid == 0 ? *reinterpret_cast<volatile int*>(err) : 0)) return;
    const int m0 = blockIdx.x * GT, n0 = blockIdx.y * GT;
    const int nkb = k / GT;
    if (tid == 0) {
        for (int s = 0; s < GT_STAGES; s++) {
            tc::mbar_init(&bars->full[s], 1);
            tc::mbar_init(&bars->empty[s], 1);
        }
        tc::mbar_init(&bars->done, 1);
        bars->abort = 0;
        bars->never = 0;
        tc::mbar_fence_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&bars->tmem_base, GT_TMEM);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort_flag = &bars->abort;
    if (warp == 0) {
        // ---------------------------------------------- TMA: the four operand tiles
        int issued = 0;
        for (int kb = 0; kb < nkb; kb++) {
            const int s = kb % GT_STAGES;
            const uint32_t ph = (uint32_t)(kb / GT_STAGES) & 1u;
            if (!tc::mbar_wait_warp(&bars->empty[s], ph ^ 1u, abort_flag)) {
                bars->abort = 1;
                atomicExch(err, 4);
                break;
            }
            uint8_t* st = smem + s * GT_STAGE;
            tc::mbar_expect_tx_e(&bars->full[s], GT_STAGE);
            tc::tma_load_2d_e(st, &mah, &bars->full[s], kb * GT, m0);
            tc::tma_load_2d_e(st + GT_TILE, &mal, &bars->full[s], kb * GT, m0);
            tc::tma_load_2d_e(st + 2 * GT_TILE, &mbh, &bars->full[s], kb * GT, n0);
            tc::tma_load_2d_e(st + 3 * GT_TILE, &mbl, &bars->full[s], kb * GT, n0);
            tc::mbar_arrive_e(&bars->full[s]);
            issued = kb + 1;
        }
        if (*abort_flag) {
            // let this warp's copies in flight land before the CTA leaves
            for (int kb = (issued > GT_STAGES ? issued - GT_STAGES : 0); kb < issued; kb++)
                tc::mbar_wait(&bars->full[kb % GT_STAGES], (uint32_t)(kb / GT_STAGES) & 1u,
                              &bars->never);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------------------------------------- MMA: HH into D0, HL + LH into D1, LL into D2
        const uint32_t idesc = tc::idesc_f16_f32(GT, GT);   // E4M3 is format code 0, as F16
        bool ok = true;
        for (int kb = 0; kb < nkb && ok; kb++) {
            const int s = kb % GT_STAGES;
            const uint32_t ph = (uint32_t)(kb / GT_STAGES) & 1u;
            if (!tc::mbar_wait_warp(&bars->full[s], ph, abort_flag)) {
                ok = false;
                break;
            }
            tc::tc_fence_after();
            const uint32_t base = tc::smem_u32(smem + s * GT_STAGE);
#pragma unroll
            for (int j = 0; j < GT / 32; j++) {          // k-steps of 32 bytes
                const uint64_t ah = tc::sdesc_kmajor_sw128(base + 32 * j);
                const uint64_t al = tc::sdesc_kmajor_sw128(base + GT_TILE + 32 * j);
                const uint64_t bh = tc::sdesc_kmajor_sw128(base + 2 * GT_TILE + 32 * j);
                const uint64_t bl = tc::sdesc_kmajor_sw128(base + 3 * GT_TILE + 32 * j);
                const uint32_t acc = (kb | j) ? 1u : 0u;
                umma_f8_e(tmem, ah, bh, idesc, acc);
                umma_f8_e(tmem + GT, ah, bl, idesc, acc);
                umma_f8_e(tmem + GT, al, bh, idesc, 1u);
                umma_f8_e(tmem + 2 * GT, al, bl, idesc, acc);
            }
            tc::umma_commit_e(&bars->empty[s]);
        }
        if (!ok) {
            bars->abort = 1;
            atomicExch(err, 2);
        }
        tc::umma_commit_e(&bars->done);
        tc::mbar_wait(&bars->done, 0, &bars->never);
        __syncwarp();
    } else if (warp >= 4) {
        // ---------------------------------------------- epilogue: 256 HH + 16 (HL + LH) + LL
        const int row = ((warp & 3) << 5) + lane;
        const uint32_t taddr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        if (tc::mbar_wait_sleep(&bars->done, 0, abort_flag) && !*abort_flag) {
            tc::tc_fence_after();
            int32_t* out = c + (int64_t)(m0 + row) * n + n0;
#pragma unroll 1
            for (int cb = 0; cb < GT; cb += 32) {
                uint32_t hh[32], cr[32], ll[32];
                tc::tmem_ld_32x32b_x32(taddr + cb, hh);
                tc::tmem_ld_32x32b_x32(taddr + GT + cb, cr);
                tc::tmem_ld_32x32b_x32(taddr + 2 * GT + cb, ll);
                tc::tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; i += 4) {
                    int v[4];
#pragma unroll
                    for (int u = 0; u < 4; u++)
                        v[u] = 256 * __float2int_rn(__uint_as_float(hh[i + u])) +
                               16 * __float2int_rn(__uint_as_float(cr[i + u])) +
                               __float2int_rn(__uint_as_float(ll[i + u]));
                    *reinterpret_cast<int4*>(out + cb + i) = make_int4(v[0], v[1], v[2], v[3]);
                }
            }
        } else {
            atomicExch(err, 3);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, GT_TMEM);
    }
}

// 2-D map over a row-major [rows][k] byte array: box 128 bytes of k x 128 rows, 128-byte
// swizzle (the K-major UMMA layout of 8-bit operands)
iq_status encode_nibbles(const uint8_t* base, int rows, int k, CUtensorMap* map) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess || !fn)
        return IQ_ERR_UNSUPPORTED;
    auto enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    cuuint64_t gdim[2] = {(cuuint64_t)k, (cuuint64_t)rows};
    cuuint64_t gstride[1] = {(cuuint64_t)k};
    cuuint32_t box[2] = {GT, GT};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), gdim,
                     gstride, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? IQ_OK : IQ_ERR_CUDA;
}

size_t gemm_nibble_ws(int32_t m, int32_t n, int32_t k) {
    return 2 * ((size_t)m + n) * k + 4 * 256;
}

}  // namespace
}  // namespace iq

using namespace iq;

extern "C" iq_status iq_gemm_s8_nibble_workspace_size(int32_t m, int32_t n, int32_t k,
                                                      size_t* bytes) {
    if (!bytes || m <= 0 || n <= 0 || k <= 0) return IQ_ERR_INVALID_ARG;
    *bytes = gemm_nibble_ws(m, n, k);
    return IQ_OK;
}

extern "C" iq_status iq_gemm_s8_nibble(const int8_t* a, const int8_t* b, int32_t* c, int32_t m,
                                       int32_t n, int32_t k, void* ws, size_t ws_bytes,
                                       iq_stream stream) {
    if (!a || !b || !c || m <= 0 || n <= 0 || k <= 0) return IQ_ERR_INVALID_ARG;
    if (m % GT || n % GT || k % GT || k > 65536) return IQ_ERR_UNSUPPORTED;
    if (((uintptr_t)a | (uintptr_t)b | (uintptr_t)c) & 15) return IQ_ERR_INVALID_ARG;
    if (!ws || ws_bytes < gemm_nibble_ws(m, n, k)) return IQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    int* err = device_status_ptr();
    if (!err) return IQ_ERR_CUDA;
    uint8_t* w = (uint8_t*)(((uintptr_t)ws + 255) & ~uintptr_t(255));
    const size_t na = (size_t)m * k, nb = (size_t)n * k;
    uint8_t* ah = w;
    uint8_t* al = ah + na;
    uint8_t* bh = al + na;
    uint8_t* bl = bh + nb;
    k_nibble_split<<<grid_for((int64_t)na / 4), kThreads, 0, st>>>(
        (const uint32_t*)a, (int64_t)na / 4, (uint32_t*)ah, (uint32_t*)al);
    IQ_LAUNCH_CHECK();
    k_nibble_split<<<grid_for((int64_t)nb / 4), kThreads, 0, st>>>(
        (const uint32_t*)b, (int64_t)nb / 4, (uint32_t*)bh, (uint32_t*)bl);
    IQ_LAUNCH_CHECK();
    CUtensorMap mah, mal, mbh, mbl;
    iq_status r = encode_nibbles(ah, m, k, &mah);
    if (r == IQ_OK) r = encode_nibbles(al, m, k, &mal);
    if (r == IQ_OK) r = encode_nibbles(bh, n, k, &mbh);
    if (r == IQ_OK) r = encode_nibbles(bl, n, k, &mbl);
    if (r != IQ_OK) return r;
    IQ_CUDA_CHECK(cudaFuncSetAttribute(k_gemm_nibble, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       GT_SMEM));
    kt_set_op(4, (double)m * n * k, (double)m * n * k);
    kt_pre(st);
    k_gemm_nibble<<<dim3((unsigned)(m / GT), (unsigned)(n / GT)), GT_THREADS, GT_SMEM, st>>>(
        mah, mal, mbh, mbl, n, k, c, err);
    IQ_LAUNCH_CHECK();
    kt_post(st, IQ_KERNEL_GEMM_NIBBLE);
    return IQ_OK;
}
