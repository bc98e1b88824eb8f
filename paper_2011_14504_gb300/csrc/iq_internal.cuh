// iq_internal.cuh -- launchers shared between the translation units of the library.
#pragma once

#include "iq_common.cuh"
#include <cuda_fp16.h>

#include <cuda.h>

namespace iq {

// Device address of the sticky status word that iq_device_status reads and clears (a kernel
// whose bounded wait gave up stores its IQ_ERR_* code there), or NULL.
int* device_status_ptr();

// streaming multiprocessors of the current device
int device_sms();

// 2-D tensor map of a row-major [m][C] array of 1- or 2-byte elements: box {box_c channels,
// box_r rows}, no swizzle, zero fill outside the array
iq_status encode_rows_2d(const void* base, int esz, int64_t m, int C, int box_c, int box_r,
                         CUtensorMap* map);

// Scratch needed by requant_int (bytes).
size_t requant_ws_bytes();

// Device address of the stochastic-rounding epoch (the fourth Philox counter word), or NULL.
unsigned long long* rq_epoch_ptr();

// SQ / RQ of an integer-coded tensor (see iq_requantize in iq.h).  `relu` applies
// to the SQ modes only.  `out` has out_dtype elements.
iq_status requant_int(const void* q, int in_dtype, int64_t n, const double* s_in, int k,
                      int mode, uint64_t seed, uint64_t layer, uint64_t step, uint64_t tag,
                      void* out, int out_dtype, double* s_out, void* ws, cudaStream_t st);

// Quantizer parameters of SQ_k / RQ_k for a tensor with max |q| = M and input scale s.
struct RqParams {
    uint64_t M;
    UDiv div;      // by 2M (SQ) or by M (RQ)
    double s_out;
    uint32_t R8;   // SQ with k = 8 and 128 < M <= 2^31: floor(2^39 / M), else 0
    float kq;      // with R8: fl(128 / M)
};

__device__ inline RqParams rq_params_make(uint64_t M, double s, int k, int mode) {
    RqParams p;
    p.M = M;
    const bool rq = mode == IQ_MODE_RQ_GQ1 || mode == IQ_MODE_RQ_GQ2;
    p.div = make_udiv(M == 0 ? 1 : (rq ? M : 2 * M));
    p.R8 = (!rq && k == 8 && M > 128 && M <= (uint64_t(1) << 31))
               ? (uint32_t)((uint64_t(1) << 39) / M) : 0u;
    p.kq = p.R8 ? __double2float_rn(__ddiv_rn(128.0, (double)M)) : 0.0f;
    if (mode == IQ_MODE_RQ_GQ2) p.s_out = ldexp(1.0, 1 - k);
    else p.s_out = M ? ldexp(__dmul_rn(s, (double)M), 1 - k) : ldexp(s, 1 - k);
    return p;
}

// where requant_apply keeps the parameters in its workspace
inline RqParams* rq_params_slot(void* ws) { return (RqParams*)((char*)ws + 256); }

// The same with max |q| already in the first 8 bytes of ws (an unsigned long long); with
// params_ready the parameters (rq_params_slot) and *s_out have been written as well.  clip:
// the SQ modes' M is not the tensor's own maximum (frozen statistics), so q is clipped to
// [-M, M] first.
// out16 (optional, int8 SQ codes only): the fp16 copy of the output codes is written too
// (n % 16 == 0, out and out16 16-byte aligned).  mask (optional, int8 SQ codes only): a code
// is kept where mask > 0 and zeroed elsewhere (the ReLU backward of the layer whose
// activation codes mask holds; the scale is the unmasked tensor's), 16-byte aligned with out16.
iq_status requant_apply(const void* q, int in_dtype, int64_t n, const double* s_in, int k,
                        int mode, uint64_t seed, uint64_t layer, uint64_t step, uint64_t tag,
                        void* out, int out_dtype, double* s_out, void* ws, cudaStream_t st,
                        bool params_ready = false, bool clip = false, __half* out16 = nullptr,
                        const int8_t* mask = nullptr);

// finished int8 codes x: zeroed in place where mask <= 0 (mask optional), and their fp16
// copy written (x16 optional: n % 16 == 0, x, mask, x16 16-byte aligned)
iq_status codes_mask_copy(int8_t* x, const int8_t* mask, int64_t n, __half* x16,
                          cudaStream_t st);

// int8 codes -> their exact fp16 copies (n % 16 == 0, both 16-byte aligned)
iq_status codes_to_f16(const int8_t* x, __half* xf, int64_t n, cudaStream_t st);
// an fp16 output copy is valid for n codes at these addresses
inline bool f16_copy_ok(const void* codes, const void* xf, int64_t n) {
    return n % 16 == 0 && (((uintptr_t)codes | (uintptr_t)xf) & 15) == 0;
}

// Per-channel statistics buffers of a BN layer, in the workspace.
struct BnStats {
    unsigned long long* s1;   // sum acc (two's complement int64)
    int* hi;                  // max acc
    int* lo;                  // min acc
    unsigned long long* dev;  // sum |acc - floor(S1/m)|
    unsigned long long* ngt;  // #(acc > floor(S1/m))
    long long* F;             // fixed-point maps acc -> X and X -> A
    long long* B;
    long long* G;
    long long* H;
    int* codes;               // [2C]: mu_q codes, sigma_q codes
    int* px;                  // shifts [2]
    double* scal;             // IQ_BN_SCALES doubles (workspace copy)
    unsigned long long* red;  // [8]: tensor-wide maxima of non-negative doubles (bit patterns)
};

size_t bn_fwd_ws_bytes(int32_t C);
BnStats bn_stats_carve(WsCursor& cur, int32_t C);
// zero sums, hi = INT_MIN, lo = INT_MAX
iq_status bn_stats_init(const BnStats& s, int32_t C, cudaStream_t st);
// channel sums / extremes of acc[m][C] (when the producer did not fuse them)
iq_status bn_stats_pass(const int32_t* acc, int64_t m, int32_t C, const BnStats& s,
                        cudaStream_t st);
// everything after the statistics: deviation pass, finalize, requant pass
iq_status bn_fwd_after_stats(const int32_t* acc, int64_t m, int32_t C, const double* s_acc,
                             const int32_t* gamma, const int32_t* beta, const iq_bn_bits& b,
                             const BnStats& s, int16_t* xhat, int8_t* a, double* s_a,
                             int32_t* bn_codes, double* bn_scales, int64_t* bn_fixed,
                             cudaStream_t st, __half* a16 = nullptr);

// the forward's element maps with frozen constants (F, B, G, H, P_x, P_a from an earlier call)
iq_status bn_apply_fixed(const int32_t* acc, int64_t m, int32_t C, const int64_t* fixed, int kx,
                         int ka, int16_t* X, int8_t* A, cudaStream_t st);

inline iq_bn_bits bn_bits_or_default(const iq_bn_bits* b) {
    if (b) return *b;
    iq_bn_bits d;
    d.k_mu = 16; d.k_sigma = 16; d.k_xhat = 16; d.k_gamma = 8; d.k_beta = 8; d.k_a = 8;
    return d;
}

inline bool bn_bits_valid(const iq_bn_bits& b) {
    return b.k_mu >= 2 && b.k_mu <= 24 && b.k_sigma >= 2 && b.k_sigma <= 24 &&
           b.k_xhat >= 2 && b.k_xhat <= 16 && b.k_gamma >= 2 && b.k_gamma <= 16 &&
           b.k_beta >= 2 && b.k_beta <= 16 && b.k_a >= 2 && b.k_a <= 8;
}


// kernel timing (iq_kernel_timing_begin / _end): the conv entry points name the operation
// and its algorithmic (in-bounds) and dense MACs, the launchers bracket their main kernel
// with kt_pre / kt_post; a bandwidth kernel is bracketed with kt_pre / kt_post_bytes and
// tagged with the bytes its pass must read and write
void kt_set_op(int op, double macs, double dense);
void kt_pre(cudaStream_t st);
void kt_post(cudaStream_t st, int kernel);
void kt_post_bytes(cudaStream_t st, int kernel, double bytes);

}  // namespace iq
