// iq_conv_tc.cuh -- tensor-core (tcgen05) convolution path.
#pragma once

#include "iq_internal.cuh"

#include <cuda_fp16.h>

namespace iq {

// per-channel statistics of the forward beyond the maximum (always written)
constexpr unsigned TC_STATS_SUM = 1;   // the column sums (the batch-norm mean)
constexpr unsigned TC_STATS_LO = 2;    // the column minima
constexpr unsigned TC_STATS_NOEXT = 16; // no extremes either: a later pass computes them

// Forward convolution on the 5th-generation tensor cores when the shape is
// supported; sets *done = false (and enqueues nothing) otherwise.  Writes the int32
// accumulators and the per-channel max, plus the sum and the min selected by st_mask
// (TC_STATS_*; the CUDA-core path writes all three).
// `ws` must hold conv_fwd_tc_ws_bytes(d) bytes (the fp16 copy of the weights).
// xf (optional): the fp16 carrier of x already written by codes_to_f16, read instead of
// converting x again.
size_t conv_fwd_tc_ws_bytes(const iq_conv_desc* d);
bool conv_fwd_tc_supported(const iq_conv_desc* d);
iq_status conv_fwd_tc(const iq_conv_desc* d, const int8_t* x, const int8_t* w, int32_t* acc,
                      unsigned long long* s1, int* hi, int* lo, void* ws, cudaStream_t st,
                      bool* done, const __half* xf = nullptr,
                      unsigned st_mask = TC_STATS_SUM | TC_STATS_LO);

// x (int8 codes, n elements, n % 16 == 0, 16-byte aligned) -> xf (fp16, 16-byte aligned)
iq_status codes_to_f16(const int8_t* x, __half* xf, int64_t n, cudaStream_t st);

// Stride-1 data gradient as a forward pass over the errors with flipped, transposed
// weights.  Writes int32 sums to out32 plus the per-channel max/min (the channel-major
// kernel also the sums) when the reduction (k r s) fits int32, else adds int64 sums into
// out64 (zeroed by the caller).
size_t conv_dgrad_tc_ws_bytes(const iq_conv_desc* d);
bool conv_dgrad_tc_supported(const iq_conv_desc* d);
int conv_dgrad_tc_slices(const iq_conv_desc* d);
iq_status conv_dgrad_tc(const iq_conv_desc* d, const int8_t* e, const int8_t* w, int32_t* out32,
                        long long* out64, unsigned long long* s1, int* hi, int* lo, void* ws,
                        cudaStream_t st, bool* done, const __half* ef = nullptr);

// Stride-2 data gradient on the tensor-core path by phase decomposition (groups 1, the
// int32 path): the four parity phases of the input run as stride-1 data gradients of
// sub-kernels and are interleaved into out32; the per-channel statistics (s1, hi, lo: C
// entries each, all written by the kernels) accumulate over the phases.  ef: the fp16 carrier
// of e when the caller wrote it.  *done = false when the shape is not covered.
size_t conv_dgrad_tc_stride2_ws_bytes(const iq_conv_desc* d);
iq_status conv_dgrad_tc_stride2(const iq_conv_desc* d, const int8_t* e, const int8_t* w,
                                int32_t* out32, unsigned long long* s1, int* hi, int* lo,
                                void* ws, size_t ws_bytes, cudaStream_t st, bool* done,
                                const __half* ef = nullptr);

// Weight gradient: writes the exact int64 sums to G (KRSC).  When *amax_done, max |G| has
// also been folded into *amax (an atomicMax cell the caller zeroed).
size_t conv_wgrad_tc_ws_bytes(const iq_conv_desc* d);
bool conv_wgrad_tc_supported(const iq_conv_desc* d);
// ef, xf (optional): fp16 carriers of e and x written by codes_to_f16.  g32 (optional):
// when the sums fit one int32 slab (a single split) they are left there, *g32 points at them
// ([K][R S C]) and G is not written.
iq_status conv_wgrad_tc(const iq_conv_desc* d, const int8_t* e, const int8_t* x, long long* G,
                        void* ws, cudaStream_t st, bool* done, unsigned long long* amax,
                        bool* amax_done, const __half* ef = nullptr, const __half* xf = nullptr,
                        const int32_t** g32 = nullptr);

}  // namespace iq
