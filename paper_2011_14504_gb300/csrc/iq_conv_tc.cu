// iq_conv_tc.cu -- tcgen05 implicit-GEMM convolution (placeholder until the kernel lands).
#include "iq_conv_tc.cuh"

namespace iq {

iq_status conv_fwd_tc(const iq_conv_desc*, const int8_t*, const int8_t*, int32_t*,
                      unsigned long long*, int*, int*, cudaStream_t, bool* done) {
    *done = false;
    return IQ_OK;
}

}  // namespace iq
