/*
 * iq.h -- C ABI of the integer quantized convolution layer for GB300 (sm_103a).
 *
 * Method: "Training and Inference for Integer-Based Semantic Segmentation
 * Network" (Yang, Deng, Yang, Xie, Li; arXiv 2011.14504), Sec. 3.
 *
 * Conventions shared by every entry point
 *  - A quantized tensor is integer codes plus one real scale: value = code * scale.
 *    Scales are IEEE fp64 values that live in DEVICE memory (a `double*`), so a
 *    chain of calls never synchronizes with the host.  An input scale is read by
 *    the kernels; an output scale is written by them.
 *  - Every tensor pointer is a device pointer to caller-owned memory.  The
 *    library allocates nothing and keeps no state between calls: scratch space is
 *    the `ws` argument, whose minimum size the matching *_workspace_size call
 *    returns (a NULL `ws` with ws_bytes == 0 is accepted when that size is 0).
 *  - Layouts: activations and errors NHWC (channels innermost), filters KRSC
 *    (K output channels, R x S taps, C/groups channels innermost), per-channel
 *    vectors length C.  All integer codes are two's complement.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *    stream).  Argument errors are reported before anything is enqueued;
 *    kernel-side failures surface as IQ_ERR_CUDA from the launch check.
 *  - Determinism: identical inputs, seed and step give identical bits on every
 *    run; all reductions are integer (order-independent) and the fp64 scale
 *    steps follow a fixed operation order.
 *  - Bit widths follow the paper's defaults (Sec. 5): k_W = k_A = k_E1 = k_G = 8,
 *    k_U = 24, k_mu = k_sigma = k_xhat = 16, k_gamma = k_beta = 8, k_E2 in {8,16}.
 */
#ifndef IQ_H
#define IQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* iq_stream; /* cudaStream_t */

typedef enum {
    IQ_OK = 0,
    IQ_ERR_INVALID_ARG = 1,   /* NULL pointer, bad size, bad bit width, bad layout */
    IQ_ERR_UNSUPPORTED = 2,   /* valid request this build does not implement */
    IQ_ERR_WORKSPACE = 3,     /* ws smaller than the *_workspace_size result */
    IQ_ERR_OVERFLOW_RISK = 4, /* int32 accumulation could overflow at this shape */
    IQ_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up */
    IQ_ERR_CUDA = 6           /* a CUDA launch or runtime call failed */
} iq_status;

/* element types */
enum { IQ_I8 = 1, IQ_I16 = 2, IQ_I32 = 3, IQ_I64 = 4, IQ_F32 = 5, IQ_U8 = 6 };

/* quantizer modes */
enum {
    IQ_MODE_UQ = 0,      /* Eq. (UQ): codes of UQ(x,k), scale 2^(1-k)                   */
    IQ_MODE_UQ2 = 1,     /* 2*UQ(x/2,k) (Sec. 3.1.1 x2 scaling): scale 2^(2-k)           */
    IQ_MODE_SQ = 2,      /* Eq. (ScaleQ): Scale(x) = max|x| over the tensor             */
    IQ_MODE_SQ_RELU = 3, /* SQ(ReLU(x)): Eq. (AQ1) after the activation                 */
    IQ_MODE_RQ_GQ1 = 4,  /* Eq. (GQ1): Scale(G) * RQ(G/Scale(G), k), stochastic (SR)    */
    IQ_MODE_RQ_GQ2 = 5   /* Eq. (GQ2): RQ(G/Scale(G), k), magnitude dropped             */
};

/* Convolution geometry and code widths (Sec. 3.2, Eqs. (WQ1), (AQ1); the problem statement of
 * Sec. 3 fixes no memory layout).  With layout IQ_LAYOUT_NHWC: input NHWC [n][h][w][c],
 * filters KRSC [k][r][s][c/groups], output and errors [n][p][q][k].  With IQ_LAYOUT_NCHW:
 * input [n][c][h][w], filters KCRS [k][c/groups][r][s], output and errors [n][k][p][q]
 * (the gradient codes and sums of iq_conv_wgrad follow the filter layout); the library
 * transposes through the workspace and computes in NHWC.  p = (h + 2 pad_h - dil_h (r-1)
 * - 1) / stride_h + 1 (q alike).  Output pixel (p,q), tap (r,s) reads input row
 * p*stride_h + r*dil_h - pad_h and column q*stride_w + s*dil_w - pad_w; outside the image the
 * input is zero.  Group g maps input channels [g c/G, (g+1) c/G) to outputs [g k/G, (g+1) k/G).
 *   k_w  bit width of the weight codes W_q = UQ(W_m, k_w) (Eq. (WQ1)), 2..8, 0 = 8: their
 *        step 2^(1-k_w) is the weight factor of the accumulator scale
 *   k_a  bit width of the output activation codes Q_A = SQ(., k_a) (Eq. (AQ1)), 2..8,
 *        0 = 8 (with batch norm the bits argument's k_a, when given, must agree)
 *   flags  0 or a combination of IQ_CONV_X_F16_READY: the x_f16 buffer given to
 *        iq_conv_fwd / iq_conv_fwd_frozen already holds the fp16 copy of this call's input
 *        codes (an earlier call on the same input, or the call that produced the input with
 *        an fp16 output copy, wrote it), so the call reads it and does not write it; and
 *        IQ_CONV_E_F16_READY: the same for the e_f16 buffer of iq_conv_dgrad and the errors
 *        e.  The caller keeps a copy and its codes in step (a copy of other codes gives
 *        wrong sums).  A storage option with no counterpart in the paper.
 * A zero-initialised descriptor tail gives the paper's setting (NHWC, 8-bit codes). */
enum { IQ_LAYOUT_NHWC = 0, IQ_LAYOUT_NCHW = 1 };
enum { IQ_CONV_X_F16_READY = 1, IQ_CONV_E_F16_READY = 2 };
typedef struct {
    int32_t n, h, w, c;
    int32_t k, r, s;
    int32_t stride_h, stride_w, pad_h, pad_w, dil_h, dil_w, groups;
    int32_t layout, k_w, k_a;
    int32_t flags;
} iq_conv_desc;

/* Bit widths of the quantized L1BN objects (Sec. 3.2.2 equation block, Eq. (AQ1)). */
typedef struct {
    int32_t k_mu, k_sigma, k_xhat, k_gamma, k_beta, k_a;
} iq_bn_bits;

/* Per-tensor fp64 values of an L1BN forward pass, written to `bn_scales`
 * (device, IQ_BN_SCALES doubles) and read back by the backward pass. */
enum {
    IQ_BN_S_XHAT = 0, /* scale of the X (= Q_xhat(xhat)) codes: M_xhat * 2^(1-k_xhat) */
    IQ_BN_M_XHAT = 1, /* max |xhat| over the tensor                                      */
    IQ_BN_M_Y = 2,    /* max ReLU(gamma_q xhat_q + beta_q) over the tensor               */
    IQ_BN_S_ACC = 3,  /* scale of the conv accumulators the pass consumed               */
    IQ_BN_S_A = 4,    /* scale of the A codes (also written to s_a)                     */
    IQ_BN_SCALES = 8
};

const char* iq_status_str(iq_status s);
int iq_version(void);

/* Number of kernels the library has enqueued in this process (host-side counter; the
 * paper has no counterpart -- it lets a caller count device launches in a region). */
unsigned long long iq_launch_count(void);

/* iq_device_status -- the library's sticky device status (the paper has no counterpart).
 * Every wait inside the tensor-core convolution kernels is bounded (about one second); a
 * wait that gives up records a code (1: operand loads, 2: MMA issue, 3: epilogue, 4: a
 * TMA-fed producer, 5: iq_wait_selftest), the kernel returns without completing its tiles, and every later
 * launch of those kernels returns at once, so the outputs of that call and of all later
 * calls are not valid.  This call synchronizes `stream`, stores the code in *code (0 when
 * nothing gave up), clears it and returns IQ_ERR_TIMEOUT when it was set, else IQ_OK.
 * Call it after a sequence of calls (a training step) to learn whether they completed. */
iq_status iq_device_status(int32_t* code, iq_stream stream);

/* iq_wait_selftest -- a check of the bounded-wait path above (the paper has no counterpart).
 * Enqueues on `stream` one kernel whose single thread makes the tensor-core kernels' bounded
 * mbarrier wait, with a limit of limit_cycles SM cycles (0 .. 2^31), on a barrier that
 * nothing arrives on.  The wait gives up, the kernel records code 5 in the sticky status and
 * returns; nothing else is in flight.  The next iq_device_status returns IQ_ERR_TIMEOUT with
 * code 5 and clears the status (until then the tensor-core convolution kernels return at
 * once).  IQ_ERR_INVALID_ARG for a limit outside the range. */
iq_status iq_wait_selftest(long long limit_cycles, iq_stream stream);

/* Kernel timing -- a measurement aid (the paper has no counterpart).  Between
 * iq_kernel_timing_begin and iq_kernel_timing_end, every launch of a convolution kernel and
 * of the main bandwidth-bound kernels (up to 8192 launches) is bracketed by a pair of CUDA
 * events recorded on its launching stream.  A convolution launch is tagged with its kernel,
 * the calling operation and the operation's multiply-accumulates (counted once per call, on
 * its first bracketed launch): `macs` counts the in-bounds products only (the taps that read
 * inside the input), `dense_macs` every tap N P Q K R S C / groups.  A bandwidth launch is
 * tagged with its kernel and `bytes`, the bytes its pass must read and write (each operand
 * once).  Use it on eagerly launched calls, not inside a CUDA graph capture.
 * iq_kernel_timing_end waits for the recorded events, writes one iq_kernel_time per
 * (kernel, op) pair seen (at most `capacity`, the count in *n_out), and stops recording.
 * Errors: IQ_ERR_INVALID_ARG for null pointers, IQ_ERR_CUDA when an event call fails. */
enum {
    IQ_KERNEL_CONV_PIXEL_MAJOR = 1,    /* all-TMA kernel, forward / data gradient (k_conv_tct)  */
    IQ_KERNEL_CONV_CHANNEL_MAJOR = 2,  /* channel-major kernel, <= 128 output channels (k_conv_tcc) */
    IQ_KERNEL_CONV_WGRAD = 3,          /* all-TMA kernel, weight gradient                       */
    IQ_KERNEL_CONV_CPASYNC = 4,        /* cp.async-fed forward kernel (k_conv_tcq)               */
    IQ_KERNEL_CONV_GATHER = 5,         /* register-gather kernel (k_conv_tcp)                    */
    IQ_KERNEL_CONV_SIMT = 6,           /* CUDA-core kernel (k_conv_simt)                         */
    IQ_KERNEL_BN_DEV = 10,             /* L1BN deviation pass (k_bn_dev)                         */
    IQ_KERNEL_BN_REQUANT = 11,         /* L1BN acc -> X -> A pass (k_bn_requant)                 */
    IQ_KERNEL_BNB_PASS1 = 12,          /* L1BN backward: max |e_y gamma| pass (k_bnb_max_s), or
                                          the one-pass histogram (k_bnb_hist) for other C      */
    IQ_KERNEL_BNB_PASS2 = 13,          /* L1BN backward sums pass (k_bnb_sums_s)                 */
    IQ_KERNEL_BNB_PASS3 = 14,          /* L1BN backward output pass (k_bnb_out_s, k_bnb_p3w)     */
    IQ_KERNEL_COMBINE_MAX = 15,        /* iq_combine, max |z| pass                               */
    IQ_KERNEL_COMBINE_CODES = 16,      /* iq_combine, codes pass                                 */
    IQ_KERNEL_SQ_CODES = 17,           /* SQ codes of int32 / int64 sums (k_sq_i32_i8x4, k_sq_int) */
    IQ_KERNEL_CODES_TO_F16 = 18,       /* fp16 carrier copy of int8 codes (k_codes_to_f16)       */
    IQ_KERNEL_ABSMAX = 19,             /* max |q| pass of SQ / RQ (k_absmax_int)                 */
    IQ_KERNEL_RQ_CODES = 20,           /* RQ codes (k_rq_int)                                    */
    IQ_KERNEL_GEMM_NIBBLE = 21         /* nibble-split fp8 GEMM (k_gemm_nibble)                  */
};
typedef struct iq_kernel_time {
    int32_t kernel;     /* IQ_KERNEL_* */
    int32_t op;         /* 1 iq_conv_fwd, 2 iq_conv_dgrad, 3 iq_conv_wgrad, 4 iq_gemm_s8_nibble;
                           0 bandwidth kernels */
    int32_t launches;   /* bracketed launches */
    int32_t pad;
    double ms;          /* summed event time of those launches, milliseconds */
    double macs;        /* summed in-bounds multiply-accumulates of their calls */
    double dense_macs;  /* summed dense multiply-accumulates of their calls */
    double bytes;       /* summed algorithmic bytes of the bandwidth launches */
} iq_kernel_time;
iq_status iq_kernel_timing_begin(void);
iq_status iq_kernel_timing_end(iq_kernel_time* out, int32_t capacity, int32_t* n_out);

/* The stochastic rounding of Eqs. (SQ),(SR) draws, for element i, the Philox4x64-10 block with
 * key (seed, layer) and counter (i/8, step, tag, epoch).  epoch is a device-resident word of
 * the library, 0 until changed: iq_rq_epoch_advance adds 1 to it as a stream operation (so a
 * training step captured in a CUDA graph, with the advance at its end, draws new numbers on
 * every replay); iq_rq_epoch_set sets it.  (The paper has no counterpart: it fixes no RNG.) */
iq_status iq_rq_epoch_advance(iq_stream stream);
iq_status iq_rq_epoch_set(uint64_t value, iq_stream stream);

/* Output size of a convolution (host-side, no device work). */
iq_status iq_conv_out_size(const iq_conv_desc* d, int32_t* p, int32_t* q);

/* Workspace sizes in bytes (host-side, no device work). */
iq_status iq_quantize_workspace_size(int64_t n, size_t* bytes);
iq_status iq_conv_fwd_workspace_size(const iq_conv_desc* d, int with_bn, size_t* bytes);
iq_status iq_conv_dgrad_workspace_size(const iq_conv_desc* d, size_t* bytes);
iq_status iq_conv_wgrad_workspace_size(const iq_conv_desc* d, size_t* bytes);
iq_status iq_bn_int_workspace_size(int64_t m, int32_t c, size_t* bytes);

/* iq_quantize -- real (fp32) tensor to k-bit codes, Sec. 3.1 (Eqs. (del),(UQ),
 * (ScaleFactor),(ScaleQ)).
 *   x        fp32[n], finite values (non-finite inputs give unspecified codes)
 *   k        2..16 for SQ, 2..24 for UQ/UQ2
 *   mode     IQ_MODE_UQ, IQ_MODE_UQ2, IQ_MODE_SQ or IQ_MODE_SQ_RELU
 *   out_dtype IQ_I8 (k <= 8), IQ_I16 (k <= 16) or IQ_I32
 *   codes    out, n elements of out_dtype
 *   scale    out, one device double: the scale of the codes
 * UQ codes: clip(floor(x 2^(k-1) + 1/2)).  SQ: S = max|x|, codes
 * clip(floor(x 2^(k-1)/S + 1/2)) (exact rational value of x/S), scale S 2^(1-k). */
iq_status iq_quantize(const float* x, int64_t n, int k, int mode, int out_dtype, void* codes,
                      double* scale, void* ws, size_t ws_bytes, iq_stream stream);

/* iq_quantize_image_u8 -- the network input: real pixel p/255 quantized with
 * Q_A = SQ(., 8) (Eq. (AQ1); Sec. 5 feeds images to the first conv).  With
 * P = max pixel, code = floor((256 p + P) / (2P)), clipped to 127; scale
 * (P/255) 2^-7.  Input uint8 NHWC (nchw = 0) or NCHW (nchw = 1) with c channels;
 * output int8 NHWC with c_out >= c channels, channels c..c_out-1 zero (padding
 * for aligned loads in the first convolution). */
iq_status iq_quantize_image_u8(const uint8_t* img, int32_t n, int32_t h, int32_t w, int32_t c,
                               int nchw, int32_t c_out, int8_t* codes, double* scale, void* ws,
                               size_t ws_bytes, iq_stream stream);

/* iq_requantize -- integer-coded tensor (codes q, device scale s_in) to k-bit codes.
 *   mode IQ_MODE_SQ / IQ_MODE_SQ_RELU: Eq. (ScaleQ) with M = max|q|:
 *        code = clip(floor((2^k q + M) / (2M))), s_out = (s_in M) 2^(1-k).
 *   mode IQ_MODE_RQ_GQ1 / IQ_MODE_RQ_GQ2: Eqs. (SQ),(SR),(GQ1),(GQ2): y = q 2^(k-1)/M
 *        rounded up with probability y - floor(y) using Philox4x64-10 with key
 *        (seed, layer) and counter (i/8, step, tag, 0) (32-bit half i%2 of word
 *        (i/2)%4 for element i); s_out = (s_in M) 2^(1-k) (GQ1) or 2^(1-k) (GQ2).
 *   in_dtype IQ_I32 or IQ_I64 (|q| < 2^40); k 2..16; out_dtype IQ_I8/IQ_I16/IQ_I32.
 *   M == 0 gives zero codes. */
iq_status iq_requantize(const void* q, int in_dtype, int64_t n, const double* s_in, int k,
                        int mode, uint64_t seed, uint64_t layer, uint64_t step, uint64_t tag,
                        void* codes, int out_dtype, double* s_out, void* ws, size_t ws_bytes,
                        iq_stream stream);

/* iq_requantize_per_channel -- Eq. (ScaleQ) with a per-channel Scale: Eq. (ScaleFactor)'s
 * maximum taken over each channel's elements instead of the whole tensor (the per-channel
 * reading of Scale(x); the paper's networks use the per-tensor form, iq_requantize).
 *   q        integer codes viewed as [outer][c][inner]: NHWC activations or errors with
 *            outer = n h w, inner = 1; NCHW with outer = n, inner = h w; KRSC filters or
 *            filter gradients by output channel with outer = 1, inner = r s c
 *   in_dtype IQ_I32 or IQ_I64 (|q| < 2^40);  s_in device double, the scale of q
 *   relu     nonzero: ReLU(q) is quantized
 *   k        2..16;  out_dtype IQ_I8 (k <= 8), IQ_I16 or IQ_I32
 *   codes    out, like q;  s_out out device double[c]
 * With M_c = max |q| over channel c: code = clip(floor((2^k q + M_c) / (2 M_c))),
 * s_out[c] = (s_in M_c) 2^(1-k); a channel with M_c = 0 gets zero codes and s_in 2^(1-k).
 * Workspace: iq_requantize_per_channel_workspace_size(c). */
iq_status iq_requantize_per_channel_workspace_size(int32_t c, size_t* bytes);
iq_status iq_requantize_per_channel(const void* q, int in_dtype, int64_t outer, int32_t c,
                                    int64_t inner, const double* s_in, int k, int relu,
                                    void* codes, int out_dtype, double* s_out, void* ws,
                                    size_t ws_bytes, iq_stream stream);

/* iq_weight_decay -- L2 weight decay of the master weights.  Sec. 5.1 gives the decay
 * coefficient (5e-4 for FCN, 1e-5 for DeepLab) but not its quantized form; it is read here as
 * a decoupled shrink applied after iq_update, with the decay step lambda lr = 2^-shift:
 * master <- master - floor(master / 2^shift + 1/2) on the k_u grid, then wq = UQ(W_m, k_w)
 * (Eq. (WQ1)).  shift 1..40; k_u, k_w as in iq_update. */
iq_status iq_weight_decay(int32_t* master, int8_t* wq, int64_t n, int shift, int k_u, int k_w,
                          iq_stream stream);

/* iq_gemm_s8_nibble -- C = A B^T for int8 A [m][k], B [n][k] (k contiguous) into int32 C
 * [m][n], exactly, on the fp8 tensor-core path: each code splits into its signed high nibble
 * and its low nibble (v = 16 h + l, both exact in e4m3), and four tcgen05 kind::f8f6f4 MMAs
 * per k-step accumulate 256 H_A H_B^T + 16 (H_A L_B^T + L_A H_B^T) + L_A L_B^T in three
 * exact fp32 sums.  An ablation of the exact tensor-core routes to the int8 products of
 * Sec. 3.2-3.3, beside the fp16 carriers of iq_conv_* (a 1x1 iq_conv_fwd is the same GEMM).
 * m, n multiples of 128, k a multiple of 128 and at most 65536 (else IQ_ERR_UNSUPPORTED);
 * pointers 16-byte aligned.  Workspace: iq_gemm_s8_nibble_workspace_size (the split
 * operands, 2 (m + n) k bytes). */
iq_status iq_gemm_s8_nibble_workspace_size(int32_t m, int32_t n, int32_t k, size_t* bytes);
iq_status iq_gemm_s8_nibble(const int8_t* a, const int8_t* b, int32_t* c, int32_t m, int32_t n,
                            int32_t k, void* ws, size_t ws_bytes, iq_stream stream);

/* iq_weight_requant -- forward weights from master weights, Eqs. (WQ0),(WQ1):
 * master codes m on the k_u grid (value m 2^(1-k_u)), wq = clip(floor((m + 2^(k_u-k_w-1))
 * / 2^(k_u-k_w))) = UQ(W_m, k_w).  Scale of wq is 2^(1-k_w) (x2 grids: 2^(2-k_w)). */
iq_status iq_weight_requant(const int32_t* master, int8_t* wq, int64_t n, int k_u, int k_w,
                            iq_stream stream);

/* iq_conv_fwd -- the quantized conv layer forward (Sec. 3.2, Fig. 4):
 * acc = conv(x, w) in exact int32 (8-bit x and W, Sec. 3.2.3), then either
 *   bn == NULL:  A = Q_A(act(acc s_acc)) = SQ(., 8), Eq. (AQ1), act = ReLU if relu else identity;
 *   bn != NULL:  quantized L1BN (Eqs. (BN2),(BN4),(BN5) and the QBN block; the same
 *                computation as iq_bn_int_fwd) + ReLU + Q_A.
 *   x      int8 NHWC [n][h][w][c];  s_x: device double (scale of x)
 *   w      int8 KRSC, codes of W_q = UQ(W_m, k_w) (scale 2^(1-k_w); s_acc = s_x 2^(1-k_w))
 *   gamma, beta  device int32[k]: codes of gamma_q = 2 UQ(gamma/2, k_gamma) etc. (bn only)
 *   bits   bit widths (bn only; NULL = paper defaults)
 *   a      out int8 NHWC [n][p][q][k];  s_a: out device double
 *   xhat   out int16 [n][p][q][k], the X codes kept for backward (bn only, may be NULL)
 *   bn_codes  out device int32[2k]: mu_q codes then sigma_q codes (bn only, may be NULL)
 *   bn_scales out device double[IQ_BN_SCALES] (bn only, may be NULL)
 *   frozen_out optional out device int64: the constants of this call's output map, for
 *             iq_conv_fwd_frozen on later batches -- with bn, int64[4k + 2]: the fixed-point
 *             F[k], B[k], G[k], H[k] of the acc -> X -> A maps and the shifts P_x, P_a; without
 *             bn, int64[1]: M, the maximum of act(acc) that Q_A divided by
 *   acc_out   optional out int32 [n][p][q][k]: the raw accumulators
 *   x_f16     optional out fp16 [n][h][w][c] (16-byte aligned, n h w c % 16 == 0, else
 *             IQ_ERR_INVALID_ARG): the exact fp16 copy of the codes x (of their NHWC
 *             transpose with IQ_LAYOUT_NCHW) that the tensor-core kernels read (every int8
 *             code is exact in fp16).  When given it is written first (not with
 *             IQ_CONV_X_F16_READY in d->flags: then it is read as it is) and the kernels read
 *             it; keep it for iq_conv_wgrad of the same layer, which then skips its own
 *             conversion of x.  (The paper has no counterpart: it is the
 *             operand format of this implementation's tensor-core path.)
 *   a_f16     optional out fp16 [n][p][q][k] (16-byte aligned, n p q k % 16 == 0, else
 *             IQ_ERR_INVALID_ARG): the exact fp16 copy of the output codes a (of their NHWC
 *             transpose with IQ_LAYOUT_NCHW), written by the pass that writes a; the x_f16 of
 *             the next layer that reads a, under IQ_CONV_X_F16_READY
 * Returns IQ_ERR_OVERFLOW_RISK when (c/groups) r s 127^2 >= 2^31. */
iq_status iq_conv_fwd(const iq_conv_desc* d, const int8_t* x, const double* s_x,
                      const int8_t* w, const int32_t* gamma, const int32_t* beta,
                      const iq_bn_bits* bits, int use_bn, int relu, int8_t* a, double* s_a,
                      int16_t* xhat, int32_t* bn_codes, double* bn_scales, int64_t* frozen_out,
                      int32_t* acc_out, void* x_f16, void* a_f16, void* ws, size_t ws_bytes,
                      iq_stream stream);

/* iq_conv_fwd_frozen -- the inference forward with frozen statistics.  The paper defines no
 * running estimate for its L1BN (Sec. 3.2.2 normalises with the batch's own statistics, and
 * Scale(x) of Eq. (ScaleQ) is the tensor's own maximum); this entry point is the stated
 * deviation that makes a single-pass inference possible: the output map of an earlier
 * iq_conv_fwd call on a calibration batch (its frozen_out) is applied to this batch.
 *   with use_bn: X = clip(floor((F acc + B) / 2^P_x), +-(2^(k_xhat-1)-1)) with the product
 *     in 128 bits, A = clip(floor((G X + H) / 2^P_a), 0, 2^(k_a-1)-1);
 *   without: A = clip(floor((2^k_a act(acc) + M) / (2M))), act = ReLU when relu.
 * The scales are the calibration call's (s_a, bn_scales), which the caller keeps; x must carry
 * the calibration's input scale for the codes to mean the same values.  No statistics are
 * taken and no scale is written.  Arguments as iq_conv_fwd; frozen int64[4k + 2] (use_bn)
 * or int64[1]; bits: the calibration's (NULL: defaults); xhat optional (use_bn only).
 * Workspace: iq_conv_fwd_workspace_size. */
iq_status iq_conv_fwd_frozen(const iq_conv_desc* d, const int8_t* x, const int8_t* w,
                             const int64_t* frozen, const iq_bn_bits* bits, int use_bn,
                             int relu, int8_t* a, int16_t* xhat, void* x_f16, void* ws,
                             size_t ws_bytes, iq_stream stream);

/* iq_conv_dgrad -- error of the layer input (Sec. 3.3.1, Eq. (EQ)):
 * dx = conv_transpose(e, w) in exact int32, then E_1 = SQ(dx, 8).
 *   e    int8 [n][p][q][k] error codes at the conv output; s_e device double
 *   w    int8 KRSC forward weights (scale 2^(1-k_w))
 *   dx   out int8 NHWC [n][h][w][c]; s_dx out device double = (s_e 2^(1-k_w) M) 2^-7
 *   acc_out optional out int32 [n][h][w][c]; must be NULL when (k/groups) r s 127^2 >= 2^31,
 *           where the sums are accumulated in int64 (IQ_ERR_UNSUPPORTED otherwise)
 *   e_f16   optional out fp16 [n][p][q][k], as x_f16 of iq_conv_fwd for the errors e: written
 *           first (not with IQ_CONV_E_F16_READY in d->flags: then it is read as it is) and
 *           read by the kernels; pass it to iq_conv_wgrad of the same layer
 *   dx_mask optional int8 [n][h][w][c]: the dx codes are zeroed where dx_mask <= 0 after Q_E
 *           (s_dx stays the unmasked tensor's): the ReLU backward of the layer whose
 *           activation codes dx_mask holds, usually this layer's own input x (what
 *           iq_relu_bwd would do next, Eq. (EQ) then the mask of Sec. 3.3.1)
 *   dx_f16  optional out fp16 [n][h][w][c]: the exact fp16 copy of the (masked) dx codes, for
 *           the layer below under IQ_CONV_E_F16_READY (16-byte aligned with dx and dx_mask,
 *           n h w c % 16 == 0, else IQ_ERR_INVALID_ARG).  dx_mask and dx_f16: NHWC only
 *           (IQ_ERR_UNSUPPORTED with IQ_LAYOUT_NCHW); no counterpart in the paper */
iq_status iq_conv_dgrad(const iq_conv_desc* d, const int8_t* e, const double* s_e,
                        const int8_t* w, int8_t* dx, double* s_dx, int32_t* acc_out,
                        void* e_f16, const int8_t* dx_mask, void* dx_f16, void* ws,
                        size_t ws_bytes, iq_stream stream);

/* iq_conv_wgrad -- weight gradient and its quantization (Sec. 3.3.2):
 * G[k][r][s][c] = sum_{n,p,q} e[n,p,q,k] x[n, h(p,r), w(q,s), c] in exact int64, then
 * G_q = Eq. (GQ1) (gq_mode 1, networks with BN) or Eq. (GQ2) (gq_mode 2, without).
 *   e, s_e  error codes at the conv output and their scale
 *   x, s_x  the forward input codes and their scale (s_G = s_e s_x)
 *   seed, layer, step  Philox key/counter words of the stochastic rounding (tag 0)
 *   g       out int8 KRSC gradient codes;  s_g out device double
 *   g_acc_out optional out int64 KRSC: the exact sums
 *   e_f16, x_f16  optional fp16 copies of e and x written by iq_conv_dgrad (e_f16) and
 *           iq_conv_fwd (x_f16) for these same codes (16-byte aligned); used instead of
 *           converting e and x again.  Results are undefined if they do not hold e and x. */
iq_status iq_conv_wgrad(const iq_conv_desc* d, const int8_t* e, const double* s_e,
                        const int8_t* x, const double* s_x, int gq_mode, uint64_t seed,
                        uint64_t layer, uint64_t step, int8_t* g, double* s_g,
                        int64_t* g_acc_out, const void* e_f16, const void* x_f16, void* ws,
                        size_t ws_bytes, iq_stream stream);

/* iq_bn_int_fwd -- quantized L1BN + ReLU + Q_A on int32 accumulators acc[m][c] with
 * scale s_acc (Sec. 3.2.2, Eqs. (BN2),(BN4),(BN5), QBN block, Eq. (AQ1)):
 *   mu_B = mean x, sigma_B = mean |x - mu_B| (exact integer sums), mu_q = 2 UQ(mu_B/2, k_mu),
 *   sigma_q = 2 UQ(sigma_B/2, k_sigma), xhat = (x - mu_q)/(sigma_q + eps) with eps one
 *   sigma_q grid step, X = SQ(xhat, k_xhat), y = gamma_q xhat_q + beta_q, A = SQ(ReLU(y), k_a).
 *   The element-wise maps acc -> X -> A are per-channel fixed-point affine maps
 *   floor((F acc + B) / 2^P) whose constants come from fixed-order fp64 steps.
 *   Batch statistics are used in training and inference alike (the paper defines
 *   no running estimate).
 *   xhat out int16 [m][c] (may be NULL for inference); a out int8 [m][c]; s_a out double
 *   bn_codes out int32[2c]; bn_scales out double[IQ_BN_SCALES]
 *   bn_fixed optional out int64[4c + 2]: F[c], B[c], G[c], H[c], P_x, P_a */
iq_status iq_bn_int_fwd(const int32_t* acc, int64_t m, int32_t c, const double* s_acc,
                        const int32_t* gamma, const int32_t* beta, const iq_bn_bits* bits,
                        int16_t* xhat, int8_t* a, double* s_a, int32_t* bn_codes,
                        double* bn_scales, int64_t* bn_fixed, void* ws, size_t ws_bytes,
                        iq_stream stream);

/* iq_bn_int_fwd_noalloc -- iq_bn_int_fwd without a workspace argument.  The paper has
 * no counterpart: it serves callers that may not allocate device memory themselves (a
 * plugin inside a host application that owns all device allocations, a real-time loop
 * that must not allocate after start-up).  Its scratch is a fixed file-scope device
 * array of 320 KB that every GPU loading the library keeps until process exit; it
 * accepts c <= 4096 channels and returns IQ_ERR_UNSUPPORTED above that.  Every call looks
 * up that array's device address in the CUDA context current at the call (the address
 * belongs to a context, not to a device, so a context the host application made current,
 * or one created after a reset, is served correctly); the first call in a context also
 * loads the library's device code there, so make it before any stream capture.  All calls
 * share the one array: every call re-initialises the statistics it needs, but calls whose
 * work overlaps on the GPU (different streams, no ordering) race on it.  Otherwise
 * identical to iq_bn_int_fwd, with the same outputs. */
iq_status iq_bn_int_fwd_noalloc(const int32_t* acc, int64_t m, int32_t c, const double* s_acc,
                                const int32_t* gamma, const int32_t* beta,
                                const iq_bn_bits* bits, int16_t* xhat, int8_t* a, double* s_a,
                                int32_t* bn_codes, double* bn_scales, int64_t* bn_fixed,
                                iq_stream stream);

/* iq_bn_int_bwd -- backward through Q_A/ReLU and the quantized L1BN (Sec. 3.3.1):
 *   e_y = e_a where a > 0 (ReLU mask of the stored activation codes);
 *   dbeta[c] = sum e_y (scale s_e), dgamma[c] = sum e_y X (scale s_e s_xhat), int64 out;
 *   E_2 = SQ(gamma_q e_y, k_e2), Eq. (EQ);
 *   dx_i = (1/(sigma_q+eps)) [g_i - mean g - mean(g xhat) (sign X_i - mean sign X)],
 *   the derivative of Eqs. (BN4),(BN5) (straight-through for the mu/sigma quantizers);
 *   e = SQ(dx, 8), the conv-output error fed to iq_conv_dgrad / iq_conv_wgrad.
 *   e_a, s_e   int8 [m][c] error codes of this layer's activation and their scale
 *   a, xhat    the forward outputs;  gamma int32[c];  bn_codes, bn_scales from the forward
 *   e          out int8 [m][c];  s_e_out out device double
 *   e_f16      optional out fp16 [m][c] (16-byte aligned, m c % 16 == 0, else
 *              IQ_ERR_INVALID_ARG): the exact fp16 copy of e, written with it, for
 *              iq_conv_dgrad under IQ_CONV_E_F16_READY (no counterpart in the paper)
 * Workspace: iq_bn_int_workspace_size(m, c) (for c not a power of two in [16, 1024] nor a
 * multiple of 1024 it grows with m: a per-code histogram of each row tile).  Returns
 * IQ_ERR_UNSUPPORTED for m > 65535 * 65536 rows. */
iq_status iq_bn_int_bwd(const int8_t* e_a, const double* s_e, const int8_t* a,
                        const int16_t* xhat, int64_t m, int32_t c, const int32_t* gamma,
                        const int32_t* bn_codes, const double* bn_scales,
                        const iq_bn_bits* bits, int k_e2, int8_t* e, double* s_e_out,
                        int64_t* dgamma, int64_t* dbeta, void* e_f16, void* ws,
                        size_t ws_bytes, iq_stream stream);

/* iq_relu_bwd -- layers without BN: e = e_a where a > 0, else 0 (same scale).  e_f16:
 * optional out fp16 [n], the exact fp16 copy of e (e_a, a, e and e_f16 16-byte aligned and
 * n % 16 == 0, else IQ_ERR_INVALID_ARG), as e_f16 of iq_bn_int_bwd. */
iq_status iq_relu_bwd(const int8_t* e_a, const int8_t* a, int64_t n, int8_t* e, void* e_f16,
                      iq_stream stream);

/* iq_update -- Eq. (UQ2): Delta W = UQ(G_q lr, k_u) with lr = 2^-lr_log2, plain SGD
 * master <- clip(master - Delta W) on the k_u grid, then wq = UQ(W_m, k_w) (Eq. (WQ1)).
 *   master int32[n] in/out (codes on the k_u grid; x2 != 0: the x2-scaled gamma/beta grid)
 *   wq     out int8[n];  g int8[n] gradient codes with device scale s_g */
iq_status iq_update(int32_t* master, int8_t* wq, const int8_t* g, const double* s_g,
                    int64_t n, int lr_log2, int k_u, int k_w, int x2, iq_stream stream);

/* ---------------------------------------------------------------- network glue
 * (Sec. 2.1 and Sec. 5: the FCN-VGG16 encoder pools, its trainable bilinear-initialised
 * transposed-convolution decoder, and its MSE loss on quantized logits.) */

/* iq_maxpool_fwd -- k x k max pooling, stride s, padding p (padding never wins), on int8
 * codes (positive scale: the scale passes through unchanged).  arg (uint8, output shape)
 * records the tap index r*k + t of the first maximum in scan order for the backward.  y_f16:
 * optional out fp16 copy of y (16-byte aligned, its size % 16 == 0, else
 * IQ_ERR_INVALID_ARG), the x_f16 of the conv that reads y under IQ_CONV_X_F16_READY. */
iq_status iq_maxpool_fwd(const int8_t* x, int32_t n, int32_t h, int32_t w, int32_t c, int32_t k,
                         int32_t s, int32_t p, int8_t* y, uint8_t* arg, void* y_f16,
                         iq_stream stream);

/* iq_maxpool_bwd -- routes each output error to its window's first maximum.  Without
 * overlap (k <= s) the codes pass through and s_ex = s_e; with overlap the int32 sums are
 * requantized with Q_E = SQ(., 8).  n, h, w, c are the INPUT dimensions. */
iq_status iq_maxpool_bwd(const int8_t* e, const double* s_e, const uint8_t* arg, int32_t n,
                         int32_t h, int32_t w, int32_t c, int32_t k, int32_t s, int32_t p,
                         int8_t* ex, double* s_ex, void* ws, size_t ws_bytes, iq_stream stream);

/* Workspace of the three upsampling calls below. */
iq_status iq_upsample_workspace_size(int32_t n, int32_t h, int32_t w, int32_t c, int32_t R,
                                     size_t* bytes);

/* iq_upsample_fwd -- per-channel (depthwise) transposed convolution, the FCN decoder:
 * out[n,H,W,c] = sum_{i,j} x[n,i,j,c] w[c][H+pad-i*stride][W+pad-j*stride] over taps inside
 * the R x R kernel, H = (h-1) stride - 2 pad + R; exact int32, then Q_A = SQ(., 8) (the
 * quantized logits).  x int8 [n][h][w][c] with device scale s_x; w int8 [c][R][R] (scale
 * 2^-7); out int8 [n][H][W][c]; s_out device double; acc_out optional int32. */
iq_status iq_upsample_fwd(const int8_t* x, const double* s_x, const int8_t* w, int32_t n,
                          int32_t h, int32_t wd, int32_t c, int32_t R, int32_t stride,
                          int32_t pad, int8_t* out, double* s_out, int32_t* acc_out, void* ws,
                          size_t ws_bytes, iq_stream stream);

/* iq_upsample_bwd -- its data gradient (Eq. (EQ)): ex[n,i,j,c] = sum_{r,t} E[n, i stride + r - pad,
 * j stride + t - pad, c] w[c][r][t] exact int32, then SQ(., 8).  Dimensions as in the forward. */
iq_status iq_upsample_bwd(const int8_t* E, const double* s_e, const int8_t* w, int32_t n,
                          int32_t h, int32_t wd, int32_t c, int32_t R, int32_t stride,
                          int32_t pad, int8_t* ex, double* s_ex, int32_t* acc_out, void* ws,
                          size_t ws_bytes, iq_stream stream);

/* iq_upsample_wgrad -- its weight gradient g[c][r][t] = sum_{n,i,j} x[n,i,j,c] E[...] exact
 * int64, then Eq. (GQ1) / (GQ2) as in iq_conv_wgrad. */
iq_status iq_upsample_wgrad(const int8_t* x, const double* s_x, const int8_t* E, const double* s_e,
                            int32_t n, int32_t h, int32_t wd, int32_t c, int32_t R, int32_t stride,
                            int32_t pad, int gq_mode, uint64_t seed, uint64_t layer,
                            uint64_t step, int8_t* g, double* s_g, int64_t* g_acc_out, void* ws,
                            size_t ws_bytes, iq_stream stream);

/* iq_mse_grad -- gradient of the MSE loss on quantized logits (Sec. 5, FCN), up to its
 * constant factor: E = z s_z - onehot(label) per pixel and class, then Q_E = SQ(E, 8).
 * z int8 [npix][c] with device scale s_z; labels uint8 [npix] (values >= c: no target);
 * E out int8 [npix][c]; s_e out device double.  ws >= 1024 bytes.  The element map is the
 * fixed-point floor((F z + B_t) / 2^P) of rhu(E 2^7 / max|E|). */
iq_status iq_mse_grad(const int8_t* z, const double* s_z, const uint8_t* labels, int64_t npix,
                      int32_t c, int8_t* E, double* s_e, void* ws, size_t ws_bytes,
                      iq_stream stream);

/* ---------------------------------------------------------------- DeepLab glue
 * (Sec. 5, DeepLabv3-ResNet50: bottleneck residual adds, the ASPP concatenation and its
 * image-pooling branch, the aligned-corner x8 bilinear upsampling of the logits and the
 * softmax cross-entropy loss.  The paper does not say how these are quantized; each call
 * evaluates the real-valued operation on the integer codes exactly (or in fixed point
 * with a 2^-50 relative step) and requantizes with Q_A / Q_E = SQ(., 8).) */

/* One operand of iq_combine.  Its real value per element is a_ch v + b_ch, with v the
 * integer code, a_ch = scale (times gamma_q,ch when gamma is given) and b_ch = beta_q,ch
 * (0 when beta is NULL): a plain quantized tensor, or the BN affine map gamma_q X s_X +
 * beta_q of the X codes of a BN layer (pass the X codes, s_X = bn_scales[IQ_BN_S_XHAT]
 * and the gamma/beta codes). */
typedef struct {
    const void* codes;      /* device codes, dtype IQ_I8 or IQ_I16; [n][hw][c], or
                               [n][c] when bcast != 0 (one value per image and channel,
                               the same at every pixel) */
    int32_t dtype;
    int32_t c;              /* channels of this operand */
    int32_t c_offset;       /* concat: first output channel it fills (sum: must be 0) */
    int32_t bcast;
    const double* scale;    /* device double */
    const int32_t* gamma;   /* optional device int32[c]: codes of gamma_q (scale 2^(2-k_gamma)) */
    const int32_t* beta;    /* optional device int32[c]: codes of beta_q (scale 2^(2-k_beta)) */
    int32_t k_gamma, k_beta;
} iq_term;

#define IQ_MAX_TERMS 8

/* Workspace of iq_combine. */
iq_status iq_combine_workspace_size(const iq_term* terms, int32_t n_terms, size_t* bytes);

/* iq_combine -- out = SQ(act(sum of operands), 8), Eq. (AQ1) / (EQ), with act = ReLU when
 * relu != 0.  concat == 0: every operand covers all c_out channels (the residual add of a
 * bottleneck, the sum of the errors that reach one tensor); concat != 0: operand t covers
 * channels [c_offset, c_offset + c) (the ASPP concatenation; overlapping ranges add).
 * The sum is evaluated in fixed point: z = sum_t (F_t,ch v + B_t,ch), F = rhu(a 2^P),
 * B = rhu(b 2^P), one shift P per call = 50 - (binary exponent of 1 + sum_t max_ch
 * (|a| vmax + |b|)) (vmax 127 or 32767), at most 62; then code = floor((256 z + M)/(2M))
 * clipped to +-127 with M = max |z|, and s_out = M 2^(-P-7) (M = 0: zero codes,
 * s_out = 2^(-P-7)).  n images of hw pixels; terms is a host array of 1..IQ_MAX_TERMS
 * descriptors (device pointers inside); out int8 [n][hw][c_out]; s_out device double.
 * out_f16: optional out fp16 copy of out (16-byte aligned, n hw c_out % 16 == 0, else
 * IQ_ERR_INVALID_ARG), the x_f16 of a conv that reads out under IQ_CONV_X_F16_READY (no
 * counterpart in the paper). */
iq_status iq_combine(const iq_term* terms, int32_t n_terms, int32_t concat, int64_t n,
                     int64_t hw, int32_t c_out, int32_t relu, int8_t* out, double* s_out,
                     void* out_f16, void* ws, size_t ws_bytes, iq_stream stream);

/* Workspace of iq_spatial_sum. */
iq_status iq_spatial_sum_workspace_size(int64_t n, int32_t c, size_t* bytes);

/* iq_spatial_sum -- per image, the sum over its hw pixels of channels [c_off, c_off + c) of
 * x [n][hw][c_total] (int8 codes, device scale s_x), then SQ(., 8) of the n x c sums.
 *   mean != 0: global average pooling (the ASPP image-pooling branch): real value s_x
 *              sum / hw, s_out = ((s_x M) / hw) 2^-7 (the 1/hw cancels in the codes);
 *   mean == 0: the backward of a broadcast over the pixels, s_out = (s_x M) 2^-7.
 * M = 0 gives zero codes and s_out = (s_x / hw or s_x) 2^-7.  out int8 [n][c]. */
iq_status iq_spatial_sum(const int8_t* x, const double* s_x, int64_t n, int64_t hw,
                         int32_t c_total, int32_t c_off, int32_t c, int32_t mean, int8_t* out,
                         double* s_out, void* ws, size_t ws_bytes, iq_stream stream);

/* iq_avgpool_bwd -- error of the input of a global average pooling: every pixel of image
 * i gets the pooled error e[i][c] / hw.  s_ex = s_e / hw (IEEE division); when ex is not
 * NULL the codes e are broadcast into ex [n][hw][c]; otherwise pass e as a bcast operand
 * with scale s_ex to iq_combine. */
iq_status iq_avgpool_bwd(const int8_t* e, const double* s_e, int64_t n, int64_t hw, int32_t c,
                         int8_t* ex, double* s_ex, iq_stream stream);

/* iq_channel_slice -- out[p][j] = x[p][c_off + j] for j < c (codes only: the error of one
 * operand of a concatenation, whose scale is that of the concatenated error). */
iq_status iq_channel_slice(const int8_t* x, int64_t npix, int32_t c_total, int32_t c_off,
                           int32_t c, int8_t* out, iq_stream stream);

/* Workspace of the two bilinear calls. */
iq_status iq_bilinear_workspace_size(int32_t n, int32_t h, int32_t w, int32_t c, size_t* bytes);

/* iq_bilinear_up_fwd -- bilinear upsampling by an integer factor f with aligned corners,
 * output (h-1) f + 1 by (w-1) f + 1 (f = 8: the DeepLab logits 65 -> 513).  Output pixel
 * (f i + r, f j + t) has the integer numerator (f-r)(f-t) x[i][j] + r(f-t) x[i+1][j] +
 * (f-r) t x[i][j+1] + r t x[i+1][j+1] (real value numerator s_x / f^2), exact; codes =
 * SQ(., 8) of the numerators, s_out = ((s_x M) / f^2) 2^-7.  x int8 [n][h][w][c];
 * out int8 [n][H][W][c]. */
iq_status iq_bilinear_up_fwd(const int8_t* x, const double* s_x, int32_t n, int32_t h,
                             int32_t w, int32_t c, int32_t f, int8_t* out, double* s_out,
                             void* ws, size_t ws_bytes, iq_stream stream);

/* iq_bilinear_up_bwd -- its adjoint on errors: ex[i][j] = sum over the outputs that read
 * x[i][j] of (integer weight) e, exact int32, then SQ(., 8); s_ex = ((s_e M) / f^2) 2^-7.
 * e int8 [n][H][W][c]; ex int8 [n][h][w][c] (h, w the INPUT size of the forward). */
iq_status iq_bilinear_up_bwd(const int8_t* e, const double* s_e, int32_t n, int32_t h,
                             int32_t w, int32_t c, int32_t f, int8_t* ex, double* s_ex,
                             void* ws, size_t ws_bytes, iq_stream stream);

/* iq_ce_grad -- gradient of the softmax cross-entropy loss (mean over labelled pixels) on
 * quantized logits, the DeepLab loss: per pixel t_c = (z_c - max z) * (float)s_z,
 * e_c = exp(t_c) by a fixed fp32 sequence (Cody-Waite reduction with ln 2 split into
 * 0x1.62e4p-1 + 0x1.7f7d1cp-20, k = floor(t log2e + 1/2), Taylor polynomial of degree 7
 * in Horner form, no fused multiply-add, 0 below t = -87), S = sum of e_c in class order,
 * p_c = e_c / S, g_c = p_c - [c == label]; pixels labelled `ignore` give g = 0.  Then
 * Q_E on the float tensor: G = max |g|, code = rhu(fl(g / G) 128) clipped to +-127, and
 * s_e = (G 2^-7) / n_valid (G = 0: zero codes, s_e = 2^-7 / max(n_valid, 1)).
 *   z int8 [npix][c] (c <= 1024), device scale s_z; labels uint8 [npix]; E out int8
 *   [npix][c]; s_e out device double; n_valid optional out device int64. */
iq_status iq_ce_grad(const int8_t* z, const double* s_z, const uint8_t* labels, int64_t npix,
                     int32_t c, int32_t ignore, int8_t* E, double* s_e, int64_t* n_valid,
                     void* ws, size_t ws_bytes, iq_stream stream);

/* iq_bn_update -- Sec. 3.3.3 for the L1BN parameters: the sums dgamma (scale s_e s_X,
 * s_X = bn_scales[IQ_BN_S_XHAT]) and dbeta (scale s_e) from iq_bn_int_bwd are quantized
 * with Eq. (GQ1) (RQ to 8 bits, Philox key (seed, layer), counter (i/8, step, tag, 0) with
 * tag 1 for gamma and 2 for beta), then master <- clip(master - UQ(G_q lr, k_u)) on the
 * x2 grid (value master 2^(2-k_u)), lr = 2^-lr_log2, and the codes gamma = UQ2(master,
 * k_gamma), beta = UQ2(master, k_beta) used by the forward.  All arrays int32[c] on the
 * device (c <= 4096, else IQ_ERR_UNSUPPORTED); gamma_master / beta_master in/out, gamma /
 * beta out.  ws / ws_bytes are reserved: the update needs no scratch, and NULL / 0 are
 * accepted.  One launch. */
iq_status iq_bn_update(int32_t* gamma_master, int32_t* beta_master, int32_t* gamma,
                       int32_t* beta, const int64_t* dgamma, const int64_t* dbeta,
                       const double* s_e, const double* bn_scales, int32_t c,
                       const iq_bn_bits* bits, int lr_log2, int k_u, uint64_t seed,
                       uint64_t layer, uint64_t step, void* ws, size_t ws_bytes,
                       iq_stream stream);

#ifdef __cplusplus
}
#endif
#endif /* IQ_H */
