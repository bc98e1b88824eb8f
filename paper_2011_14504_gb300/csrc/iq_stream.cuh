// iq_stream.cuh -- streaming of row-major [m][C] tensors through shared memory for the
// bandwidth-bound per-channel passes (integer L1BN forward and backward).
//
// A block of kStreamThreads threads (one per SM) owns a slab of CB channels (all C
// channels when C is a power of two up to 4 kStreamThreads = 2048, else 1024 of them) and a
// strided sequence of row chunks of that slab.  Thread 0 keeps kStreamStages chunks in flight with 1-D bulk copies
// (cp.async.bulk, one per array per chunk when the slab is the whole row, else one per row)
// whose bytes complete an mbarrier; the warps read a landed chunk from shared memory and
// release its stage on a second mbarrier (one arrival per warp), after which thread 0
// refills it.  The copy engine, not the registers of many resident threads, keeps the
// bytes in flight: about 130 KB per SM, against roughly 45 KB that 768 threads with four
// 16-byte loads each keep.
//
// Thread t owns channel group g = t % (CB / 4) (four channels) of the slab and row lane
// t / (CB / 4); a chunk is RL = 2048 / CB row lanes x kStreamRPT rows, so every stage holds
// 16384 elements of each array whatever C is.
#pragma once

#include "iq_common.cuh"
#include "iq_tc_ptx.cuh"

namespace iq {

constexpr int kStreamThreads = 512;
constexpr int kStreamStages = 3;
constexpr int kStreamRPT = 8;                 // rows per thread per chunk
constexpr int kStreamMaxArr = 3;
constexpr int kStreamElems = kStreamThreads * 4 * kStreamRPT;   // elements per array per chunk

struct RowStream {
    const uint8_t* src[kStreamMaxArr];
    int32_t esz[kStreamMaxArr];               // element bytes; 0: no such array
    int32_t off[kStreamMaxArr];               // byte offset of each array in a stage
    int64_t m;                                // rows
    int32_t C, CB;                            // channels; channels per slab
    int32_t R;                                // rows per chunk
    int32_t RL;                               // row lanes
    int32_t stage_bytes;
    int64_t nchunk;                           // chunks per slab
};

// Host: plan the streaming of up to three [m][C] arrays (src[i] with esz[i]-byte elements,
// 16-byte aligned).  False when the shape does not fit: C must be a power of two in
// [16, 2048] or a multiple of 1024.  A slab of whole rows lands with one copy per array
// per chunk, a narrower one with one copy per row.
inline bool row_stream_plan(RowStream& s, int64_t m, int32_t C, const void* const* src,
                            const int* esz, int narr) {
    if (m <= 0 || narr < 1 || narr > kStreamMaxArr) return false;
    if (C >= 16 && C <= 4 * kStreamThreads && (C & (C - 1)) == 0) s.CB = C;
    else if (C > 1024 && C % 1024 == 0) s.CB = 1024;
    else return false;
    s.m = m;
    s.C = C;
    s.RL = kStreamThreads / (s.CB / 4);
    s.R = s.RL * kStreamRPT;
    int off = 0;
    for (int i = 0; i < kStreamMaxArr; i++) {
        s.src[i] = i < narr ? static_cast<const uint8_t*>(src[i]) : nullptr;
        s.esz[i] = i < narr ? esz[i] : 0;
        s.off[i] = off;
        if (i < narr) {
            if (reinterpret_cast<uintptr_t>(src[i]) & 15) return false;
            off += s.R * s.CB * esz[i];
        }
    }
    s.stage_bytes = (off + 127) & ~127;
    s.nchunk = (m + s.R - 1) / s.R;
    return true;
}

inline size_t row_stream_smem(const RowStream& s) {
    return (size_t)kStreamStages * s.stage_bytes + 2 * kStreamStages * sizeof(uint64_t);
}

// grid: (slabs, row-chunk lanes), one block per SM in all
inline dim3 row_stream_grid(const RowStream& s, int sms) {
    const int nslab = s.C / s.CB;
    int64_t gy = sms / nslab;
    if (gy < 1) gy = 1;
    if (gy > s.nchunk) gy = s.nchunk;
    if (gy > 65535) gy = 65535;
    return dim3((unsigned)nslab, (unsigned)gy);
}

// thread 0: issue the copies of chunk k of slab `slab` into `stage`, counted on `bar`
__device__ __forceinline__ void stream_issue(const RowStream& s, uint8_t* stage, uint64_t* bar,
                                             int64_t k, int slab) {
    const int64_t r0 = k * s.R;
    const int rows = (int)((s.m - r0) < s.R ? (s.m - r0) : s.R);
    uint32_t bytes = 0;
#pragma unroll
    for (int a = 0; a < kStreamMaxArr; a++) bytes += (uint32_t)(rows * s.CB * s.esz[a]);
    tc::mbar_arrive_expect_tx(bar, bytes);
#pragma unroll
    for (int a = 0; a < kStreamMaxArr; a++) {
        const int e = s.esz[a];
        if (!e) continue;
        if (s.CB == s.C) {
            tc::bulk_g2s(stage + s.off[a], s.src[a] + r0 * s.C * e, (uint32_t)(rows * s.C * e),
                         bar);
        } else {
            for (int r = 0; r < rows; r++)
                tc::bulk_g2s(stage + s.off[a] + (size_t)r * s.CB * e,
                             s.src[a] + ((r0 + r) * s.C + (int64_t)slab * s.CB) * e,
                             (uint32_t)(s.CB * e), bar);
        }
    }
}

// The block's pipeline over chunks k = blockIdx.y + i gridDim.y (i = 0, 1, ...) of the
// block's slab, nchunk chunks of R rows each (m rows in all): thread 0 keeps S stages in
// flight, issue(stage, bar, k) arriving on `bar` with the chunk's transaction bytes and
// starting its copies; body(stage, rows, r0) runs on every thread for every landed chunk
// (rows of the chunk, first row).  Every wait is bounded: when one gives up (about a
// second), the kernel stores IQ_ERR_TIMEOUT in *err, waits (bounded again) for the copies
// it issued and every thread returns false.  `smem` holds the S stages of stage_bytes and
// then 2 S barriers.
template <int S, class Issue, class Body>
__device__ __forceinline__ bool pipe_chunks(int64_t nchunk, int R, int64_t m, int stage_bytes,
                                            uint8_t* smem, int* err, Issue&& issue,
                                            Body&& body) {
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * stage_bytes);
    uint64_t* empty = full + S;
    __shared__ int abort_flag, never;
    const int tid = threadIdx.x;
    if (tid == 0) {
        abort_flag = 0;
        never = 0;
        for (int i = 0; i < S; i++) {
            tc::mbar_init(&full[i], 1);
            tc::mbar_init(&empty[i], blockDim.x >> 5);
        }
        tc::mbar_fence_init();
    }
    __syncthreads();
    int issued = 0;                          // thread 0: chunks issued so far
    if (tid == 0) {
        for (int i = 0; i < S; i++) {
            const int64_t k = blockIdx.y + (int64_t)i * gridDim.y;
            if (k >= nchunk) break;
            issue(smem + i * stage_bytes, &full[i], k);
            issued++;
        }
    }
    volatile int* ab = &abort_flag;
    for (int i = 0;; i++) {
        const int64_t k = blockIdx.y + (int64_t)i * gridDim.y;
        if (k >= nchunk) break;
        const int st = i % S;
        const uint32_t par = (uint32_t)((i / S) & 1);
        if (!tc::mbar_wait(&full[st], par, ab)) {
            *ab = 1;
            break;
        }
        const int64_t r0 = k * R;
        const int rows = (int)((m - r0) < R ? (m - r0) : R);
        body(smem + st * stage_bytes, rows, r0);
        __syncwarp();
        if ((tid & 31) == 0) tc::mbar_arrive(&empty[st]);
        if (tid == 0) {
            const int64_t kn = k + (int64_t)S * gridDim.y;
            if (kn < nchunk) {
                // every warp has read this stage: refill it
                if (!tc::mbar_wait(&empty[st], par, ab)) {
                    *ab = 1;
                    break;
                }
                issue(smem + st * stage_bytes, &full[st], kn);
                issued++;
            }
        }
    }
    const bool failed = __syncthreads_or(*ab);
    if (failed) {
        if (tid == 0) {
            atomicExch(err, (int)IQ_ERR_TIMEOUT);
            // let the copies in flight land before the block leaves
            for (int j = (issued > S ? issued - S : 0); j < issued; j++)
                tc::mbar_wait(&full[j % S], (uint32_t)((j / S) & 1), &never);
        }
        __syncthreads();
        return false;
    }
    return true;
}

// the pipeline over a RowStream's chunks of slab blockIdx.x (1-D bulk copies)
template <class Body>
__device__ __forceinline__ bool stream_chunks(const RowStream& s, uint8_t* smem, int* err,
                                              Body&& body) {
    const int slab = blockIdx.x;
    return pipe_chunks<kStreamStages>(
        s.nchunk, s.R, s.m, s.stage_bytes, smem, err,
        [&](uint8_t* stage, uint64_t* bar, int64_t k) { stream_issue(s, stage, bar, k, slab); },
        body);
}

}  // namespace iq
