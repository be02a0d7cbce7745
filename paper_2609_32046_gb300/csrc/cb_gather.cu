// Message rows by index (Sec. 3.1 "State Representation", App. C.3 "Message encoding"):
// the continuous-row encoding sends one row of the sender's per-position table (its hidden
// states, 8 KiB per position for Qwen3-8B) for every selected position; the token-ID encoding
// sends the token IDs of the selected source positions (4-byte rows) and continuous rows for
// the latent positions.  Both are this gather: row j of a sender's message = row idx[j] of its
// table.
//
//   k_gather_vec   rows of a multiple of 16 bytes at 16-byte aligned addresses: one warp per
//                  output row, lanes copy consecutive 16-byte pieces (L1-bypassing loads,
//                  streaming stores)
//   k_gather_word  anything else (4-byte multiples, e.g. token IDs): consecutive threads copy
//                  consecutive 4-byte words of consecutive rows
// Indices are bounds-checked: a bad one is skipped and recorded in the device error word.
#include <cstdint>
#include <cuda_runtime.h>

#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void st_stream(uint4* p, uint4 v) {
    asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

// Grid: x = groups of 8 output rows (grid-stride), y = sender.
__global__ void __launch_bounds__(kThreads) k_gather_vec(const __grid_constant__ GatherBatch bt) {
    const GatherSender& sd = bt.s[blockIdx.y];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t W = bt.row_bytes >> 4;   // 16-byte pieces per row
    for (int64_t j = (int64_t)blockIdx.x * (kThreads / 32) + warp; j < sd.count;
         j += (int64_t)gridDim.x * (kThreads / 32)) {
        const int32_t t = __ldg(sd.idx + j);
        if (t < 0 || t >= sd.T) {
            if (lane == 0) atomicOr(bt.err, kErrGatherIndex);
            continue;
        }
        const uint4* src = reinterpret_cast<const uint4*>(sd.src + (int64_t)t * sd.src_stride);
        uint4* dst = reinterpret_cast<uint4*>(bt.out + (sd.out_off + j) * bt.out_stride);
        int64_t c = lane;
        for (; c + 96 < W; c += 128) {       // four pieces in flight per lane
            const uint4 a = ld_stream(src + c), b = ld_stream(src + c + 32), e = ld_stream(src + c + 64),
                        f = ld_stream(src + c + 96);
            st_stream(dst + c, a);
            st_stream(dst + c + 32, b);
            st_stream(dst + c + 64, e);
            st_stream(dst + c + 96, f);
        }
        for (; c < W; c += 32) st_stream(dst + c, ld_stream(src + c));
    }
}

// Grid: x = blocks over the flattened (row, word) space (grid-stride), y = sender.
__global__ void __launch_bounds__(kThreads) k_gather_word(const __grid_constant__ GatherBatch bt) {
    const GatherSender& sd = bt.s[blockIdx.y];
    const int64_t W = bt.row_bytes >> 2;   // 4-byte words per row
    const int64_t total = sd.count * W;
    for (int64_t f = (int64_t)blockIdx.x * kThreads + threadIdx.x; f < total; f += (int64_t)gridDim.x * kThreads) {
        const int64_t j = f / W, w = f - j * W;
        const int32_t t = __ldg(sd.idx + j);
        if (t < 0 || t >= sd.T) {
            if (w == 0) atomicOr(bt.err, kErrGatherIndex);
            continue;
        }
        const uint32_t v = __ldg(reinterpret_cast<const uint32_t*>(sd.src + (int64_t)t * sd.src_stride) + w);
        reinterpret_cast<uint32_t*>(bt.out + (sd.out_off + j) * bt.out_stride)[w] = v;
    }
}

}  // namespace

cudaError_t launch_gather(const GatherBatch& b, cudaStream_t st, int num_sms) {
    int64_t max_rows = 0;
    bool vec = (b.row_bytes % 16) == 0 && (b.out_stride % 16) == 0 && (reinterpret_cast<uintptr_t>(b.out) % 16) == 0;
    for (int i = 0; i < b.n; ++i) {
        max_rows = b.s[i].count > max_rows ? b.s[i].count : max_rows;
        vec = vec && (b.s[i].src_stride % 16) == 0 && (reinterpret_cast<uintptr_t>(b.s[i].src) % 16) == 0;
    }
    if (max_rows == 0) return cudaSuccess;
    // about 8 resident blocks per SM over the batch
    const int64_t want = ((int64_t)num_sms * 8 + b.n - 1) / b.n;
    if (vec) {
        int64_t gx = (max_rows + kThreads / 32 - 1) / (kThreads / 32);
        gx = gx < want ? gx : want;
        k_gather_vec<<<dim3((unsigned)(gx < 1 ? 1 : gx), (unsigned)b.n), kThreads, 0, st>>>(b);
    } else {
        int64_t gx = (max_rows * (b.row_bytes / 4) + kThreads - 1) / kThreads;
        gx = gx < want ? gx : want;
        k_gather_word<<<dim3((unsigned)(gx < 1 ? 1 : gx), (unsigned)b.n), kThreads, 0, st>>>(b);
    }
    return cudaGetLastError();
}

}  // namespace cbk
