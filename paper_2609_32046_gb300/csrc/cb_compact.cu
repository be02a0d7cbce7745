// Gather-compact of the selected positions' K/V rows for every layer and KV head
// into the caller's send buffer (the message of App. C.3 carried as K/V rows).
//
// A sender's rows are enumerated as ((kv * n_layers + l) * Hkv + g) * B + j, so
// consecutive threads copy consecutive 16-byte pieces of consecutive output rows
// (coalesced stores, one index load per row).  Each thread moves UNROLL pieces
// per iteration with all loads issued before the stores, keeping enough bytes in
// flight for HBM; loads bypass L1 and stores are marked streaming.  Indices are
// bounds-checked: a bad one is skipped and recorded in the device error word.
#include <cstdint>
#include <cuda_runtime.h>

#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;

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

template <int D>
__global__ void __launch_bounds__(kThreads) k_compact(const __grid_constant__ CompactBatch bt) {
    constexpr int CH = D / 8;  // 16-byte pieces per row
    const CompactSender& sd = bt.s[blockIdx.y];
    const int nL = bt.n_layers, Hkv = bt.n_kv_heads;
    const int64_t B = sd.B;
    const int64_t pieces = (int64_t)2 * nL * Hkv * B * CH;
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    for (int64_t base = (int64_t)blockIdx.x * kThreads + threadIdx.x; base < pieces; base += stride * kUnroll) {
        uint4 val[kUnroll];
        uint4* dst[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            dst[u] = nullptr;
            const int64_t e = base + u * stride;
            if (e >= pieces) continue;
            // pieces of one sender stay below 2^31 (checked on the host): 32-bit index math
            const uint32_t row = (uint32_t)e / CH;
            const int ch = (int)((uint32_t)e % CH);
            const uint32_t j = row % (uint32_t)B;
            uint32_t rest = row / (uint32_t)B;
            const int g = (int)(rest % (uint32_t)Hkv);
            rest /= (uint32_t)Hkv;
            const int l = (int)(rest % (uint32_t)nL);
            const int kv = (int)(rest / (uint32_t)nL);
            const int32_t t = __ldg(sd.idx + j);
            if (t < 0 || t >= sd.T) {
                atomicOr(bt.err, kErrCompactIndex);
                continue;
            }
            const uint16_t* src = (kv ? sd.v : sd.k) + (int64_t)l * sd.ks_l + (int64_t)g * sd.ks_h +
                                  (int64_t)t * sd.ks_p + ch * 8;
            uint16_t* out = (kv ? bt.v_out : bt.k_out) + (int64_t)l * bt.o_layer + (int64_t)g * bt.o_head +
                            (sd.out_off + j) * D + ch * 8;
            val[u] = ld_stream(reinterpret_cast<const uint4*>(src));
            dst[u] = reinterpret_cast<uint4*>(out);
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (dst[u]) st_stream(dst[u], val[u]);
    }
}

}  // namespace

cudaError_t launch_compact(const CompactBatch& b, cudaStream_t st, int num_sms) {
    int64_t max_pieces = 0;
    for (int i = 0; i < b.n; ++i) {
        const int64_t p = (int64_t)2 * b.n_layers * b.n_kv_heads * b.s[i].B * (b.head_dim / 8);
        max_pieces = p > max_pieces ? p : max_pieces;
    }
    if (max_pieces == 0) return cudaSuccess;
    // about 8 resident blocks per SM over the whole batch
    int64_t per = ((int64_t)num_sms * 8 + b.n - 1) / b.n;
    const int64_t need = (max_pieces + (int64_t)kThreads * kUnroll - 1) / ((int64_t)kThreads * kUnroll);
    if (per > need) per = need;
    if (per < 1) per = 1;
    dim3 grid((unsigned)per, (unsigned)b.n);
    if (b.head_dim == 128)
        k_compact<128><<<grid, kThreads, 0, st>>>(b);
    else
        k_compact<64><<<grid, kThreads, 0, st>>>(b);
    return cudaGetLastError();
}

}  // namespace cbk
