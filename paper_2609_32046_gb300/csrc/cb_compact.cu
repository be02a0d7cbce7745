// Gather-compact of the selected positions' K/V rows for every layer and KV head
// into the caller's send buffer (the message of App. C.3 carried as K/V rows).
//
// One block per (K or V, layer, KV head) segment of a sender (and slice of its rows):
// consecutive threads copy consecutive 16-byte pieces of consecutive output rows
// (coalesced stores, one index load per row, no per-piece division).  Each thread moves UNROLL pieces
// per iteration with all loads issued before the stores, keeping enough bytes in
// flight for HBM; loads bypass L1 and stores are marked streaming.  Indices (and, for a paged
// cache, block-table entries) are bounds-checked: a bad one is skipped and recorded in the
// device error word.
#include <cstdint>
#include <cuda_runtime.h>

#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 2;

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

// Grid: x = (kv, layer, head) segment of a sender, y = sender, z = slice of the segment's rows.
// Within a segment, row j and 16-byte piece c come from the thread index by shifts only.
template <int D>
__global__ void __launch_bounds__(kThreads) k_compact(const __grid_constant__ CompactBatch bt) {
    constexpr int CH = D / 8;              // 16-byte pieces per row
    constexpr int ROWS = kThreads / CH;    // rows per block pass
    const CompactSender& sd = bt.s[blockIdx.y];
    const int seg = blockIdx.x;
    const int g = seg % bt.n_kv_heads;
    const int l = (seg / bt.n_kv_heads) % bt.n_layers;
    const int kv = seg / (bt.n_kv_heads * bt.n_layers);
    const int64_t B = sd.B;
    const uint16_t* src = (kv ? sd.v : sd.k) + (int64_t)l * sd.ks_l + (int64_t)g * sd.ks_h;
    uint16_t* dst = (kv ? bt.v_out : bt.k_out) + (int64_t)l * bt.o_layer + (int64_t)g * bt.o_head +
                    sd.out_off * D;
    const int ch = threadIdx.x % CH;
    const int64_t stride = (int64_t)ROWS * gridDim.z;
    for (int64_t j0 = (int64_t)blockIdx.z * ROWS + threadIdx.x / CH; j0 < B; j0 += stride * kUnroll) {
        uint4 val[kUnroll];
        bool ok[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int64_t j = j0 + u * stride;
            ok[u] = false;
            if (j >= B) continue;
            const int32_t t = __ldg(sd.idx + j);
            if (t < 0 || t >= sd.T) {
                atomicOr(bt.err, kErrCompactIndex);
                continue;
            }
            const int64_t ro = row_offset(sd.pm, sd.ks_p, t);
            if (ro < 0) {
                atomicOr(bt.err, kErrPageIndex);
                continue;
            }
            val[u] = ld_stream(reinterpret_cast<const uint4*>(src + ro + ch * 8));
            ok[u] = true;
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (ok[u]) st_stream(reinterpret_cast<uint4*>(dst + (j0 + u * stride) * D + ch * 8), val[u]);
    }
}

}  // namespace

cudaError_t launch_compact(const CompactBatch& b, cudaStream_t st, int num_sms) {
    int64_t max_B = 0;
    for (int i = 0; i < b.n; ++i) max_B = b.s[i].B > max_B ? b.s[i].B : max_B;
    if (max_B == 0) return cudaSuccess;
    const int segs = 2 * b.n_layers * b.n_kv_heads;
    const int rows_per_pass = kThreads / (b.head_dim / 8);
    // about 24 blocks per SM over the batch (three waves of eight resident blocks); each block
    // walks its slice of rows (two loads in flight a thread over many blocks moved more bytes
    // than four over fewer)
    int64_t slices = ((int64_t)num_sms * 24) / ((int64_t)segs * b.n);
    const int64_t need = (max_B + (int64_t)rows_per_pass * kUnroll - 1) / ((int64_t)rows_per_pass * kUnroll);
    if (slices > need) slices = need;
    if (slices < 1) slices = 1;
    if (slices > 65535) slices = 65535;
    dim3 grid((unsigned)segs, (unsigned)b.n, (unsigned)slices);
    if (b.head_dim == 128)
        k_compact<128><<<grid, kThreads, 0, st>>>(b);
    else
        k_compact<64><<<grid, kThreads, 0, st>>>(b);
    return cudaGetLastError();
}

}  // namespace cbk
