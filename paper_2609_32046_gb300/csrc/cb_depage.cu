// Contiguous copy of paged sender caches (the tcgen05 score passes read K through TMA tensor
// maps, whose fixed tile shape a page boundary inside a tile would break).
//
// Position t of a paged sender is row t mod P of page pages[t / P] (the block table); the copy
// is K[l][g][t][:] in the plain [nL][Hkv][T][d] layout.  Consecutive threads take consecutive
// 16-byte pieces of the rows of one position, heads next, positions last, so reads follow a
// vLLM page ([row][head][d] contiguous) and writes are whole 256-byte rows.  Each thread moves
// kUnroll pieces with all loads issued before the stores.  A block-table entry outside the
// pool is never dereferenced: its rows are written as zeros and the error word records it.
#include <cstdint>
#include <cuda_runtime.h>

#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;
constexpr int kPieces = 16;   // 16-byte pieces of a d = 128 row

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// Grid: x = slice of (position, head, piece) triples, y = sender, z = layer.
__global__ void __launch_bounds__(kThreads) k_depage(const __grid_constant__ DepageBatch db) {
    const DepageSender& sd = db.s[blockIdx.y];
    const int l = blockIdx.z;
    const int Hkv = db.n_kv_heads;
    const int64_t total = sd.T * Hkv * kPieces;
    const uint16_t* src = sd.k + (int64_t)l * sd.ks_l;
    uint16_t* dst = sd.out + (int64_t)l * Hkv * sd.T * 128;
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    for (int64_t e0 = (int64_t)blockIdx.x * kThreads + threadIdx.x; e0 < total; e0 += stride * kUnroll) {
        uint4 v[kUnroll];
        int64_t at[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int64_t e = e0 + u * stride;
            at[u] = -1;
            if (e >= total) continue;
            const int piece = (int)(e & (kPieces - 1));
            const int64_t rest = e >> 4;
            int g;
            int64_t t;
            if (rest <= 0xffffffffll) {   // 32-bit division where it suffices
                g = (int)((uint32_t)rest % (uint32_t)Hkv);
                t = (int64_t)((uint32_t)rest / (uint32_t)Hkv);
            } else {
                g = (int)(rest % Hkv);
                t = rest / Hkv;
            }
            at[u] = ((int64_t)g * sd.T + t) * 128 + piece * 8;
            const int64_t ro = row_offset(sd.pm, sd.ks_p, t);
            if (ro < 0) {
                if (piece == 0) atomicOr(db.err, kErrPageIndex);
                v[u] = make_uint4(0u, 0u, 0u, 0u);
            } else {
                v[u] = ld_stream(reinterpret_cast<const uint4*>(src + (int64_t)g * sd.ks_h + ro + piece * 8));
            }
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (at[u] >= 0) *reinterpret_cast<uint4*>(dst + at[u]) = v[u];
    }
}

}  // namespace

cudaError_t launch_depage(const DepageBatch& b, cudaStream_t st, int num_sms) {
    if (b.n == 0) return cudaSuccess;
    int64_t maxT = 0;
    for (int i = 0; i < b.n; ++i) maxT = b.s[i].T > maxT ? b.s[i].T : maxT;
    const int64_t pieces = maxT * b.n_kv_heads * kPieces;
    // about 48 blocks per SM over the whole grid (six waves of eight resident blocks): more,
    // shorter blocks kept more of the copy in flight than one wave of long ones
    int64_t x = ((int64_t)num_sms * 48) / ((int64_t)b.n * b.n_layers);
    const int64_t need = (pieces + (int64_t)kThreads * kUnroll - 1) / ((int64_t)kThreads * kUnroll);
    if (x > need) x = need;
    if (x < 1) x = 1;
    dim3 grid((unsigned)x, (unsigned)b.n, (unsigned)b.n_layers);
    k_depage<<<grid, kThreads, 0, st>>>(b);
    return cudaGetLastError();
}

}  // namespace cbk
