// Compaction with the positional re-index direct K/V transfer needs: rotary embeddings rotate
// each pair of K's dimensions by pos * theta_k (theta_k = base^(-2k/d)), so a row rotated for
// sender position t becomes the row for receiver position p by one more rotation by
// (p - t) * theta_k.  App. C.3 notes this sender/receiver mismatch of sending K/V rows as they are
// (the paper re-prefills instead).  Row j of a sender's message sits at receiver position
// pos0 + out_off + j.  V rows are copied unchanged.
//
// The angle is reduced exactly in fixed point: with F_k = theta_k / (2 pi) * 2^64 (host, long
// double), (p - t) * F_k modulo 2^64 is the angle in turns; its top 32 bits give the angle in
// [-pi, pi) to 2^-32 of a turn, whose sine and cosine come from the hardware approximations
// (absolute error near 2^-21, far below the bf16 rounding of the result).  Pairs are
// (k, k + d/2) (style 0, halves) or (2k, 2k + 1) (style 1, interleaved).
#include <cmath>
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kThreads = 256;

struct RopeBatch {
    CompactBatch c;
    int64_t pos0;
    uint64_t turns[64];   // F_k for k < d/2
};

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

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t bf_pack(float lo, float hi) {
    return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo)) |
           ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi)) << 16);
}

// sin and cos of delta * theta_k from the fixed-point turns F_k.
__device__ __forceinline__ void rot(int64_t delta, uint64_t F, float& s, float& c) {
    const uint64_t turns = (uint64_t)delta * F;                       // modulo 2^64: exact reduction
    const float ang = (float)(int32_t)(uint32_t)(turns >> 32) * 1.4629180792671596e-09f;   // 2 pi / 2^32
    s = __sinf(ang);
    c = __cosf(ang);
}

// Grid: x = (K or V, layer, head) segment, y = sender, z = slice of the segment's rows.
// K segments, style 0: a thread owns pieces c and c + D/16 (the two halves of 8 pairs);
// style 1 and V segments: a thread owns one 16-byte piece.
template <int D, int STYLE>
__global__ void __launch_bounds__(kThreads) k_compact_rope(const __grid_constant__ RopeBatch rb) {
    const CompactBatch& bt = rb.c;
    const CompactSender& sd = bt.s[blockIdx.y];
    const int seg = blockIdx.x;
    const int g = seg % bt.n_kv_heads;
    const int l = (seg / bt.n_kv_heads) % bt.n_layers;
    const int kv = seg / (bt.n_kv_heads * bt.n_layers);
    const uint16_t* src = (kv ? sd.v : sd.k) + (int64_t)l * sd.ks_l + (int64_t)g * sd.ks_h;
    uint16_t* dst = (kv ? bt.v_out : bt.k_out) + (int64_t)l * bt.o_layer + (int64_t)g * bt.o_head + sd.out_off * D;
    const bool halves = kv == 0 && STYLE == 0;
    const int per_row = halves ? D / 16 : D / 8;          // threads per row
    const int rows = kThreads / per_row;                   // rows per block pass
    const int ch = threadIdx.x % per_row;
    const int64_t stride = (int64_t)rows * gridDim.z;
    for (int64_t j = (int64_t)blockIdx.z * rows + threadIdx.x / per_row; j < sd.B; j += stride) {
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
        const uint16_t* srow = src + ro;
        uint16_t* drow = dst + j * D;
        if (kv) {
            st_stream(reinterpret_cast<uint4*>(drow + ch * 8), ld_stream(reinterpret_cast<const uint4*>(srow + ch * 8)));
            continue;
        }
        const int64_t delta = rb.pos0 + sd.out_off + j - t;
        if (halves) {
            // elements 8 ch .. +7 pair with 8 ch + D/2 .. +7 (pairs k = 8 ch + e)
            const uint4 a = ld_stream(reinterpret_cast<const uint4*>(srow + ch * 8));
            const uint4 b = ld_stream(reinterpret_cast<const uint4*>(srow + ch * 8 + D / 2));
            const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
            uint32_t oa[4], ob[4];
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                float s0, c0, s1, c1;
                rot(delta, rb.turns[ch * 8 + 2 * w], s0, c0);
                rot(delta, rb.turns[ch * 8 + 2 * w + 1], s1, c1);
                const float xa0 = bf_lo(aw[w]), xa1 = bf_hi(aw[w]), xb0 = bf_lo(bw[w]), xb1 = bf_hi(bw[w]);
                oa[w] = bf_pack(xa0 * c0 - xb0 * s0, xa1 * c1 - xb1 * s1);
                ob[w] = bf_pack(xb0 * c0 + xa0 * s0, xb1 * c1 + xa1 * s1);
            }
            st_stream(reinterpret_cast<uint4*>(drow + ch * 8), make_uint4(oa[0], oa[1], oa[2], oa[3]));
            st_stream(reinterpret_cast<uint4*>(drow + ch * 8 + D / 2), make_uint4(ob[0], ob[1], ob[2], ob[3]));
        } else {
            // interleaved: each 32-bit word is one pair (2k, 2k + 1), k = 4 ch + w
            const uint4 a = ld_stream(reinterpret_cast<const uint4*>(srow + ch * 8));
            const uint32_t aw[4] = {a.x, a.y, a.z, a.w};
            uint32_t o[4];
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                float s, c;
                rot(delta, rb.turns[ch * 4 + w], s, c);
                const float x0 = bf_lo(aw[w]), x1 = bf_hi(aw[w]);
                o[w] = bf_pack(x0 * c - x1 * s, x1 * c + x0 * s);
            }
            st_stream(reinterpret_cast<uint4*>(drow + ch * 8), make_uint4(o[0], o[1], o[2], o[3]));
        }
    }
}

}  // namespace

cudaError_t launch_compact_rope(const CompactBatch& b, double base, int style, int64_t pos0, cudaStream_t st,
                                int num_sms) {
    int64_t max_B = 0;
    for (int i = 0; i < b.n; ++i) max_B = b.s[i].B > max_B ? b.s[i].B : max_B;
    if (max_B == 0) return cudaSuccess;
    RopeBatch* rb = new RopeBatch();
    rb->c = b;
    rb->pos0 = pos0;
    const int half = b.head_dim / 2;
    const long double two_pi = 6.283185307179586476925286766559L;
    for (int k = 0; k < half; ++k) {
        const long double f = powl((long double)base, -2.0L * k / b.head_dim) / two_pi;   // turns per position
        rb->turns[k] = (uint64_t)ldexpl(f, 64);
    }
    const int segs = 2 * b.n_layers * b.n_kv_heads;
    // about 48 blocks per SM over the batch (six waves of eight resident blocks); each block walks a
    // slice of its segment's rows
    const int rows_per_pass = kThreads / (b.head_dim / 8);
    int64_t slices = ((int64_t)num_sms * 48) / ((int64_t)segs * b.n);
    const int64_t need = (max_B + rows_per_pass - 1) / rows_per_pass;
    if (slices > need) slices = need;
    if (slices < 1) slices = 1;
    if (slices > 65535) slices = 65535;
    dim3 grid((unsigned)segs, (unsigned)b.n, (unsigned)slices);
    if (b.head_dim == 128) {
        if (style == 0) k_compact_rope<128, 0><<<grid, kThreads, 0, st>>>(*rb);
        else k_compact_rope<128, 1><<<grid, kThreads, 0, st>>>(*rb);
    } else {
        if (style == 0) k_compact_rope<64, 0><<<grid, kThreads, 0, st>>>(*rb);
        else k_compact_rope<64, 1><<<grid, kThreads, 0, st>>>(*rb);
    }
    delete rb;
    return cudaGetLastError();
}

}  // namespace cbk
