// Span selection (App. C.2, "Budgets and position selection"), one CTA per sender.
//
//   1. S'_0 <- max_t S_t (when a sink is kept); span means over [w j, min(T, w j + w))
//      summed in fp32 in index order and divided by the span's own length.
//   2. The forced positions (first n_sink, last n_latent) count toward B; the
//      remaining need = B - |forced| is filled by spans in rank order
//      (mean descending, earlier span first).  Instead of sorting, a
//      most-significant-digit radix select over the order-preserving key bits of
//      the means, weighted by each span's number of unforced positions, finds
//      the key of the span where the budget runs out.  Spans above that key are
//      taken whole; spans at it are taken in index order (the tie-break), the
//      last one partially.
//   3. The partial span contributes its unforced positions nearest its
//      highest-scoring unforced position (ties to the lower index): a contiguous
//      run of its unforced positions grown outward from that position.
//   4. A block-wide exclusive scan over spans gives each span's output offset,
//      so indices come out in source order.
#include <cfloat>
#include <cstdint>
#include <cuda_runtime.h>

#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kWarps = kSelThreads / 32;

__device__ __forceinline__ uint32_t order_key(float f) {
    const uint32_t u = __float_as_uint(f == 0.f ? 0.f : f);  // -0 ranks with +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

struct Forced {
    int64_t a;   // [0, a) forced (sink)
    int64_t b;   // [b, T) forced (latent)
    __device__ bool at(int64_t t) const { return t < a || t >= b; }
    // number of forced positions in [lo, hi)
    __device__ int64_t count(int64_t lo, int64_t hi) const {
        if (a >= b) return hi - lo;
        const int64_t x = (a < hi ? a : hi) - lo;
        const int64_t y = hi - (b > lo ? b : lo);
        return (x > 0 ? x : 0) + (y > 0 ? y : 0);
    }
};

// Block-wide exclusive scan of one int64 per thread; returns the exclusive prefix, total in *total.
__device__ int64_t block_exclusive_scan(int64_t v, int64_t* sh, int64_t* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int64_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int64_t w = sh[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        sh[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    const int64_t before_warp = warp ? sh[warp - 1] : 0;
    *total = sh[kWarps - 1];
    __syncthreads();
    return before_warp + x - v;
}

__global__ void __launch_bounds__(kSelThreads) k_select(const __grid_constant__ SelectBatch bt) {
    __shared__ uint32_t hist[kWarps][256];
    __shared__ int64_t hsum[256];
    __shared__ int64_t scan_sh[32];
    __shared__ float red[32];
    __shared__ int64_t sel_bucket, sel_before;

    const SelectSender& sd = bt.s[blockIdx.x];
    const int64_t T = sd.T, B = sd.B;
    const int w = bt.span_w;
    const int64_t nsp = (T + w - 1) / w;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float* S = sd.scores;
    Forced F;
    F.a = bt.n_sink < T ? bt.n_sink : T;
    F.b = T - bt.n_latent > 0 ? T - bt.n_latent : 0;

    // 1. maximum score and span means
    float mx = -INFINITY;
    for (int64_t t = tid; t < T; t += kSelThreads) mx = fmaxf(mx, S[t]);
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (lane == 0) red[warp] = mx;
    __syncthreads();
    if (warp == 0) {
        float v = red[lane];
#pragma unroll
        for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) red[0] = v;
    }
    __syncthreads();
    const float smax = red[0];
    for (int64_t j = tid; j < nsp; j += kSelThreads) {
        const int64_t lo = j * w, hi = lo + w < T ? lo + w : T;
        float acc = 0.f;
        for (int64_t t = lo; t < hi; ++t) acc += (t == 0 && bt.n_sink > 0) ? smax : S[t];
        sd.span_keys[j] = __fdiv_rn(acc, (float)(hi - lo));
    }
    const int64_t need = B - F.count(0, T);
    __syncthreads();

    // 2. weighted radix select of the threshold key
    uint32_t prefix = 0u, pmask = 0u;
    int64_t rem = need;
    if (need > 0) {
        for (int pass = 0; pass < 4; ++pass) {
            const int shift = 24 - 8 * pass;
            for (int k = tid; k < kWarps * 256; k += kSelThreads) (&hist[0][0])[k] = 0u;
            __syncthreads();
            for (int64_t j = tid; j < nsp; j += kSelThreads) {
                const uint32_t key = order_key(sd.span_keys[j]);
                if ((key & pmask) != prefix) continue;
                const int64_t lo = j * w, hi = lo + w < T ? lo + w : T;
                const uint32_t u = (uint32_t)((hi - lo) - F.count(lo, hi));
                if (u) atomicAdd(&hist[warp][(key >> shift) & 255u], u);
            }
            __syncthreads();
            if (tid < 256) {
                int64_t v = 0;
                for (int k = 0; k < kWarps; ++k) v += hist[k][tid];
                hsum[tid] = v;
            }
            __syncthreads();
            if (warp == 0) {
                // lane L owns buckets 255-8L .. 248-8L (descending key order)
                int64_t mine = 0;
#pragma unroll
                for (int k = 0; k < 8; ++k) mine += hsum[255 - 8 * lane - k];
                int64_t incl = mine;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int64_t y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const int64_t excl = incl - mine;
                const bool crosses = (excl < rem) && (rem <= incl);
                const unsigned ballot = __ballot_sync(0xffffffffu, crosses);
                if (crosses && lane == __ffs(ballot) - 1) {
                    int64_t before = excl;
                    for (int k = 0; k < 8; ++k) {
                        const int bucket = 255 - 8 * lane - k;
                        if (before + hsum[bucket] >= rem) { sel_bucket = bucket; sel_before = before; break; }
                        before += hsum[bucket];
                    }
                }
            }
            __syncthreads();
            prefix |= (uint32_t)sel_bucket << shift;
            pmask |= 255u << shift;
            rem -= sel_before;
            __syncthreads();
        }
    }
    const uint32_t kappa = prefix;

    // 3. per-span counts; each thread owns a contiguous range of spans
    const int64_t per = (nsp + kSelThreads - 1) / kSelThreads;
    const int64_t j0 = (int64_t)tid * per < nsp ? (int64_t)tid * per : nsp;
    const int64_t j1 = j0 + per < nsp ? j0 + per : nsp;
    int64_t tie_mine = 0;
    if (need > 0)
        for (int64_t j = j0; j < j1; ++j)
            if (order_key(sd.span_keys[j]) == kappa) {
                const int64_t lo = j * w, hi = lo + w < T ? lo + w : T;
                tie_mine += (hi - lo) - F.count(lo, hi);
            }
    int64_t tie_total;
    int64_t tie_before = block_exclusive_scan(tie_mine, scan_sh, &tie_total);
    int64_t cnt_mine = 0;
    {
        int64_t tb = tie_before;
        for (int64_t j = j0; j < j1; ++j) {
            const int64_t lo = j * w, hi = lo + w < T ? lo + w : T;
            const int64_t f = F.count(lo, hi), u = (hi - lo) - f;
            int64_t take = 0;
            if (need > 0) {
                const uint32_t key = order_key(sd.span_keys[j]);
                if (key > kappa) take = u;
                else if (key == kappa) {
                    take = rem - tb;
                    take = take < 0 ? 0 : (take > u ? u : take);
                    tb += u;
                }
            }
            cnt_mine += f + take;
        }
    }
    int64_t total;
    int64_t out = block_exclusive_scan(cnt_mine, scan_sh, &total);
    if (tid == 0 && total != B) atomicOr(bt.err, kErrSelectBudget);

    // 4. write positions in source order
    {
        int64_t tb = tie_before;
        for (int64_t j = j0; j < j1; ++j) {
            const int64_t lo = j * w, hi = lo + w < T ? lo + w : T;
            const int64_t f = F.count(lo, hi), u = (hi - lo) - f;
            int64_t take = 0;
            if (need > 0) {
                const uint32_t key = order_key(sd.span_keys[j]);
                if (key > kappa) take = u;
                else if (key == kappa) {
                    take = rem - tb;
                    take = take < 0 ? 0 : (take > u ? u : take);
                    tb += u;
                }
            }
            if (take == u) {
                for (int64_t t = lo; t < hi; ++t)
                    if (out < B) sd.idx[out++] = (int32_t)t;
            } else if (take == 0) {
                for (int64_t t = lo; t < hi; ++t)
                    if (F.at(t) && out < B) sd.idx[out++] = (int32_t)t;
            } else {
                // highest-scoring unforced position (lowest index on ties)
                int64_t c = -1;
                for (int64_t t = lo; t < hi; ++t)
                    if (!F.at(t) && (c < 0 || S[t] > S[c])) c = t;
                // grow a run of unforced positions around c, nearer first, lower index on ties
                int64_t left = c, right = c, got = 1;
                int64_t nl = c - 1, nr = c + 1;
                while (nl >= lo && F.at(nl)) --nl;
                while (nr < hi && F.at(nr)) ++nr;
                while (got < take) {
                    const bool has_l = nl >= lo, has_r = nr < hi;
                    const bool go_left = has_l && (!has_r || (c - nl) <= (nr - c));
                    if (go_left) {
                        left = nl;
                        --nl;
                        while (nl >= lo && F.at(nl)) --nl;
                    } else {
                        right = nr;
                        ++nr;
                        while (nr < hi && F.at(nr)) ++nr;
                    }
                    ++got;
                }
                for (int64_t t = lo; t < hi; ++t)
                    if ((F.at(t) || (t >= left && t <= right)) && out < B) sd.idx[out++] = (int32_t)t;
            }
        }
    }
}

}  // namespace

cudaError_t launch_select(const SelectBatch& b, cudaStream_t st) {
    k_select<<<(unsigned)b.n, kSelThreads, 0, st>>>(b);
    return cudaGetLastError();
}

}  // namespace cbk
