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
#include <cstdio>
#include <cstring>
#include <mutex>
#include <cuda_runtime.h>

#include "cacheback.h"
#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kWarps = kSelThreads / 32;
constexpr int kScoreTile = 8192;                       // scores staged in shared memory per step
constexpr int kPadTile = kScoreTile + kScoreTile / 32;  // one pad word per 32 (span sums free of bank conflicts)
constexpr int kPerThread = kScoreTile / kSelThreads;    // scores each thread stages per tile
constexpr int kSmemSpans = 8192;     // span means kept in shared memory when there are at most this many
// two score tiles, the span means, and (one span a thread) each span's [left, right] run
constexpr size_t kSelDynSmem = (size_t)(2 * kPadTile + kSmemSpans + kSelThreads) * sizeof(float);
constexpr int kDirectPer = 4;        // width-16 spans a thread reads directly (up to 4096 spans)

__device__ __forceinline__ int pad(int k) { return k + (k >> 5); }

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
    __shared__ uint32_t hist[256];
    __shared__ int64_t scan_sh[32];
    __shared__ float red[32];
    __shared__ float head[kMaxSpanWidth];   // scores of the first span
    __shared__ int64_t sel_bucket, sel_before;
    __shared__ int64_t part_j;      // the span taken in part, when its run is found by a warp
    __shared__ int32_t part_take;

    // this block's sender in shared memory: reads of the parameter array at a run-time index
    // are slow, and with 64 registers a thread the compiler re-reads such values in loops
    __shared__ SelectSender sd;
    if (threadIdx.x == 0) {
        sd = bt.s[blockIdx.x];
        part_j = -1;
    }
    __syncthreads();
    const int64_t T = sd.T, B = sd.B;
    const int w = bt.span_w;
    const int64_t nsp = (T + w - 1) / w;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float* S = sd.scores;
    Forced F;
    F.a = bt.n_sink < T ? bt.n_sink : T;
    F.b = T - bt.n_latent > 0 ? T - bt.n_latent : 0;

    // 1. maximum score and span means.  Scores pass through shared memory a tile of whole spans
    // at a time (coalesced loads, two buffers: the next tile is loaded into registers while the
    // current one is summed); each thread sums its spans there, in index order.  The first span
    // (whose first score is replaced by the maximum) is summed last, once the maximum is known.
    extern __shared__ float dsm[];
    float* keys = nsp <= kSmemSpans ? dsm + 2 * kPadTile : sd.span_keys;
    const bool sink = bt.n_sink > 0;
    const int64_t tile = (int64_t)(kScoreTile / w) * w;     // whole spans per tile
    const int64_t ntile = (T + tile - 1) / tile;
    // width-16 spans, up to four a thread (spans tid, tid + 1024, ...): each thread reads its
    // spans' scores with four 16-byte loads each (scores are 16-byte aligned) and sums them in
    // index order, with no staging
    const bool direct = w == 16 && nsp <= (int64_t)kDirectPer * kSelThreads;
    float mx = -INFINITY;
#pragma unroll
    for (int q8 = 0; q8 < kDirectPer; ++q8) {
        const int64_t js = tid + (int64_t)q8 * kSelThreads;
        if (!direct || js >= nsp) break;
        const int64_t lo = js * 16;
        const int n = (int)(T - lo < 16 ? T - lo : 16);
        float v[16];
        if (n == 16) {
            const float4* p = reinterpret_cast<const float4*>(S + lo);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 x = p[q];
                v[4 * q] = x.x;
                v[4 * q + 1] = x.y;
                v[4 * q + 2] = x.z;
                v[4 * q + 3] = x.w;
            }
        } else {
#pragma unroll
            for (int k = 0; k < 16; ++k) v[k] = k < n ? S[lo + k] : 0.f;
        }
        float acc = 0.f;
#pragma unroll
        for (int k = 0; k < 16; ++k)
            if (k < n) {
                mx = fmaxf(mx, v[k]);
                acc += v[k];
                if (js == 0) head[k] = v[k];
            }
        if (!(js == 0 && sink)) keys[js] = __fdiv_rn(acc, (float)n);
    }
    float nxt[kPerThread];
#pragma unroll
    for (int q = 0; q < kPerThread; ++q) {
        const int k = tid + q * kSelThreads;
        nxt[q] = !direct && k < tile && k < T ? S[k] : 0.f;
    }
    for (int64_t it = 0; it < (direct ? 0 : ntile); ++it) {
        const int64_t t0 = it * tile, n = T - t0 < tile ? T - t0 : tile;
        float* ts = dsm + (it & 1) * kPadTile;
#pragma unroll
        for (int q = 0; q < kPerThread; ++q) {
            const int k = tid + q * kSelThreads;
            if (k < n) {
                ts[pad(k)] = nxt[q];
                mx = fmaxf(mx, nxt[q]);
                if (it == 0 && k < w) head[k] = nxt[q];
            }
        }
        __syncthreads();   // this tile is in place; the tile before the previous one is summed
        if (it + 1 < ntile) {
            const int64_t t1 = t0 + tile, n1 = T - t1 < tile ? T - t1 : tile;
#pragma unroll
            for (int q = 0; q < kPerThread; ++q) {
                const int k = tid + q * kSelThreads;
                nxt[q] = k < n1 ? S[t1 + k] : 0.f;
            }
        }
        const int64_t ja = t0 / w, jb = (t0 + n + w - 1) / w;
        for (int64_t j = ja + tid; j < jb; j += kSelThreads) {
            if (j == 0 && sink) continue;
            const int lo = (int)(j * w - t0), hi = (int)((j * w + w < T ? j * w + w : T) - t0);
            float acc = 0.f;
            for (int k = lo; k < hi; ++k) acc += ts[pad(k)];
            keys[j] = __fdiv_rn(acc, (float)(hi - lo));
        }
    }
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
    if (sink && tid == 0) {
        const int hi = w < T ? w : (int)T;
        float acc = 0.f;
        for (int k = 0; k < hi; ++k) acc += k == 0 ? smax : head[k];
        keys[0] = __fdiv_rn(acc, (float)hi);
    }
    // a single tile still holds every score (the partial span's best position is looked up there)
    const float* all_s = ntile == 1 && !direct ? dsm : nullptr;
    const int64_t need = B - F.count(0, T);
    __syncthreads();

    // 2. weighted radix select of the threshold key
    uint32_t my_key[kDirectPer], my_u[kDirectPer];   // direct: the thread's spans' keys and unforced positions
#pragma unroll
    for (int q8 = 0; q8 < kDirectPer; ++q8) {
        const int64_t js = tid + (int64_t)q8 * kSelThreads;
        my_key[q8] = 0u;
        my_u[q8] = 0u;
        if (direct && js < nsp) {
            const int64_t lo = js * w, hi = lo + w < T ? lo + w : T;
            my_key[q8] = order_key(keys[js]);
            my_u[q8] = (uint32_t)((hi - lo) - F.count(lo, hi));
        }
    }
    uint32_t prefix = 0u, pmask = 0u;
    int64_t rem = need;
    if (need > 0) {
        for (int pass = 0; pass < 4; ++pass) {
            const int shift = 24 - 8 * pass;
            if (tid < 256) hist[tid] = 0u;
            __syncthreads();
            if (direct) {
                // the thread's spans: their keys and unforced counts were found once, before the passes
#pragma unroll
                for (int q8 = 0; q8 < kDirectPer; ++q8)
                    if (my_u[q8] && (my_key[q8] & pmask) == prefix)
                        atomicAdd(&hist[(my_key[q8] >> shift) & 255u], my_u[q8]);
            } else {
                for (int64_t j = tid; j < nsp; j += kSelThreads) {
                    const uint32_t key = order_key(keys[j]);
                    if ((key & pmask) != prefix) continue;
                    const int64_t lo = j * w, hi = lo + w < T ? lo + w : T;
                    const uint32_t u = (uint32_t)((hi - lo) - F.count(lo, hi));
                    if (u) atomicAdd(&hist[(key >> shift) & 255u], u);
                }
            }
            __syncthreads();
            if (warp == 0) {
                // lane L owns buckets 255-8L .. 248-8L (descending key order)
                int64_t mine = 0;
#pragma unroll
                for (int k = 0; k < 8; ++k) mine += hist[255 - 8 * lane - k];
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
                        if (before + hist[bucket] >= rem) { sel_bucket = bucket; sel_before = before; break; }
                        before += hist[bucket];
                    }
                }
            }
            __syncthreads();
            prefix |= (uint32_t)sel_bucket << shift;
            pmask |= 255u << shift;
            rem -= sel_before;
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
            if (order_key(keys[j]) == kappa) {
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
                const uint32_t key = order_key(keys[j]);
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

    // 4. write positions in source order.  Each thread settles what its spans contribute:
    // everything, only the forced positions, or the forced ones plus the run [left, right]
    // around the partial span's best position.  With one span a thread, or when the scores were
    // read directly (the staging buffers then hold the runs), a span's output start (in place of
    // its mean, which is no longer needed) and its run go to shared memory and each warp then
    // writes whole spans, 32 consecutive positions per step, so the stores are coalesced;
    // otherwise every thread writes its own spans.
    const bool coop = nsp <= kSelThreads || direct;
    int32_t* span_at = reinterpret_cast<int32_t*>(keys);
    int32_t* span_run = reinterpret_cast<int32_t*>(direct ? dsm : dsm + 2 * kPadTile + kSmemSpans);
    {
        int64_t tb = tie_before;
        for (int64_t j = j0; j < j1; ++j) {
            const int64_t lo = j * w, hi = lo + w < T ? lo + w : T;
            const int64_t f = F.count(lo, hi), u = (hi - lo) - f;
            int64_t take = 0;
            if (need > 0) {
                const uint32_t key = order_key(keys[j]);
                if (key > kappa) take = u;
                else if (key == kappa) {
                    take = rem - tb;
                    take = take < 0 ? 0 : (take > u ? u : take);
                    tb += u;
                }
            }
            int64_t left = lo, right = lo - 1;   // empty run: only the forced positions
            if (take == u) {
                left = lo;
                right = hi - 1;
            } else if (take > 0 && coop && w <= 32) {
                part_j = j;                // its run is found by a warp below (at most one such span)
                part_take = (int32_t)take;
            } else if (take > 0) {
                // highest-scoring unforced position (lowest index on ties)
                int64_t c = -1;
                float best = 0.f;
                for (int64_t t = lo; t < hi; ++t)
                    if (!F.at(t)) {
                        const float v = all_s ? all_s[pad((int)t)] : S[t];
                        if (c < 0 || v > best) {
                            c = t;
                            best = v;
                        }
                    }
                // grow a run of unforced positions around c, nearer first, lower index on ties
                int64_t got = 1, nl = c - 1, nr = c + 1;
                left = right = c;
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
            }
            if (coop) {
                span_at[j] = (int32_t)out;   // B < 2^31
                span_run[j] = (int32_t)((left - lo + 1) | ((right - lo + 1) << 16));
            } else {
                for (int64_t t = lo; t < hi; ++t)
                    if ((F.at(t) || (t >= left && t <= right)) && out < B) sd.idx[out] = (int32_t)t, ++out;
                continue;
            }
            out += f + take;
        }
    }
    if (coop) {
        __syncthreads();
        if (part_j >= 0 && warp == 0) {
            // the partial span's take unforced positions nearest its highest-scoring unforced one
            // (lowest index on ties), distance ties to the lower index: ranked by (distance, index)
            const int64_t j = part_j, lo = j * w, hi = lo + w < T ? lo + w : T;
            const int64_t t = lo + lane;
            const bool unf = t < hi && !F.at(t);
            const float v = unf ? S[t] : -INFINITY;
            float vm = v;
#pragma unroll
            for (int o = 16; o; o >>= 1) vm = fmaxf(vm, __shfl_xor_sync(0xffffffffu, vm, o));
            const int cl = __ffs(__ballot_sync(0xffffffffu, unf && v == vm)) - 1;
            const int d = unf ? abs(lane - cl) : (1 << 20);
            int rank = 0;
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                const int dk = __shfl_sync(0xffffffffu, d, k);
                rank += (dk < d || (dk == d && k < lane)) ? 1 : 0;
            }
            const unsigned sel = __ballot_sync(0xffffffffu, unf && rank < part_take);
            if (lane == 0) span_run[j] = (int32_t)((__ffs(sel)) | ((32 - __clz(sel)) << 16));
        }
        __syncthreads();
        // 32-bit arithmetic throughout (T < 2^31): this loop is bound by instruction issue
        const int32_t T32 = (int32_t)T, B32 = (int32_t)(B < T ? B : T), fa = (int32_t)F.a, fb = (int32_t)F.b;
        const int32_t nsp32 = (int32_t)nsp;
        const unsigned below = (1u << lane) - 1u;
        int32_t* const idx = sd.idx;
        // each warp takes 32 spans at a time: one lane a span finds whether anything of it is
        // kept, and the warp then writes only those spans
        for (int32_t jb = warp * 32; jb < nsp32; jb += kWarps * 32) {
            const int32_t jl = jb + lane;
            int32_t run = 0;
            bool kept = false;
            if (jl < nsp32) {
                const int32_t lo = jl * w, hi = lo + w < T32 ? lo + w : T32;
                run = span_run[jl];
                const int32_t left = lo + (run & 0xffff) - 1, right = lo + (run >> 16) - 1;
                kept = !(right < left && lo >= fa && hi <= fb);
            }
            unsigned km = __ballot_sync(0xffffffffu, kept);
            while (km) {
                const int src = __ffs(km) - 1;
                km &= km - 1;
                const int32_t j = jb + src;
                const int32_t rj = __shfl_sync(0xffffffffu, run, src);
                const int32_t lo = j * w, hi = lo + w < T32 ? lo + w : T32;
                const int32_t left = lo + (rj & 0xffff) - 1, right = lo + (rj >> 16) - 1;
                int32_t base = span_at[j];
                for (int32_t c0 = lo; c0 < hi; c0 += 32) {
                    const int32_t t = c0 + lane;
                    const bool sel = t < hi && (t < fa || t >= fb || (t >= left && t <= right));
                    const unsigned m = __ballot_sync(0xffffffffu, sel);
                    const int32_t o = base + __popc(m & below);
                    if (sel && o < B32) idx[o] = t;
                    base += __popc(m);
                }
            }
        }
    }
}

}  // namespace

cudaError_t launch_select(const SelectBatch& b, cudaStream_t st) {
    // per device (the attribute belongs to the current device's copy of the kernel)
    const cudaError_t attr =
        cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSelDynSmem);
    if (attr != cudaSuccess) return attr;
    k_select<<<(unsigned)b.n, kSelThreads, kSelDynSmem, st>>>(b);
    return cudaGetLastError();
}

}  // namespace cbk

// ---------------------------------------------------------------------------
// Allocation-free selection.
//
// Some callers cannot allocate device memory at all: code that runs inside a
// memory pool or arena it does not own, a host that forbids cudaMalloc after
// start-up, or an engine whose allocator is busy or not reentrant at the point
// of the call.  cb_select_noalloc serves them: it runs the same selection kernel
// as cb_select, needs no context, and keeps its scratch (the span means and a
// status word) in a fixed array compiled into this library instead of calling
// cudaMalloc.  Every GPU that loads the library holds that array until the
// process exits.
// ---------------------------------------------------------------------------
namespace cbk {
namespace {

constexpr int64_t kNoAllocMaxSpans = 65536;   // span means per call: 256 KiB of floats

static __device__ __align__(256) float g_noalloc_scratch[kNoAllocMaxSpans + 64];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
float* g_noalloc_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up once
// per device, with that device current, and cached.
cb_status noalloc_scratch(int dev, float** out, char* msg, size_t len) {
    if (dev < 0 || dev >= kMaxDevices) {
        snprintf(msg, len, "device ordinal %d not supported", dev);
        return CB_EINVAL;
    }
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) {
            cudaGetLastError();
            snprintf(msg, len, "cannot resolve the scratch array on device %d: %s", dev, cudaGetErrorString(e));
            return CB_ECUDA;
        }
        g_noalloc_addr[dev] = static_cast<float*>(p);
    }
    *out = g_noalloc_addr[dev];
    return CB_OK;
}

cb_status noalloc_check_ptr(const void* p, int dev, const char* what, int i, char* msg, size_t len) {
    if (!p || (reinterpret_cast<uintptr_t>(p) & 15u)) {
        snprintf(msg, len, "%s[%d] is NULL or not 16-byte aligned", what, i);
        return CB_EINVAL;
    }
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        snprintf(msg, len, "%s[%d]: cannot query pointer", what, i);
        return CB_EINVAL;
    }
    if (a.type == cudaMemoryTypeManaged) return CB_OK;
    if (a.type != cudaMemoryTypeDevice || a.device != dev) {
        snprintf(msg, len, "%s[%d] is not device memory of device %d", what, i, dev);
        return CB_EINVAL;
    }
    return CB_OK;
}

}  // namespace
}  // namespace cbk

extern "C" cb_status cb_select_noalloc(int32_t n, const float* const* scores, const int64_t* T,
                                       const int64_t* budget, int32_t* const* idx, int32_t n_sink,
                                       int32_t n_latent, int32_t span_width, void* stream) {
    using namespace cbk;
    char msg[256] = "";
    cb_status st = CB_OK;
    int dev = 0;
    float* scratch = nullptr;
    set_context_free_error("");
    if (n < 1 || n > 4096) {
        snprintf(msg, sizeof msg, "n = %d not in [1, 4096]", n);
        st = CB_ESHAPE;
    } else if (!scores || !T || !budget || !idx) {
        snprintf(msg, sizeof msg, "scores, T, budget or idx is NULL");
        st = CB_EINVAL;
    } else if (span_width < 1 || span_width > kMaxSpanWidth || n_sink < 0 || n_latent < 0) {
        snprintf(msg, sizeof msg, "span_width must be in [1, %d]; n_sink, n_latent >= 0", kMaxSpanWidth);
        st = CB_EINVAL;
    } else if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        snprintf(msg, sizeof msg, "no CUDA device");
        st = CB_ECUDA;
    }
    // Only senders with more than kSmemSpans spans keep their span means in the array (the
    // kernel holds fewer in shared memory); each launch of up to kMaxBatch senders places its
    // own such senders from slot 0, so the largest launch decides what the call needs.
    int64_t group_slots = 0, max_slots = 0;
    for (int i = 0; st == CB_OK && i < n; ++i) {
        if (T[i] < 1 || T[i] > INT32_MAX) {
            snprintf(msg, sizeof msg, "T[%d] = %lld not in [1, 2^31)", i, (long long)T[i]);
            st = CB_ESHAPE;
            break;
        }
        const int64_t a = n_sink < T[i] ? n_sink : T[i];
        const int64_t b = T[i] - n_latent > 0 ? T[i] - n_latent : 0;
        const int64_t forced = a >= b ? T[i] : a + (T[i] - b);
        if (budget[i] < forced || budget[i] > T[i]) {
            snprintf(msg, sizeof msg, "budget[%d] = %lld outside [%lld, %lld]", i, (long long)budget[i],
                     (long long)forced, (long long)T[i]);
            st = CB_EBUDGET;
            break;
        }
        if (i % kMaxBatch == 0) group_slots = 0;
        const int64_t nsp = (T[i] + span_width - 1) / span_width;
        if (nsp > kSmemSpans) group_slots += nsp;
        max_slots = group_slots > max_slots ? group_slots : max_slots;
        if ((st = noalloc_check_ptr(scores[i], dev, "scores", i, msg, sizeof msg))) break;
        if ((st = noalloc_check_ptr(idx[i], dev, "idx", i, msg, sizeof msg))) break;
    }
    if (st == CB_OK && max_slots > kNoAllocMaxSpans) {
        snprintf(msg, sizeof msg, "one launch of the call needs %lld span slots for senders of more than %d "
                 "spans; this entry point holds at most %lld (use cb_select with a context for larger calls)",
                 (long long)max_slots, kSmemSpans, (long long)kNoAllocMaxSpans);
        st = CB_ESHAPE;
    }
    if (st == CB_OK) st = noalloc_scratch(dev, &scratch, msg, sizeof msg);
    if (st != CB_OK) {
        set_context_free_error(msg);
        return st;
    }
    cudaStream_t strm = reinterpret_cast<cudaStream_t>(stream);
    uint32_t* status_word = reinterpret_cast<uint32_t*>(scratch + kNoAllocMaxSpans);
    // the array keeps the previous call's contents: the status word must start at zero
    cudaError_t e = cudaMemsetAsync(status_word, 0, sizeof(uint32_t), strm);
    for (int b0 = 0; e == cudaSuccess && b0 < n; b0 += kMaxBatch) {
        const int nb = n - b0 < kMaxBatch ? n - b0 : kMaxBatch;
        SelectBatch bt;
        memset(&bt, 0, sizeof bt);
        bt.n = nb;
        bt.n_sink = n_sink;
        bt.n_latent = n_latent;
        bt.span_w = span_width;
        bt.err = status_word;
        int64_t off = 0;
        for (int k = 0; k < nb; ++k) {
            const int64_t nsp = (T[b0 + k] + span_width - 1) / span_width;
            bt.s[k].scores = scores[b0 + k];
            bt.s[k].idx = idx[b0 + k];
            bt.s[k].T = T[b0 + k];
            bt.s[k].B = budget[b0 + k];
            bt.s[k].span_keys = nsp > kSmemSpans ? scratch + off : nullptr;   // else unused by the kernel
            if (nsp > kSmemSpans) off += nsp;
        }
        e = launch_select(bt, strm);
    }
    if (e != cudaSuccess) {
        snprintf(msg, sizeof msg, "select launch failed: %s", cudaGetErrorString(e));
        set_context_free_error(msg);
        return CB_ECUDA;
    }
    return CB_OK;
}

extern "C" cb_status cb_select_noalloc_status(void* stream) {
    using namespace cbk;
    char msg[256] = "";
    set_context_free_error("");
    int dev = 0;
    float* scratch = nullptr;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        set_context_free_error("no CUDA device");
        return CB_ECUDA;
    }
    cb_status st = noalloc_scratch(dev, &scratch, msg, sizeof msg);
    if (st != CB_OK) {
        set_context_free_error(msg);
        return st;
    }
    cudaStream_t strm = reinterpret_cast<cudaStream_t>(stream);
    uint32_t* status_word = reinterpret_cast<uint32_t*>(scratch + kNoAllocMaxSpans);
    uint32_t word = 0;
    cudaError_t e = cudaMemcpyAsync(&word, status_word, sizeof word, cudaMemcpyDeviceToHost, strm);
    if (e == cudaSuccess) e = cudaStreamSynchronize(strm);
    if (e == cudaSuccess && word) {
        e = cudaMemsetAsync(status_word, 0, sizeof(uint32_t), strm);
        if (e == cudaSuccess) e = cudaStreamSynchronize(strm);
    }
    if (e != cudaSuccess) {
        snprintf(msg, sizeof msg, "device error: %s", cudaGetErrorString(e));
        set_context_free_error(msg);
        return CB_ECUDA;
    }
    if (word) {
        snprintf(msg, sizeof msg, "the selection kernel's own check failed (code 0x%x:%s)", word,
                 (word & kErrSelectBudget) ? " selected count differs from the budget" : "");
        set_context_free_error(msg);
        return CB_EDEVICE;
    }
    return CB_OK;
}
