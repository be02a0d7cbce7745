// Score kernels: CacheBack position scores (App. C.1, App. D.2).
//
//   pass 1  k_stats     per (sender, KV group s, 256-position chunk): row max and
//                       sum of exp of the logits of every (query token r, head h)
//   combine k_combine   per (sender, s): chunk partials -> one log2 offset per row
//   pass 2  k_accum     per (sender, s, 128-position chunk + 8-position halo):
//                       a/G = exp2(z - offset), b = sum over the group's heads,
//                       N_s = sum_r Pool(b_r)^p, bsum = sum_r b  ->  U_s, N_s, D_s
//   k_finalize          per (sender, 240-position tile, slice of the groups): fixed-order
//                       sums over s, Q = Pool(U), C = (N/D)^(1/(p-1)), S = Q * C^alpha
//
// Both logit passes use the bf16 tensor cores through mma.sync m16n8k16 with fp32
// accumulation.  Rows of one m16 tile are (8 query tokens) x (2 heads of the
// group), so every thread holds all G heads of one token and the head sum needs
// no shuffles.  The softmax is exact: pass 1 finds each row's max and
// normaliser over all T positions, pass 2 recomputes the logits and normalises.
#include <cfloat>
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "cb_internal.cuh"

namespace cbk {
namespace {

constexpr int kThreads = 256;
constexpr int kAccumPos = kAccumChunk + 2 * kHalo;   // 144 positions held per pass-2 block
constexpr int kBStride = kAccumPos + 8;              // row stride of the b tile in smem (floats)
constexpr int kSlab = 64;                            // query tokens per pass-2 slab (8 warps x 8)

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float lg2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// x^p for x >= 0 (p > 1): exact square for p = 2, exp2(p log2 x) otherwise.
__device__ __forceinline__ float powp(float x, float p, bool p_is_2) {
    if (p_is_2) return x * x;
    return x > 0.f ? ex2(p * lg2(x)) : 0.f;
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem));
}

__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;\n" ::: "memory");
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t r[4], const void* smem) {
    unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(s));
}

__device__ __forceinline__ void mma16816(float c[4], const uint32_t a[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Which sender a flat block index belongs to (senders are laid out back to back).
template <typename F>
__device__ __forceinline__ int find_sender(int n, int64_t blk, F begin_of) {
    int i = 0;
    while (i + 1 < n && begin_of(i + 1) <= blk) ++i;
    return i;
}

// Stage K rows [tbase, tbase + npos) of one (l, g) slice into smem as 16-byte
// chunks, chunk c of row n stored at column c ^ (n & 7) (conflict-free ldmatrix).
// Rows outside [0, T), and rows whose block-table entry is out of range (recorded in the
// error word), are zero.
template <int D>
__device__ __forceinline__ void stage_keys(uint4* ksm, const uint16_t* kbase, int64_t ks_p, const PageMap& pm,
                                           int64_t tbase, int npos, int64_t T, uint32_t* err) {
    constexpr int CH = D / 8;
    for (int e = threadIdx.x; e < npos * CH; e += kThreads) {
        const int n = e / CH, ch = e % CH;
        uint4* dst = ksm + n * CH + (ch ^ (n & 7));
        const int64_t t = tbase + n;
        const int64_t ro = (t >= 0 && t < T) ? row_offset(pm, ks_p, t) : -1;
        if (ro >= 0) {
            cp_async16(dst, kbase + ro + ch * 8);
        } else {
            *dst = make_uint4(0u, 0u, 0u, 0u);
            if (t >= 0 && t < T && ch == 0) atomicOr(err, kErrPageIndex);
        }
    }
    cp_async_wait_all();
    __syncthreads();
}

// A fragments of the warp's 8 query tokens x G heads (m16 tile tt holds heads 2tt, 2tt+1).
// Rows of absent tokens or heads are zero.
template <int D, int G>
__device__ __forceinline__ void load_query_frags(uint32_t (&af)[(G + 1) / 2][D / 16][4], const ScoreSender& sd,
                                                 int l, int g, int r) {
    const int qd = threadIdx.x & 3;
#pragma unroll
    for (int tt = 0; tt < (G + 1) / 2; ++tt)
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int j = 2 * tt + half;
            const bool ok = (r < sd.m) && (j < G);
            const uint16_t* row = sd.q + (int64_t)l * sd.qs_l + (int64_t)(ok ? r : 0) * sd.qs_t +
                                  (int64_t)(g * G + (ok ? j : 0)) * sd.qs_h;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
                uint32_t lo = 0u, hi = 0u;
                if (ok) {
                    lo = __ldg(reinterpret_cast<const uint32_t*>(row + 16 * ks + 2 * qd));
                    hi = __ldg(reinterpret_cast<const uint32_t*>(row + 16 * ks + 8 + 2 * qd));
                }
                af[tt][ks][half] = lo;
                af[tt][ks][2 + half] = hi;
            }
        }
}

// Logits of the warp's 32 rows against n8 block `nb` of the staged keys, accumulated into acc.
template <int D, int G>
__device__ __forceinline__ void logits_block(float (&acc)[(G + 1) / 2][4], const uint32_t (&af)[(G + 1) / 2][D / 16][4],
                                             const uint4* ksm, int nb) {
    constexpr int CH = D / 8;
    const int lane = threadIdx.x & 31;
    const int n = nb * 8 + (lane & 7);
    const int mi = lane >> 3;
#pragma unroll
    for (int kc = 0; kc < D / 32; ++kc) {
        uint32_t b[4];
        const int ch = 4 * kc + mi;
        ldmatrix_x4(b, ksm + n * CH + (ch ^ (n & 7)));
#pragma unroll
        for (int tt = 0; tt < (G + 1) / 2; ++tt) {
            mma16816(acc[tt], af[tt][2 * kc], b[0], b[1]);
            mma16816(acc[tt], af[tt][2 * kc + 1], b[2], b[3]);
        }
    }
}

__device__ __forceinline__ void online_merge(float& m, float& l, float mo, float lo) {
    const float mn = fmaxf(m, mo);
    if (mn == -INFINITY) return;
    const float a = (m == -INFINITY) ? 0.f : l * ex2(m - mn);
    const float b = (mo == -INFINITY) ? 0.f : lo * ex2(mo - mn);
    m = mn;
    l = a + b;
}

// ---------------------------------------------------------------------------
// pass 1: row statistics over one 256-position chunk
// ---------------------------------------------------------------------------
template <int D, int G>
__global__ void __launch_bounds__(kThreads, 2) k_stats(const __grid_constant__ ScoreBatch bt) {
    constexpr int GT = (G + 1) / 2;
    constexpr int NBS = 4;  // n8 blocks per online-softmax step
    extern __shared__ __align__(128) uint4 ksm[];
    const int64_t blk = blockIdx.x;
    const int i = find_sender(bt.n, blk, [&](int k) { return bt.s[k].blk1_begin; });
    const ScoreSender& sd = bt.s[i];
    const int64_t local = blk - sd.blk1_begin;
    const int s = (int)(local / sd.n_chunk1), c = (int)(local % sd.n_chunk1);
    const int l = s / bt.n_kv_heads, g = s % bt.n_kv_heads;
    const int64_t T = sd.T, t0 = (int64_t)c * kStatsChunk;
    stage_keys<D>(ksm, sd.k + (int64_t)l * sd.ks_l + (int64_t)g * sd.ks_h, sd.ks_p, sd.pm, t0, kStatsChunk, T,
                  bt.err);

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int qd = lane & 3, rr = lane >> 2;
    const int R = sd.m * G;
    const float sl2e = bt.scale_log2e;
    for (int tb = warp; tb * 8 < sd.m; tb += kThreads / 32) {
        const int r = tb * 8 + rr;
        uint32_t af[GT][D / 16][4];
        load_query_frags<D, G>(af, sd, l, g, r);
        float mrun[GT][2], lrun[GT][2];
#pragma unroll
        for (int tt = 0; tt < GT; ++tt)
#pragma unroll
            for (int h = 0; h < 2; ++h) { mrun[tt][h] = -INFINITY; lrun[tt][h] = 0.f; }
        for (int nb0 = 0; nb0 < kStatsChunk / 8; nb0 += NBS) {
            if (t0 + nb0 * 8 >= T) break;
            float acc[NBS][GT][4];
#pragma unroll
            for (int nb = 0; nb < NBS; ++nb)
#pragma unroll
                for (int tt = 0; tt < GT; ++tt)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[nb][tt][e] = 0.f;
#pragma unroll
            for (int nb = 0; nb < NBS; ++nb) logits_block<D, G>(acc[nb], af, ksm, nb0 + nb);
#pragma unroll
            for (int tt = 0; tt < GT; ++tt)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float v[NBS * 2];
                    float vmax = -INFINITY;
#pragma unroll
                    for (int nb = 0; nb < NBS; ++nb)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int64_t pos = t0 + (nb0 + nb) * 8 + 2 * qd + e;
                            float x = acc[nb][tt][2 * h + e] * sl2e;
                            x = pos < T ? x : -INFINITY;
                            v[nb * 2 + e] = x;
                            vmax = fmaxf(vmax, x);
                        }
                    const float mn = fmaxf(mrun[tt][h], vmax);
                    if (mn == -INFINITY) continue;
                    float sum = 0.f;
#pragma unroll
                    for (int k = 0; k < NBS * 2; ++k) sum += ex2(v[k] - mn);
                    lrun[tt][h] = lrun[tt][h] * ex2(mrun[tt][h] - mn) + sum;
                    mrun[tt][h] = mn;
                }
        }
#pragma unroll
        for (int tt = 0; tt < GT; ++tt)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
#pragma unroll
                for (int off = 1; off <= 2; off <<= 1) {
                    const float mo = __shfl_xor_sync(0xffffffffu, mrun[tt][h], off);
                    const float lo = __shfl_xor_sync(0xffffffffu, lrun[tt][h], off);
                    online_merge(mrun[tt][h], lrun[tt][h], mo, lo);
                }
                const int j = 2 * tt + h;
                if (qd == 0 && r < sd.m && j < G)
                    bt.stats[sd.stats_off + ((int64_t)s * sd.n_chunk1 + c) * R + r * G + j] =
                        make_float2(mrun[tt][h], lrun[tt][h]);
            }
    }
}

// ---------------------------------------------------------------------------
// combine: per-row log2 offset = max + log2(sum) + log2(G) over all chunks
// ---------------------------------------------------------------------------
// A row of one (sender, group s) merges its partial slots as four chains (slots j, j + 4, j + 8,
// ... for j = 0..3, each with an online max / sum in slot order), then the four chain results in
// chain order: a fixed order, so the offsets are deterministic and the same for both layouts.
// TPR = 1: one thread a row merges all four chains (many rows: the grid then fits in one wave);
// TPR = 4: four threads a row, one a chain, exchanging their results by shuffles (few rows with
// many slots each, e.g. long senders: four times the threads in flight).  A batch of slots is
// loaded before any is merged (the partials mostly come from DRAM).
constexpr int kCombThreads = 256;
constexpr int kCombBatch = 32;     // slots of a row loaded before they are merged
constexpr int kSelfChunk = 64;     // query self keys staged in shared memory at a time

// One logit x (log2 domain) into the running offset M and sum L.
__device__ __forceinline__ void merge_logit1(float x, float& M, float& L) {
    if (x > M) {
        L = (M == -INFINITY ? 0.f : L * ex2(M - x)) + 1.f;
        M = x;
    } else {
        L += ex2(x - M);
    }
}

// The query tokens' own keys of one block's group (l, g) join its rows' statistics: row (token
// r, head h) attends to keys 0..r, key u merged on chain u mod 4 in increasing u (NC = 4: the
// thread merges every chain; NC = 1: only chain c0l).  The block stages the keys in shared memory
// 64 at a time and each thread holds its query row in registers; the dot products add in the
// order of the per-row version.  Every thread of the block calls it (it synchronises the block);
// `act` selects the threads with a row.
template <int D, int NC>
__device__ __forceinline__ void self_keys_staged(const ScoreSender& sd, int l, int g, int r_tok, int c0l,
                                                 const uint16_t* qrow, float sl2e, bool act, float (&M)[NC],
                                                 float (&L)[NC], uint4* ks) {
    constexpr int P = D / 8;   // 16-byte pieces of a key
    uint32_t qw[D / 2];
#pragma unroll
    for (int p = 0; p < P; ++p) {
        const uint4 a = act ? *reinterpret_cast<const uint4*>(qrow + 8 * p) : make_uint4(0u, 0u, 0u, 0u);
        qw[4 * p] = a.x;
        qw[4 * p + 1] = a.y;
        qw[4 * p + 2] = a.z;
        qw[4 * p + 3] = a.w;
    }
    const uint16_t* kbase = sd.kself + (int64_t)l * sd.kss_l + (int64_t)g * sd.kss_h;
    for (int u0 = 0; u0 < sd.m; u0 += kSelfChunk) {
        const int nk = sd.m - u0 < kSelfChunk ? sd.m - u0 : kSelfChunk;
        __syncthreads();   // the previous chunk is no longer read
        for (int e = threadIdx.x; e < nk * P; e += blockDim.x)
            ks[e] = *reinterpret_cast<const uint4*>(kbase + (int64_t)(u0 + e / P) * sd.kss_t + 8 * (e % P));
        __syncthreads();
        const int uend = r_tok + 1 < u0 + nk ? r_tok + 1 : u0 + nk;
        if (!act) continue;
        for (int ub = u0; ub < uend; ub += 4) {
#pragma unroll
            for (int k = 0; k < NC; ++k) {
                const int u = ub + (NC == 1 ? c0l : k);
                if (u >= uend) break;
                const uint4* kr = ks + (u - u0) * P;
                float dot = 0.f;
#pragma unroll
                for (int p = 0; p < P; ++p) {
                    const uint4 b = kr[p];
                    const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        dot = fmaf(__uint_as_float(qw[4 * p + w] << 16), __uint_as_float(bw[w] << 16), dot);
                        dot = fmaf(__uint_as_float(qw[4 * p + w] & 0xFFFF0000u), __uint_as_float(bw[w] & 0xFFFF0000u),
                                   dot);
                    }
                }
                merge_logit1(dot * sl2e, M[k], L[k]);
            }
        }
    }
}

// SELF: some sender of the batch has query self keys (an instantiation of its own: the staged
// self keys and the query row in registers would halve the occupancy of the plain merge).
template <int TPR, bool SELF>
__global__ void __launch_bounds__(kCombThreads) k_combine(const __grid_constant__ ScoreBatch bt, int G) {
    __shared__ uint4 ks_sm[SELF ? kSelfChunk * 16 : 1];   // staged query self keys (d <= 128)
    constexpr int RPB = kCombThreads / TPR;   // rows per block
    constexpr int NC = 4 / TPR;               // chains a thread merges
    const int nS = bt.n_layers * bt.n_kv_heads;
    int i = 0;
    int64_t blk = blockIdx.x;
    // blocks are laid out sender by sender, nS * ceil(rows / RPB) of them per sender
    for (; i < bt.n; ++i) {
        const int R_i = bt.s[i].m * G;
        const int rows_i = bt.ext ? (int)rows_pad128(R_i) : R_i;
        const int64_t nb = (int64_t)nS * ((rows_i + RPB - 1) / RPB);
        if (blk < nb) break;
        blk -= nb;
    }
    if (i >= bt.n) return;
    const ScoreSender& sd = bt.s[i];
    const int R = sd.m * G;
    const int rows = bt.ext ? (int)rows_pad128(R) : R;
    const int nrb = (rows + RPB - 1) / RPB;
    const int s = (int)(blk / nrb);
    const int row = (int)(blk % nrb) * RPB + (int)threadIdx.x / TPR;
    const int c0l = TPR == 1 ? 0 : (int)threadIdx.x % TPR;   // the thread's first chain
    const bool in_rows = row < rows;   // (the four threads of a row together)
    const unsigned gmask = TPR == 1 ? 0u : 0xFu << ((threadIdx.x & 31) & ~3u);
    const int l = s / bt.n_kv_heads, g = s % bt.n_kv_heads;
    const int r_tok = row / G, hh = row - r_tok * G;
    const uint16_t* qrow = sd.q + (int64_t)l * sd.qs_l + (int64_t)r_tok * sd.qs_t + (int64_t)(g * G + hh) * sd.qs_h;
    // one logit (log2 domain) into the running offset M and sum L
    auto merge_logit = [](float x, float& M, float& L) {
        if (x > M) {
            L = (M == -INFINITY ? 0.f : L * ex2(M - x)) + 1.f;
            M = x;
        } else {
            L += ex2(x - M);
        }
    };
    // <q_row, k> in fp32 over the head dimension (bf16 inputs)
    auto dot_row = [&](const uint16_t* krow) {
        float dot = 0.f;
        for (int k = 0; k < bt.head_dim; k += 8) {
            const uint4 a = *reinterpret_cast<const uint4*>(qrow + k);
            const uint4 b = *reinterpret_cast<const uint4*>(krow + k);
            const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                dot = fmaf(__uint_as_float(aw[w] << 16), __uint_as_float(bw[w] << 16), dot);
                dot = fmaf(__uint_as_float(aw[w] & 0xFFFF0000u), __uint_as_float(bw[w] & 0xFFFF0000u), dot);
            }
        }
        return dot;
    };
    // the query tokens' own keys: row (token r, head h) also attends to query keys 0..r, key u
    // on chain u mod 4 (each chain in increasing u); logits in the statistics' log2 domain
    auto merge_self_keys = [&](float (&M)[NC], float (&L)[NC]) {
#pragma unroll
        for (int k = 0; k < NC; ++k)
            for (int u = c0l + k; u <= r_tok; u += 4)
                merge_logit(dot_row(sd.kself + (int64_t)l * sd.kss_l + (int64_t)u * sd.kss_t + (int64_t)g * sd.kss_h) *
                                bt.scale_log2e, M[k], L[k]);
    };
    float off = 0.f;
    float M[NC], L[NC];
#pragma unroll
    for (int k = 0; k < NC; ++k) { M[k] = -INFINITY; L[k] = 0.f; }
    if (row < R) {
        const float2* st = bt.stats + sd.stats_off + (int64_t)s * sd.n_chunk1 * R + row;
        for (int cb = 0; cb < sd.n_chunk1; cb += kCombBatch) {
            constexpr int NL = kCombBatch / TPR;   // this thread's slots of the batch
            float2 vv[NL];
#pragma unroll
            for (int q = 0; q < NL; ++q) {
                const int c = cb + (TPR == 1 ? q : 4 * q + c0l);   // chain c mod 4 (cb a multiple of 32)
                vv[q] = c < sd.n_chunk1 ? st[(int64_t)c * R] : make_float2(-INFINITY, 0.f);
            }
#pragma unroll
            for (int q = 0; q < NL; ++q) {
                const float2 v = vv[q];
                const int k = TPR == 1 ? (q & 3) : 0;
                if (v.x == -INFINITY) continue;
                if (v.x > M[k]) {
                    L[k] = (M[k] == -INFINITY ? 0.f : L[k] * ex2(M[k] - v.x)) + v.y;
                    M[k] = v.x;
                } else {
                    L[k] += v.y * ex2(v.x - M[k]);
                }
            }
        }
    }
    if (SELF && sd.kself) {   // the whole block (a block's rows belong to one group)
        if (bt.head_dim == 128)
            self_keys_staged<128, NC>(sd, l, g, r_tok, c0l, qrow, bt.scale_log2e, row < R, M, L, ks_sm);
        else
            self_keys_staged<64, NC>(sd, l, g, r_tok, c0l, qrow, bt.scale_log2e, row < R, M, L, ks_sm);
    }
    if (row < R) {
        // A chunk partial whose sum left fp32 range makes the row's sum infinite (pass 1 of the
        // tensor-memory path offsets each chunk by the maximum of its first 32 logits, so a logit
        // far larger later in the chunk overflows exp2).  Such rows, rare, are recomputed here
        // from Q and K directly: position t on chain t mod 4.
        bool bad = false;
#pragma unroll
        for (int k = 0; k < NC; ++k) bad = bad || !(L[k] <= FLT_MAX);
        if (TPR == 4) {
            bad = __shfl_xor_sync(gmask, (int)bad, 1) != 0 || bad;
            bad = __shfl_xor_sync(gmask, (int)bad, 2) != 0 || bad;
        }
        if (bad) {
#pragma unroll
            for (int k = 0; k < NC; ++k) { M[k] = -INFINITY; L[k] = 0.f; }
            const uint16_t* kbase = sd.k + (int64_t)l * sd.ks_l + (int64_t)g * sd.ks_h;
#pragma unroll
            for (int k = 0; k < NC; ++k)
                for (int64_t t = c0l + k; t < sd.T; t += 4) {
                    const int64_t ro = row_offset(sd.pm, sd.ks_p, t);
                    merge_logit(ro < 0 ? 0.f : dot_row(kbase + ro) * bt.scale_log2e, M[k], L[k]);   // a bad page reads as zeros
                }
            if (sd.kself) merge_self_keys(M, L);
        }
        // the four chains in chain order
        float Mc[4], Lc[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (TPR == 1) {
                Mc[k] = M[k];
                Lc[k] = L[k];
            } else {
                const int src = ((int)threadIdx.x & 31 & ~3) + k;
                Mc[k] = __shfl_sync(gmask, M[0], src);
                Lc[k] = __shfl_sync(gmask, L[0], src);
            }
        }
        float Mx = -INFINITY;
#pragma unroll
        for (int k = 0; k < 4; ++k) Mx = fmaxf(Mx, Mc[k]);
        float Lx = 0.f;
#pragma unroll
        for (int k = 0; k < 4; ++k)
            if (Mc[k] != -INFINITY) Lx += Lc[k] * ex2(Mc[k] - Mx);
        off = Mx + log2f(Lx) + log2f((float)G);
        if (c0l == 0) bt.offs[sd.offs_off + (int64_t)s * R + row] = off;
    }
    if (!in_rows || c0l != 0) return;
    if (bt.ext) {
        // the tcgen05 pass 2 adds -off / scale_log2e to the logit inside the contraction
        // (one more K-step against a column of ones): three bf16 terms carry it to ~24 bits
        uint32_t w0 = 0, w1 = 0;
        if (row < R) {
            const float x = -off / bt.scale_log2e;
            const __nv_bfloat16 hi = __float2bfloat16_rn(x);
            const float r1 = x - __bfloat162float(hi);
            const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
            const __nv_bfloat16 lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));
            w0 = (uint32_t)__bfloat16_as_ushort(hi) | ((uint32_t)__bfloat16_as_ushort(mid) << 16);
            w1 = (uint32_t)__bfloat16_as_ushort(lo);
        } else {
            w0 = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(-1e30f));   // exp2 of it is 0
        }
        uint4* dst = reinterpret_cast<uint4*>(bt.ext + sd.ext_off + ((int64_t)s * rows + row) * kExtCols);
        dst[0] = make_uint4(w0, w1, 0u, 0u);
        dst[1] = make_uint4(0u, 0u, 0u, 0u);
    }
}

// ---------------------------------------------------------------------------
// pass 2: normalised attention, head mean, Pool, per-group partial sums
// ---------------------------------------------------------------------------
template <int D, int G>
__global__ void __launch_bounds__(kThreads, 2) k_accum(const __grid_constant__ ScoreBatch bt) {
    constexpr int GT = (G + 1) / 2;
    constexpr int NB = kAccumPos / 8;   // 18 n8 blocks
    constexpr int NBS = 3;              // n8 blocks per step
    extern __shared__ __align__(128) uint4 smem_raw[];
    uint4* ksm = smem_raw;                                                      // [144][D/8]
    float* bsm = reinterpret_cast<float*>(smem_raw + kAccumPos * (D / 8));     // [64][kBStride]
    float* bsum = bsm + kSlab * kBStride;                                       // [144]
    float* nred = bsum + kAccumPos;                                             // [2][128]
    float* offs = nred + 2 * kAccumChunk;                                       // [m*G]

    const int nS = bt.n_layers * bt.n_kv_heads;
    const int64_t blk = blockIdx.x;
    const int i = find_sender(bt.n, blk, [&](int k) { return bt.s[k].blk2_begin; });
    const ScoreSender& sd = bt.s[i];
    const int64_t local = blk - sd.blk2_begin;
    const int s = (int)(local / sd.n_chunk2), c = (int)(local % sd.n_chunk2);
    const int l = s / bt.n_kv_heads, g = s % bt.n_kv_heads;
    const int64_t T = sd.T, t0 = (int64_t)c * kAccumChunk, tbase = t0 - kHalo;
    const int R = sd.m * G;
    for (int row = threadIdx.x; row < R; row += kThreads) offs[row] = bt.offs[sd.offs_off + (int64_t)s * R + row];
    for (int k = threadIdx.x; k < kAccumPos; k += kThreads) bsum[k] = 0.f;
    stage_keys<D>(ksm, sd.k + (int64_t)l * sd.ks_l + (int64_t)g * sd.ks_h, sd.ks_p, sd.pm, tbase, kAccumPos, T,
                  bt.err);

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int qd = lane & 3, rr = lane >> 2;
    const float sl2e = bt.scale_log2e;
    const bool p2 = (bt.p == 2.f);
    const int ph = bt.pool_half;
    const int pp = threadIdx.x & (kAccumChunk - 1), hf = threadIdx.x >> 7;  // pool-phase roles
    float nacc = 0.f;

    for (int slab = 0; slab * kSlab < sd.m; ++slab) {
        const int tb = slab * (kSlab / 8) + warp;
        const int r = tb * 8 + rr;
        float* brow = bsm + (warp * 8 + rr) * kBStride;
        if (tb * 8 < sd.m) {
            uint32_t af[GT][D / 16][4];
            load_query_frags<D, G>(af, sd, l, g, r);
            float off[GT][2];
#pragma unroll
            for (int tt = 0; tt < GT; ++tt)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int j = 2 * tt + h;
                    off[tt][h] = (r < sd.m && j < G) ? offs[r * G + j] : INFINITY;
                }
            for (int nb0 = 0; nb0 < NB; nb0 += NBS) {
                float acc[NBS][GT][4];
#pragma unroll
                for (int nb = 0; nb < NBS; ++nb)
#pragma unroll
                    for (int tt = 0; tt < GT; ++tt)
#pragma unroll
                        for (int e = 0; e < 4; ++e) acc[nb][tt][e] = 0.f;
#pragma unroll
                for (int nb = 0; nb < NBS; ++nb) logits_block<D, G>(acc[nb], af, ksm, nb0 + nb);
#pragma unroll
                for (int nb = 0; nb < NBS; ++nb) {
                    const int col = (nb0 + nb) * 8 + 2 * qd;
                    float bv[2];
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        float sum = 0.f;
#pragma unroll
                        for (int tt = 0; tt < GT; ++tt)
#pragma unroll
                            for (int h = 0; h < 2; ++h) sum += ex2(acc[nb][tt][2 * h + e] * sl2e - off[tt][h]);
                        const int64_t pos = tbase + col + e;
                        bv[e] = (pos >= 0 && pos < T) ? sum : 0.f;
                    }
                    *reinterpret_cast<float2*>(brow + col) = make_float2(bv[0], bv[1]);
                }
            }
        } else {
            for (int k = 2 * qd; k < kAccumPos; k += 8) *reinterpret_cast<float2*>(brow + k) = make_float2(0.f, 0.f);
        }
        __syncthreads();
        // N_s: sum over this slab's tokens of Pool(b_r)^p at the block's output positions
        {
            const int col = pp + kHalo;
            const int rend = min(kSlab, sd.m - slab * kSlab);
            for (int rl = hf * (kSlab / 2); rl < min(rend, (hf + 1) * (kSlab / 2)); ++rl) {
                const float* row = bsm + rl * kBStride + col;
                float mx = row[-ph];
                for (int u = -ph + 1; u <= ph; ++u) mx = fmaxf(mx, row[u]);
                nacc = bt.p_inf ? fmaxf(nacc, mx) : nacc + powp(mx, bt.p, p2);
            }
            for (int k = threadIdx.x; k < kAccumPos; k += kThreads) {
                float acc = 0.f;
                for (int rl = 0; rl < rend; ++rl) acc += bsm[rl * kBStride + k];
                bsum[k] += acc;
            }
        }
        __syncthreads();
    }
    nred[hf * kAccumChunk + pp] = nacc;
    __syncthreads();
    if (threadIdx.x < kAccumChunk) {
        const int64_t t = t0 + threadIdx.x;
        if (t < T) {
            const int col = threadIdx.x + kHalo;
            const float inv_m = 1.f / (float)sd.m;
            float mx = bsum[col - ph];
            for (int u = -ph + 1; u <= ph; ++u) mx = fmaxf(mx, bsum[col + u]);
            // p = infinity: the largest pooled token value and the pooled token mean itself
            const float Nv = bt.p_inf ? fmaxf(nred[threadIdx.x], nred[kAccumChunk + threadIdx.x])
                                      : (nred[threadIdx.x] + nred[kAccumChunk + threadIdx.x]) * inv_m;
            const float Dv = bt.p_inf ? mx * inv_m : powp(mx * inv_m, bt.p, p2);
            const float Uv = bsum[col] * inv_m / (float)bt.n_kv_heads;
            float* part = bt.part + sd.part_off;
            part[((int64_t)0 * nS + s) * T + t] = Uv;
            part[((int64_t)1 * nS + s) * T + t] = Nv;
            part[((int64_t)2 * nS + s) * T + t] = Dv;
        }
    }
}

// ---------------------------------------------------------------------------
// finalize: fixed-order sums over the groups, Pool(U), C, S -- one launch
// ---------------------------------------------------------------------------
// Block (64-position tile, sender); thread (slice k, quad q) sums slice k of the groups
// (s = k, k + 16, ... in increasing order) for the four consecutive positions of quad q:
// quads 2..17 are the tile (U, N and D), quads 0, 1 and 18, 19 the kHalo positions on each
// side (U only, for Pool).  A batch of groups' loads is issued before they are added (the partials
// mostly come from DRAM, so the kernel needs many bytes in flight), with one 16-byte load per
// quad where the sender's partial rows are 16-byte aligned.  The 16 slice sums of every
// position are then added in slice order in shared memory, U is pooled and C and S written.
// Each sum has a fixed order, so the scores are deterministic.
constexpr int kFinPos = 64;                          // output positions per block
constexpr int kFinQuads = kFinPos / 4 + kHalo / 2;   // 16 tile quads + 2 on each side
constexpr int kFinSpan = 4 * kFinQuads;              // positions whose U is summed
constexpr int kFinThreads = kFinSlices * kFinQuads;  // 320

// BATCH: groups of a slice loaded before they are added (9 for 288 groups; fewer groups, e.g. 64,
// take a smaller batch, whose smaller register footprint fits several blocks an SM)
template <int BATCH>
__global__ void __launch_bounds__(kFinThreads) k_finalize(const __grid_constant__ ScoreBatch bt) {
    constexpr int kFinBatch = BATCH;
    __shared__ float su[kFinSlices][kFinSpan];
    __shared__ float sn[kFinSlices][kFinPos];
    __shared__ float sdn[kFinSlices][kFinPos];
    __shared__ float us[kFinSpan];
    const ScoreSender& sd = bt.s[blockIdx.y];
    const int64_t T = sd.T;
    const int64_t t0 = (int64_t)blockIdx.x * kFinPos;
    if (t0 >= T) return;
    const int sl = threadIdx.x / kFinQuads, q = threadIdx.x % kFinQuads;
    const int nS = bt.n_layers * bt.n_kv_heads;
    const float* part = bt.part + sd.part_off;
    const int64_t rN = (int64_t)nS * T, rD = 2 * rN;    // first N and D rows
    const bool pinf = bt.p_inf;
    const bool full = q >= kHalo / 4 && q < kHalo / 4 + kFinPos / 4;   // a tile quad: N and D too
    const int64_t t = t0 - kHalo + 4 * q;
    float u[4] = {0.f, 0.f, 0.f, 0.f}, n[4] = {0.f, 0.f, 0.f, 0.f}, d[4] = {0.f, 0.f, 0.f, 0.f};
    auto add = [&](float (&acc)[4], const float4 v, bool mx) {
        if (mx) {
            acc[0] = fmaxf(acc[0], v.x); acc[1] = fmaxf(acc[1], v.y);
            acc[2] = fmaxf(acc[2], v.z); acc[3] = fmaxf(acc[3], v.w);
        } else {
            acc[0] += v.x; acc[1] += v.y; acc[2] += v.z; acc[3] += v.w;
        }
    };
    if ((T & 3) == 0 && (sd.part_off & 3) == 0) {
        // 16-byte aligned rows: the quad lies wholly inside or wholly outside [0, T)
        if (t >= 0 && t < T) {
            const float4* p = reinterpret_cast<const float4*>(part + t);
            const int64_t rs = T / 4;   // row stride in float4
            for (int s0 = sl; s0 < nS; s0 += kFinSlices * kFinBatch) {
                float4 a[kFinBatch], b[kFinBatch], c[kFinBatch];
#pragma unroll
                for (int k = 0; k < kFinBatch; ++k) {
                    const int s = s0 + k * kFinSlices;
                    if (s < nS) {
                        a[k] = __ldcs(p + (int64_t)s * rs);
                        if (full) {
                            b[k] = __ldcs(p + (rN / 4) + (int64_t)s * rs);
                            c[k] = __ldcs(p + (rD / 4) + (int64_t)s * rs);
                        }
                    }
                }
#pragma unroll
                for (int k = 0; k < kFinBatch; ++k) {
                    if (s0 + k * kFinSlices >= nS) break;
                    add(u, a[k], false);
                    if (full) {
                        add(n, b[k], pinf);   // p = infinity: N and D are maxima over the groups
                        add(d, c[k], pinf);
                    }
                }
            }
        }
    } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int64_t te = t + e;
            if (te < 0 || te >= T) continue;   // outside the sender: U = 0 adds nothing to Pool
            const float* p = part + te;
            for (int s = sl; s < nS; s += kFinSlices) {
                u[e] += __ldcs(p + (int64_t)s * T);
                if (!full) continue;
                const float b = __ldcs(p + rN + (int64_t)s * T), c = __ldcs(p + rD + (int64_t)s * T);
                n[e] = pinf ? fmaxf(n[e], b) : n[e] + b;
                d[e] = pinf ? fmaxf(d[e], c) : d[e] + c;
            }
        }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        su[sl][4 * q + e] = u[e];
        if (full) {
            sn[sl][4 * q - kHalo + e] = n[e];
            sdn[sl][4 * q - kHalo + e] = d[e];
        }
    }
    __syncthreads();
    const int x = threadIdx.x;
    if (x < kFinSpan) {
        float U = 0.f;
#pragma unroll
        for (int k = 0; k < kFinSlices; ++k) U += su[k][x];
        us[x] = U;
    }
    float Nv = 0.f, Dv = 0.f;
    if (x < kFinPos) {
#pragma unroll
        for (int k = 0; k < kFinSlices; ++k) {
            Nv = pinf ? fmaxf(Nv, sn[k][x]) : Nv + sn[k][x];
            Dv = pinf ? fmaxf(Dv, sdn[k][x]) : Dv + sdn[k][x];
        }
    }
    __syncthreads();
    if (x < kFinPos && t0 + x < T) {
        const int ph = bt.pool_half;
        const int c = x + kHalo;
        float Q = us[c - ph];
        for (int v = -ph + 1; v <= ph; ++v) Q = fmaxf(Q, us[c + v]);
        const float C = Dv > FLT_MIN ? (pinf ? Nv / Dv : powf(Nv / Dv, 1.f / (bt.p - 1.f))) : 1.f;
        sd.scores[t0 + x] = bt.alpha == 0.f ? Q : Q * powf(C, bt.alpha);
    }
}

}  // namespace

namespace {

cudaError_t launch_finalize(const ScoreBatch& b, cudaStream_t st) {
    int64_t maxT = 0;
    for (int i = 0; i < b.n; ++i) maxT = b.s[i].T > maxT ? b.s[i].T : maxT;
    dim3 grid((unsigned)((maxT + kFinPos - 1) / kFinPos), (unsigned)b.n);
    const int per_slice = (b.n_layers * b.n_kv_heads + kFinSlices - 1) / kFinSlices;
    if (per_slice <= 4)
        k_finalize<4><<<grid, kFinThreads, 0, st>>>(b);
    else
        k_finalize<9><<<grid, kFinThreads, 0, st>>>(b);
    return cudaGetLastError();
}

// Rows of all senders of a batch; few rows (long senders, few groups) take four threads a row.
int64_t combine_rows(const ScoreBatch& b) {
    const int G = b.n_q_heads / b.n_kv_heads;
    const int64_t nS = (int64_t)b.n_layers * b.n_kv_heads;
    int64_t rows = 0;
    for (int i = 0; i < b.n; ++i) {
        const int64_t R = (int64_t)b.s[i].m * G;
        rows += nS * (b.ext ? rows_pad128(R) : R);
    }
    return rows;
}

template <int TPR>
cudaError_t launch_combine_t(const ScoreBatch& b, cudaStream_t st) {
    bool self = false;
    for (int i = 0; i < b.n; ++i) self = self || b.s[i].kself != nullptr;
    const int G = b.n_q_heads / b.n_kv_heads;
    const int64_t nS = (int64_t)b.n_layers * b.n_kv_heads;
    constexpr int RPB = kCombThreads / TPR;
    int64_t nb = 0;
    for (int i = 0; i < b.n; ++i) {
        const int64_t R = (int64_t)b.s[i].m * G;
        const int64_t rows = b.ext ? rows_pad128(R) : R;
        nb += nS * ((rows + RPB - 1) / RPB);
    }
    if (self)
        k_combine<TPR, true><<<(unsigned)nb, kCombThreads, 0, st>>>(b, G);
    else
        k_combine<TPR, false><<<(unsigned)nb, kCombThreads, 0, st>>>(b, G);
    return cudaGetLastError();
}

cudaError_t launch_combine(const ScoreBatch& b, cudaStream_t st) {
    // four threads a row while that stays well within one wave of resident threads
    return combine_rows(b) <= 40000 ? launch_combine_t<4>(b, st) : launch_combine_t<1>(b, st);
}


template <int D, int G>
size_t accum_smem(int max_rows) {
    return (size_t)kAccumPos * D * 2 + (size_t)kSlab * kBStride * 4 + kAccumPos * 4 + 2 * kAccumChunk * 4 +
           (size_t)max_rows * 4;
}

template <int D, int G>
cudaError_t launch_dg(const ScoreBatch& b, cudaStream_t st) {
    int64_t nblk1 = 0, nblk2 = 0;
    int max_rows = 0;
    const int nS = b.n_layers * b.n_kv_heads;
    for (int i = 0; i < b.n; ++i) {
        nblk1 += (int64_t)nS * b.s[i].n_chunk1;
        nblk2 += (int64_t)nS * b.s[i].n_chunk2;
        max_rows = max_rows > b.s[i].m * G ? max_rows : b.s[i].m * G;
    }
    const size_t smem1 = (size_t)kStatsChunk * D * 2;
    const size_t smem2 = accum_smem<D, G>(max_rows);
    cudaError_t e = cudaFuncSetAttribute(k_stats<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_accum<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
    if (e != cudaSuccess) return e;
    stage_mark(b.timer, kStageStart, st);
    k_stats<D, G><<<(unsigned)nblk1, kThreads, smem1, st>>>(b);
    stage_mark(b.timer, kStageStats, st);
    launch_combine(b, st);
    stage_mark(b.timer, kStageCombine, st);
    k_accum<D, G><<<(unsigned)nblk2, kThreads, smem2, st>>>(b);
    stage_mark(b.timer, kStageAccum, st);
    launch_finalize(b, st);
    stage_mark(b.timer, kStageFinalize, st);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score_tc(ScoreBatch& b, cudaStream_t st, int num_sms, uint32_t* err,
                            cudaError_t (*combine)(const ScoreBatch&, cudaStream_t));

cudaError_t launch_score(const ScoreBatch& b_in, cudaStream_t st, int num_sms, int* path_out) {
    const int G = b_in.n_q_heads / b_in.n_kv_heads;
    const ScoreBatch& b = b_in;
    if (b.use_tc) {
        ScoreBatch* w = new ScoreBatch(b);
        cudaError_t e = launch_score_tc(*w, st, num_sms, b.err, launch_combine);
        if (e == cudaErrorNotSupported) {
            // the driver rejected a tensor map for these strides: use the mma.sync passes
            delete w;
            ScoreBatch* v = new ScoreBatch(b);
            v->use_tc = 0;
            e = launch_score(*v, st, num_sms, path_out);
            delete v;
            return e;
        }
        *path_out = 2;
        if (e == cudaSuccess) {
            launch_finalize(*w, st);
            stage_mark(w->timer, kStageFinalize, st);
            e = cudaGetLastError();
        }
        delete w;
        return e;
    }
    *path_out = 1;
    if (b.head_dim == 128) {
        if (G == 4) return launch_dg<128, 4>(b, st);
        if (G == 2) return launch_dg<128, 2>(b, st);
        if (G == 1) return launch_dg<128, 1>(b, st);
    } else if (b.head_dim == 64) {
        if (G == 4) return launch_dg<64, 4>(b, st);
        if (G == 2) return launch_dg<64, 2>(b, st);
        if (G == 1) return launch_dg<64, 1>(b, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace cbk
