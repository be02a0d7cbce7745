// Score passes on the 5th-generation tensor cores (tcgen05 + TMEM + TMA), sm_103a.
//
// Both passes contract the receiver query Q_s = [(r, h) rows x d] of one KV group
// s = (l, g) with that group's keys K_s = [positions x d] (App. C.1: a_{l,h,r,t} is the
// softmax over t of scale * <q, k>).  Operands are K-major bf16 tiles in the 128-byte
// swizzled layout, staged by TMA; one thread issues tcgen05.mma (fp32 accumulation in TMEM);
// the epilogue warps read TMEM with tcgen05.ld.  A paged sender cache is first copied into a
// contiguous staging buffer by k_depage (TMA needs a fixed tile shape, which a page boundary
// inside a tile breaks), and both passes read that copy.
//
//   k_stats_tc  pass 1, D = Q_s K_tile^T: TMEM lane = row (r, h), column = position.
//               Each epilogue thread owns one row and keeps its running max and
//               sum of exp2 over its group's tiles of a 1024-position chunk.
//   k_accum_tc  pass 2, D = K_tile Q_s^T (+ a ninth K-step of ones x the rows' offset terms,
//               so TMEM holds z - offset / scale): TMEM lane = position, column = row (r, h).
//               Each thread owns one position: exp2 of its logits (a / G), the head mean b
//               and the sums over tokens stay in registers; Pool over positions runs
//               across lanes with shuffles.  A tile's four 32-row quarters start 3 positions
//               before their 26 output positions (104 per tile).
//
// Warp roles (576 threads, one CTA per SM, persistent over a contiguous range of work
// units): warp 0 producer, warp 1 MMA issuer and TMEM owner, warps 2-17 epilogue (two
// groups of eight taking alternate tiles; warp w reads TMEM lanes 32*(w%4)..+31).  K tiles
// flow through a ring of smem stages; TMEM holds four 128-column accumulator buffers.
// Every mbarrier wait is bounded (1 s); on a timeout the kernel records kErrTimeout, drains
// its copies and MMAs, frees TMEM and returns.
#include <cfloat>
#include <cstdint>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <mutex>
#include <vector>

#include "cb_internal.cuh"
#include "cb_sm100.cuh"

namespace cbk {
namespace {
using namespace sm100;

constexpr int kWarpsTc = 18;                // 0 TMA, 1 MMA, 2..17 epilogue
constexpr int kThreadsTc = kWarpsTc * 32;
constexpr int kMaxStages = 4;
constexpr int kTileRows = 128;          // K rows per tile
constexpr int kTileBytes = kTileRows * 256;   // d = 128: two 64-column swizzled blocks
constexpr int kChunk1 = kStatsChunkTc;  // pass-1 positions per chunk
constexpr int kMargin = 3;              // pass-2 lanes before/after the output positions
constexpr int kOutW = 32 - 2 * kMargin;          // 26 output positions per pass-2 warp
constexpr int kOut2 = 4 * kOutW;                 // 104 output positions per pass-2 tile
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitNs = 1000000000ull;      // 1 s per wait
constexpr uint32_t kPollNs = 1000000u;           // longest suspension of one poll (woken at completion)
constexpr int kMaxTcSenders = 32;

struct TcSender {
    CUtensorMap kmap;     // 4D {d, T, Hkv, nL}, box {64, 128, 1, 1}
    CUtensorMap kmap32;   // same tensor, box {64, 32, 1, 1}
    CUtensorMap qmap;     // 4D {d, Hq, m, nL}, box {64, G, qbox_tok, 1}
    CUtensorMap emap;     // 3D {16, R_pad, nS} offset terms of pass 2, box {16, ebox_rows, 1}, 32-byte swizzle
    float2* stats;        // this sender's pass-1 partials [nS][n_chunk1][R]
    const float* offs;    // this sender's per-row offsets [nS][R]
    float* part;          // this sender's partials [3][nS][T]
    int64_t T;
    int32_t m, R, R_pad;
    int32_t n_chunk1, n_tile2;
    int32_t qbox_tok, n_qbox;
    int32_t ebox_rows, n_ebox;
    float inv_m, inv_mh;  // 1 / m and 1 / (m Hkv)
    int64_t unit1_begin, unit2_begin;
};

struct TcBatch {
    CUtensorMap omap;     // 2D {16, 128} block of ones columns, one box, 32-byte swizzle
    int32_t n;
    int32_t nL, Hq, Hkv, G;
    int32_t stages, rpad_max;
    float sl2e, p;
    int32_t p_is_2, p_inf, ph;
    int64_t units1, units2;
    uint64_t wait_ns;     // limit of one bounded mbarrier wait
    int32_t stall;        // 1: CTA 0's pass-1 MMA issuer first waits on a barrier nothing arrives on
    uint32_t* err;
    TcSender s[kMaxTcSenders];
};

struct Ctl {
    uint64_t k_full[kMaxStages], k_empty[kMaxStages];
    uint64_t t_full[4], t_empty[4];   // TMEM buffers of 128 columns (pass 1: group g owns 2g and 2g + 1;
                                      // pass 2: buffer 2g + h is column half h of group g)
    uint64_t q_full, q_empty, drain, o_full;
    uint64_t stall;         // failure-detection test: a barrier nothing arrives on
    uint64_t wait_ns;       // limit of one bounded wait
    uint64_t xb[2][2][4];   // pass 2: column-half exchange [tile parity][group][lane quarter]: written
    uint64_t xe[2][2][4];   //   and read (half 1 reuses a slot only after half 0 has read it)
    uint32_t tmem_base;
    int abort;
};
static_assert(sizeof(Ctl) <= 512, "the epilogue exchange area starts 512 bytes after Ctl");

__device__ __forceinline__ uint64_t now_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait: true when the phase completed, false on abort (set by anyone) or timeout.
// `tag` names the wait in the device error word (bit 8 + tag) when it times out.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, Ctl* ctl, uint32_t* err, int tag) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = now_ns();
    for (uint32_t i = 1; i < (1u << 30); ++i) {
        if (mbar_try_wait_hint(bar, parity, kPollNs)) return true;
        if ((i & 63) == 0) {
            if (*reinterpret_cast<volatile int*>(&ctl->abort)) return false;
            if (now_ns() - t0 > ctl->wait_ns) {
                *reinterpret_cast<volatile int*>(&ctl->abort) = 1;
                atomicOr(err, kErrTimeout | (1u << (8 + tag)));
                return false;
            }
        }
    }
    *reinterpret_cast<volatile int*>(&ctl->abort) = 1;
    atomicOr(err, kErrTimeout);
    return false;
}

// Wait used only on the way out (drain): bounded by kWaitNs whatever the configured limit
// (the copies and MMAs it waits for always complete), ignores the abort flag.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
    const uint64_t t0 = now_ns();
    while (!mbar_try_wait(bar, parity))
        if (now_ns() - t0 > kWaitNs) return;
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
    return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

struct Unit {
    int i, s, c;   // sender, group, chunk (pass 1) or tile (pass 2)
};

__device__ __forceinline__ Unit decode1(const TcBatch& bt, int64_t u) {
    int i = 0;
    while (i + 1 < bt.n && bt.s[i + 1].unit1_begin <= u) ++i;
    const int64_t local = u - bt.s[i].unit1_begin;
    const int nch = bt.s[i].n_chunk1 / 4;   // n_chunk1 counts (chunk, group, half) partial slots
    return Unit{i, (int)(local / nch), (int)(local % nch)};
}

__device__ __forceinline__ Unit decode2(const TcBatch& bt, int64_t u) {
    int i = 0;
    while (i + 1 < bt.n && bt.s[i + 1].unit2_begin <= u) ++i;
    const int64_t local = u - bt.s[i].unit2_begin;
    return Unit{i, (int)(local / bt.s[i].n_tile2), (int)(local % bt.s[i].n_tile2)};
}

// Pass-2 units in order without a division per unit: (sender, group, tile) advanced by one.
__device__ __forceinline__ void next2(const TcBatch& bt, Unit& un) {
    if (un.i >= bt.n) return;   // past the last unit
    if (++un.c == bt.s[un.i].n_tile2) {
        un.c = 0;
        if (++un.s == bt.nL * bt.Hkv) {
            un.s = 0;
            ++un.i;
        }
    }
}

// Pass-1 units likewise (sender, group, chunk).
__device__ __forceinline__ void next1(const TcBatch& bt, Unit& un) {
    if (un.i >= bt.n) return;
    if (++un.c == bt.s[un.i].n_chunk1 / 4) {
        un.c = 0;
        if (++un.s == bt.nL * bt.Hkv) {
            un.s = 0;
            ++un.i;
        }
    }
}

// Contiguous share of `total` units for this CTA.
__device__ __forceinline__ void my_range(int64_t total, int64_t* b, int64_t* e) {
    *b = total * blockIdx.x / gridDim.x;
    *e = total * (blockIdx.x + 1) / gridDim.x;
}

// Shared memory: [Q: 2 blocks x rpad x 128 B][offset terms: rpad x 32 B][ones: 4 KB]
// [K ring: stages x 32 KB][Ctl][epilogue scratch]
struct Smem {
    uint8_t* q;
    uint8_t* ext;     // pass 2: offset terms of Q's rows [rpad][32 B], 32-byte swizzle
    uint8_t* ones;    // pass 2: ones columns [128][32 B], 32-byte swizzle
    uint8_t* k;
    Ctl* ctl;
    float* epi;
};

__device__ __forceinline__ Smem carve(uint8_t* raw, const TcBatch& bt) {
    Smem sm;
    uint8_t* base = align1024(raw);
    sm.q = base;
    sm.ext = base + (size_t)2 * bt.rpad_max * 128;
    sm.ones = sm.ext + (size_t)bt.rpad_max * 32;
    sm.k = sm.ones + 128 * 32;
    sm.ctl = reinterpret_cast<Ctl*>(sm.k + (size_t)bt.stages * kTileBytes);
    sm.epi = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(sm.ctl) + 512);
    return sm;
}

// `releasers`: warps that arrive on a TMEM buffer's empty barrier (pass 1: the eight warps of a
// group; pass 2: the four warps of one column half).
__device__ __forceinline__ void init_ctl(Ctl* ctl, int stages, int releasers, uint64_t wait_ns) {
    for (int k = 0; k < stages; ++k) {
        mbar_init(&ctl->k_full[k], 1);
        mbar_init(&ctl->k_empty[k], 1);
    }
    for (int b = 0; b < 4; ++b) {
        mbar_init(&ctl->t_full[b], 1);
        mbar_init(&ctl->t_empty[b], releasers);
    }
    mbar_init(&ctl->q_full, 1);
    mbar_init(&ctl->q_empty, 1);
    mbar_init(&ctl->drain, 1);
    mbar_init(&ctl->o_full, 1);
    mbar_init(&ctl->stall, 1);
    ctl->wait_ns = wait_ns;
    for (int k = 0; k < 16; ++k) {
        mbar_init(&ctl->xb[k >> 3][(k >> 2) & 1][k & 3], 1);
        mbar_init(&ctl->xe[k >> 3][(k >> 2) & 1][k & 3], 1);
    }
    ctl->abort = 0;
    fence_barrier_init();
}

// Producer: Q of group s (all rows, both column blocks) into the Q region.
// Pass 2 (with_ext) also brings the rows' offset terms of group s = l * Hkv + g.
__device__ __forceinline__ void load_q(const TcBatch& bt, const TcSender& sd, const Smem& sm, int l, int g,
                                       bool with_ext) {
    const uint32_t bytes = (uint32_t)sd.R_pad * (with_ext ? 256u + 32u : 256u);
    mbar_arrive_expect_tx(&sm.ctl->q_full, bytes);
    if (with_ext)
        for (int b = 0; b < sd.n_ebox; ++b)
            tma_load_3d(sm.ext + (size_t)b * sd.ebox_rows * 32, &sd.emap, &sm.ctl->q_full, 0, b * sd.ebox_rows,
                        l * bt.Hkv + g);
    for (int kb = 0; kb < 2; ++kb)
        for (int b = 0; b < sd.n_qbox; ++b)
            tma_load_4d(sm.q + (size_t)kb * bt.rpad_max * 128 + (size_t)b * sd.qbox_tok * bt.G * 128, &sd.qmap,
                        &sm.ctl->q_full, 64 * kb, g * bt.G, b * sd.qbox_tok, l);
}

__device__ __forceinline__ void load_k(const TcSender& sd, const Smem& sm, int stage, int l, int g, int32_t t_start) {
    uint8_t* dst = sm.k + (size_t)stage * kTileBytes;
    mbar_arrive_expect_tx(&sm.ctl->k_full[stage], kTileBytes);
    tma_load_4d(dst, &sd.kmap, &sm.ctl->k_full[stage], 0, t_start, g, l);
    tma_load_4d(dst + kTileBytes / 2, &sd.kmap, &sm.ctl->k_full[stage], 64, t_start, g, l);
}

// One K = 128 contraction (8 UMMA K-steps).  a_base / b_base: first column block of each
// operand (rows of 128 B); the second column block sits `a_blk` / `b_blk` bytes later.
// The descriptors are built once; a K-step only moves the start-address field.
__device__ __forceinline__ void mma_k128(uint32_t d_tmem, uint32_t a_base, uint32_t a_blk, uint32_t b_base,
                                        uint32_t b_blk, uint32_t idesc) {
    const uint64_t ad0 = smem_desc_sw128(a_base), bd0 = smem_desc_sw128(b_base);
    const uint64_t ad1 = ad0 + (a_blk >> 4), bd1 = bd0 + (b_blk >> 4);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const uint64_t off = (uint64_t)((k & 3) * 2);   // 32 bytes >> 4
        umma_bf16(d_tmem, (k < 4 ? ad0 : ad1) + off, (k < 4 ? bd0 : bd1) + off, idesc, k > 0 ? 1u : 0u);
    }
}

// One 32-column block of pass 1 for this lane's row: running offset m (log2 domain) and
// sum of exp2(c z - m).  The first block of a chunk (known from the loop indices: testing m
// instead cost 2%) sets m to its max, or to -FLT_MAX when it holds no position, in which case
// neither does the rest of the chunk; later blocks reuse m without a check (a per-block test
// and redo cost 11% of this kernel).  Values up to 2^127 above
// the first block are exact; a logit so far above it that exp2 or the sum overflows leaves an
// infinite sum, and the combine kernel recomputes that row's statistics from Q and K.
__device__ __forceinline__ void stats_block(float (&v)[32], int nvalid, float c, uint64_t cc, float& m, float& sum,
                                            bool first) {
    if (nvalid < 32) {
#pragma unroll
        for (int q = 0; q < 32; ++q) v[q] = q < nvalid ? v[q] : -INFINITY;
    }
    if (first) m = fmaxf(max_tree1(v) * c, -FLT_MAX);
    const uint64_t nm = pack2(-m, -m);
    float acc[4] = {0.f, 0.f, 0.f, 0.f};   // exp2 results are summed as scalars (no pair packing)
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        float a0, a1;
        unpack2(ffma2(pack2(v[2 * q], v[2 * q + 1]), cc, nm), a0, a1);
        acc[(2 * q) & 3] += ex2(a0);
        acc[(2 * q + 1) & 3] += ex2(a1);
    }
    sum += (acc[0] + acc[1]) + (acc[2] + acc[3]);
}

// ===========================================================================
// pass 1
// ===========================================================================
// Epilogue: the two groups of four warps take alternate K tiles (tile index within the
// chunk, even -> group 0).  Thread = TMEM lane = row 128 h + lane of every half h; it keeps
// the running max and sum of exp2 of its rows over its group's tiles of the chunk and writes
// them as partial (chunk, group); the combine kernel merges all partials of a group s.
__global__ void __launch_bounds__(kThreadsTc, 1) k_stats_tc(const __grid_constant__ TcBatch bt) {
    extern __shared__ uint8_t smem_raw[];
    const Smem sm = carve(smem_raw, bt);
    Ctl* ctl = sm.ctl;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) init_ctl(ctl, bt.stages, 8, bt.wait_ns);
    if (warp == 1) {
        tmem_alloc(&ctl->tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = ctl->tmem_base;
    int64_t ub, ue;
    my_range(bt.units1, &ub, &ue);
    const int stages = bt.stages;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (elect_one()) {
            int64_t kt = 0, qn = 0;   // K tiles and Q loads issued
            int st = 0;               // ring slot of the next K tile and its phase parity
            uint32_t ph = 0;
            int prev = -1;
            bool ok = true;
            Unit un = decode1(bt, ub);
            for (int64_t u = ub; u < ue && ok; ++u, next1(bt, un)) {
                const TcSender& sd = bt.s[un.i];
                const int l = un.s / bt.Hkv, g = un.s % bt.Hkv;
                const int key = un.i * 65536 + un.s;
                if (key != prev) {
                    if (!(ok = wait_bar(&ctl->q_empty, (uint32_t)((qn & 1) ^ 1), ctl, bt.err, 0))) break;
                    load_q(bt, sd, sm, l, g, false);
                    ++qn;
                    prev = key;
                }
                const int64_t c0 = (int64_t)un.c * kChunk1;
                const int nt = (int)((min((int64_t)kChunk1, sd.T - c0) + kTileRows - 1) / kTileRows);
                for (int tile = 0; tile < nt; ++tile) {
                    if (!(ok = wait_bar(&ctl->k_empty[st], ph ^ 1u, ctl, bt.err, 1))) break;
                    load_k(sd, sm, st, l, g, (int32_t)(c0 + tile * kTileRows));
                    ++kt;
                    if (++st == stages) { st = 0; ph ^= 1u; }
                }
            }
            // drain: every issued load must land before the CTA exits
            for (int64_t k = kt - stages > 0 ? kt - stages : 0; k < kt; ++k)
                drain_wait(&ctl->k_full[k % stages], (uint32_t)((k / stages) & 1));
            if (qn > 0) drain_wait(&ctl->q_full, (uint32_t)((qn - 1) & 1));
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            int64_t qn = 0, jg0 = 0, jg1 = 0;   // Q loads consumed; items issued per epilogue group
            int st = 0;                          // ring slot of the next K tile and its phase parity
            uint32_t ph = 0;
            int prev = -1;
            bool ok = true;
            // failure-detection test: wait on a barrier that nothing arrives on, so the bounded
            // wait gives up, sets the abort flag and every role of this CTA leaves
            if (bt.stall && blockIdx.x == 0) ok = wait_bar(&ctl->stall, 0, ctl, bt.err, 6);
            Unit un = decode1(bt, ub);
            for (int64_t u = ub; u < ue && ok; ++u, next1(bt, un)) {
                const TcSender& sd = bt.s[un.i];
                const int key = un.i * 65536 + un.s;
                if (key != prev) {
                    if (prev >= 0) umma_commit(&ctl->q_empty);
                    if (!(ok = wait_bar(&ctl->q_full, (uint32_t)(qn & 1), ctl, bt.err, 2))) break;
                    tc_fence_after();
                    ++qn;
                    prev = key;
                }
                const int halves = sd.R_pad / 128;
                const int64_t c0 = (int64_t)un.c * kChunk1;
                const int nt = (int)((min((int64_t)kChunk1, sd.T - c0) + kTileRows - 1) / kTileRows);
                for (int tile = 0; tile < nt && ok; ++tile) {
                    if (!(ok = wait_bar(&ctl->k_full[st], ph, ctl, bt.err, 3))) break;
                    tc_fence_after();
                    const uint32_t kaddr = smem_u32(sm.k + (size_t)st * kTileBytes);
                    const int grp = tile & 1;     // epilogue group that owns this tile
                    for (int h = 0; h < halves; ++h) {
                        const int64_t j = grp ? jg1++ : jg0++;
                        const int buf = 2 * grp + (int)(j & 1);
                        if (!(ok = wait_bar(&ctl->t_empty[buf], (uint32_t)(((j >> 1) & 1) ^ 1), ctl, bt.err, 4))) break;
                        tc_fence_after();
                        mma_k128(tmem + buf * 128, smem_u32(sm.q) + h * 128 * 128, (uint32_t)bt.rpad_max * 128,
                                 kaddr, kTileBytes / 2, idesc_bf16_f32(128, 128));
                        umma_commit(&ctl->t_full[buf]);
                    }
                    umma_commit(&ctl->k_empty[st]);
                    if (++st == stages) { st = 0; ph ^= 1u; }
                }
            }
            umma_commit(&ctl->drain);
            drain_wait(&ctl->drain, 0);
        }
    } else {
        // ---------------- epilogue: running max / sum per row ----------------
        // 16 warps: quad = (warp - 2) / 4; group = quad / 2 takes the tiles whose index in the
        // chunk has its parity, half = quad % 2 takes positions half*64 .. +64 of each tile.
        const int quad = (warp - 2) >> 2, grp = quad >> 1, hf = quad & 1;
        const int sp = warp & 3;                 // TMEM lane quarter
        const int L = sp * 32 + lane;
        const uint32_t lane_addr = (uint32_t)(sp * 32) << 16;
        const float c = bt.sl2e;
        const uint64_t cc = pack2(c, c);
        int64_t j = 0;                           // items of this group so far
        bool ok = true;
        Unit un = decode1(bt, ub);
        for (int64_t u = ub; u < ue && ok; ++u, next1(bt, un)) {
            const TcSender& sd = bt.s[un.i];
            const int halves = sd.R_pad / 128;
            const int64_t c0 = (int64_t)un.c * kChunk1;
            const int nt = (int)((min((int64_t)kChunk1, sd.T - c0) + kTileRows - 1) / kTileRows);
            float M[4], S[4];                    // per half: offset (log2 domain) and sum of exp2(c z - offset)
#pragma unroll
            for (int h = 0; h < 4; ++h) { M[h] = -INFINITY; S[h] = 0.f; }
            for (int tile = 0; tile < nt && ok; ++tile) {
                if ((tile & 1) != grp) continue;
                const int nvalid = (int)min((int64_t)kTileRows, sd.T - (c0 + tile * kTileRows)) - hf * 64;
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    if (h >= halves) break;
                    const int buf = 2 * grp + (int)(j & 1);
                    if (!(ok = wait_bar(&ctl->t_full[buf], (uint32_t)((j >> 1) & 1), ctl, bt.err, 5))) break;
                    ++j;
                    tc_fence_after();
                    const uint32_t ta = tmem + lane_addr + buf * 128 + hf * 64;
                    float m = M[h], sum = S[h];
#pragma unroll
                    for (int half32 = 0; half32 < 2; ++half32) {
                        float v[32];
                        tmem_ld32(ta + 32 * half32, v);
                        tmem_wait_ld(v);
                        if (half32 == 1) {
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(&ctl->t_empty[buf]);   // registers hold the rest
                        }
                        stats_block(v, nvalid - 32 * half32, c, cc, m, sum, tile == grp && half32 == 0);
                    }
                    M[h] = m;
                    S[h] = sum;
                }
            }
            if (!ok) break;
            // this warp's partial statistics for the chunk: slot 4 c + 2 grp + hf (rows of
            // tiles it saw none of stay (-inf, 0), rows of positions past T (-FLT_MAX, 0), both
            // of which add nothing); the combine kernel merges all slots
            float2* dst = sd.stats + ((int64_t)un.s * sd.n_chunk1 + 4 * un.c + 2 * grp + hf) * sd.R;
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                const int row = h * 128 + L;
                if (h < halves && row < sd.R) dst[row] = make_float2(M[h], S[h]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ===========================================================================
// pass 2
// ===========================================================================
// Window max over lanes lane-PH .. lane+PH of x (valid for lanes 3..28, the output lanes).
template <int PH>
__device__ __forceinline__ float lane_pool(float x) {
    if (PH == 0) return x;
    if (PH == 1) {
        const float a = __shfl_up_sync(0xffffffffu, x, 1);
        const float b = __shfl_down_sync(0xffffffffu, x, 1);
        return fmaxf(x, fmaxf(a, b));
    }
    if (PH == 2) {
        const float a1 = fmaxf(x, __shfl_down_sync(0xffffffffu, x, 1));        // [l, l+1]
        const float b1 = __shfl_up_sync(0xffffffffu, a1, 2);                   // [l-2, l-1]
        return fmaxf(fmaxf(a1, b1), __shfl_down_sync(0xffffffffu, x, 2));      // [l-2, l+2]
    }
    const float a1 = fmaxf(x, __shfl_down_sync(0xffffffffu, x, 1));            // [l, l+1]
    const float a2 = fmaxf(a1, __shfl_down_sync(0xffffffffu, a1, 2));          // [l, l+3]
    return fmaxf(a2, __shfl_up_sync(0xffffffffu, a2, 3));                      // [l-3, l+3]
}

template <bool P2>
__device__ __forceinline__ float pow_p(float x, float p) {
    if (P2) return x * x;
    return x > 0.f ? ex2(p * lg2(x)) : 0.f;
}

// One 32-column block of pass 2 for this lane's position: a / G = exp2(c z - offset) per
// column, b = sum over the G heads of each token, then Pool over positions and the sums.
// Tokens 2i and 2i + 1 share one packed f32x2 add or fma: lane 0 of each pair is the chain of
// even tokens and lane 1 that of odd tokens, the same order of additions as two scalar chains.
template <int G, int PH, bool P2>
__device__ __forceinline__ void accum_block(const float (&v)[32], uint64_t cc, bool valid, bool all_valid, float p,
                                            bool p_inf, float (&nacc)[2], float (&bsum)[2]) {
    float e[32];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        float a0, a1, a2, a3;
        unpack2(fmul2(pack2(v[4 * q], v[4 * q + 1]), cc), a0, a1);
        unpack2(fmul2(pack2(v[4 * q + 2], v[4 * q + 3]), cc), a2, a3);
        e[4 * q] = ex2(a0);
        e[4 * q + 1] = ex2(a1);
        e[4 * q + 2] = ex2(a2);
        e[4 * q + 3] = ex2(a3);
    }
    constexpr int NP = 16 / G;   // token pairs in these 32 columns
    uint64_t b[NP];
#pragma unroll
    for (int i = 0; i < NP; ++i) {
        if (G == 1) b[i] = pack2(e[2 * i], e[2 * i + 1]);
        if (G == 2) b[i] = fadd2(pack2(e[4 * i], e[4 * i + 2]), pack2(e[4 * i + 1], e[4 * i + 3]));
        if (G == 4)
            b[i] = fadd2(fadd2(pack2(e[8 * i], e[8 * i + 4]), pack2(e[8 * i + 1], e[8 * i + 5])),
                         fadd2(pack2(e[8 * i + 2], e[8 * i + 6]), pack2(e[8 * i + 3], e[8 * i + 7])));
    }
    if (!all_valid) {
#pragma unroll
        for (int i = 0; i < NP; ++i) b[i] = valid ? b[i] : 0ull;
    }
    uint64_t bs = pack2(bsum[0], bsum[1]), na = pack2(nacc[0], nacc[1]);
#pragma unroll
    for (int i = 0; i < NP; ++i) {
        float b0, b1;
        unpack2(b[i], b0, b1);
        const float p0 = lane_pool<PH>(b0), p1 = lane_pool<PH>(b1);
        bs = fadd2(bs, b[i]);
        if (P2) {
            const uint64_t pp = pack2(p0, p1);
            na = ffma2(pp, pp, na);
        } else if (p_inf) {   // p = infinity: largest pooled value
            nacc[0] = fmaxf(nacc[0], p0);
            nacc[1] = fmaxf(nacc[1], p1);
        } else {
            nacc[0] += pow_p<false>(p0, p);
            nacc[1] += pow_p<false>(p1, p);
        }
    }
    unpack2(bs, bsum[0], bsum[1]);
    if (P2) unpack2(na, nacc[0], nacc[1]);
}

// Pass 2, G = 4: head sums of the four tokens in 16 columns (exp2(c z - offset) summed over
// each token's four heads) as the pairs (b0, b1) and (b2, b3); the packed adds keep each
// token's order (e0 + e1) + (e2 + e3).
__device__ __forceinline__ void head_sums16(const float (&v)[16], uint64_t cc, uint64_t& b01, uint64_t& b23) {
    float e[16];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        float a0, a1, a2, a3;
        unpack2(fmul2(pack2(v[4 * q], v[4 * q + 1]), cc), a0, a1);
        unpack2(fmul2(pack2(v[4 * q + 2], v[4 * q + 3]), cc), a2, a3);
        e[4 * q] = ex2(a0);
        e[4 * q + 1] = ex2(a1);
        e[4 * q + 2] = ex2(a2);
        e[4 * q + 3] = ex2(a3);
    }
    b01 = fadd2(fadd2(pack2(e[0], e[4]), pack2(e[1], e[5])), fadd2(pack2(e[2], e[6]), pack2(e[3], e[7])));
    b23 = fadd2(fadd2(pack2(e[8], e[12]), pack2(e[9], e[13])), fadd2(pack2(e[10], e[14]), pack2(e[11], e[15])));
}

// Epilogue: each warp owns 32 TMEM lanes = positions t0 + 26 w - 3 + lane (w = lane quarter);
// lanes 3..28 are its output positions, the 3 lanes on each side their Pool margin (the K
// rows of the four quarters overlap by 6 positions).  The two groups take alternate tiles.
template <int G, int PH, bool P2>
__global__ void __launch_bounds__(kThreadsTc, 1) k_accum_tc(const __grid_constant__ TcBatch bt) {
    extern __shared__ uint8_t smem_raw[];
    const Smem sm = carve(smem_raw, bt);
    Ctl* ctl = sm.ctl;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) init_ctl(ctl, bt.stages, 4, bt.wait_ns);
    if (warp == 1) {
        tmem_alloc(&ctl->tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = ctl->tmem_base;
    int64_t ub, ue;
    my_range(bt.units2, &ub, &ue);
    const int stages = bt.stages;

    if (warp == 0) {
        if (elect_one()) {
            int64_t kt = 0, qn = 0;   // K tiles and Q loads issued
            int st = 0;               // ring slot of the next K tile and its phase parity
            uint32_t ph = 0;
            int prev = -1;
            bool ok = true;
            // the ones columns of the offset K-step, once per CTA
            mbar_arrive_expect_tx(&ctl->o_full, 128 * 32);
            tma_load_2d(sm.ones, &bt.omap, &ctl->o_full, 0, 0);
            Unit un = decode2(bt, ub);
            for (int64_t u = ub; u < ue && ok; ++u, next2(bt, un)) {
                const TcSender& sd = bt.s[un.i];
                const int l = un.s / bt.Hkv, g = un.s % bt.Hkv;
                const int key = un.i * 65536 + un.s;
                if (key != prev) {
                    if (!(ok = wait_bar(&ctl->q_empty, (uint32_t)((qn & 1) ^ 1), ctl, bt.err, 8))) break;
                    load_q(bt, sd, sm, l, g, true);
                    ++qn;
                    prev = key;
                }
                if (!(ok = wait_bar(&ctl->k_empty[st], ph ^ 1u, ctl, bt.err, 9))) break;
                // four 32-row boxes: quarter w holds positions t0 + 26 w - 3 .. + 31
                uint8_t* dst = sm.k + (size_t)st * kTileBytes;
                mbar_arrive_expect_tx(&ctl->k_full[st], kTileBytes);
                const int32_t t0 = (int32_t)((int64_t)un.c * kOut2);
                for (int w = 0; w < 4; ++w)
                    for (int kb = 0; kb < 2; ++kb)
                        tma_load_4d(dst + kb * (kTileBytes / 2) + w * 32 * 128, &sd.kmap32, &ctl->k_full[st],
                                    64 * kb, t0 + kOutW * w - kMargin, g, l);
                ++kt;
                if (++st == stages) { st = 0; ph ^= 1u; }
            }
            for (int64_t k = kt - stages > 0 ? kt - stages : 0; k < kt; ++k)
                drain_wait(&ctl->k_full[k % stages], (uint32_t)((k / stages) & 1));
            if (qn > 0) drain_wait(&ctl->q_full, (uint32_t)((qn - 1) & 1));
            drain_wait(&ctl->o_full, 0);
        }
    } else if (warp == 1) {
        if (elect_one()) {
            int64_t qn = 0;              // Q loads consumed
            uint32_t jpar = 0;           // bit b: parity of the items issued into TMEM buffer b
            int st = 0;                  // ring slot of the next K tile and its phase parity
            uint32_t ph = 0;
            int prev = -1;
            bool ok = wait_bar(&ctl->o_full, 0, ctl, bt.err, 15);
            tc_fence_after();
            const uint64_t ones_desc = smem_desc_sw32(smem_u32(sm.ones));
            const uint64_t ext_desc = smem_desc_sw32(smem_u32(sm.ext));
            Unit un = decode2(bt, ub);
            for (int64_t u = ub; u < ue && ok; ++u, next2(bt, un)) {
                const TcSender& sd = bt.s[un.i];
                const int key = un.i * 65536 + un.s;
                if (key != prev) {
                    if (prev >= 0) umma_commit(&ctl->q_empty);
                    if (!(ok = wait_bar(&ctl->q_full, (uint32_t)(qn & 1), ctl, bt.err, 10))) break;
                    tc_fence_after();
                    ++qn;
                    prev = key;
                }
                if (!(ok = wait_bar(&ctl->k_full[st], ph, ctl, bt.err, 11))) break;
                tc_fence_after();
                const uint32_t kaddr = smem_u32(sm.k + (size_t)st * kTileBytes);
                const int grp = (int)((u - ub) & 1);   // epilogue group that owns this tile
                if (sd.R_pad == 256) {
                    // both halves in one 256-column MMA (faster when the tile has no other rows);
                    // it waits for both halves' buffers and completes both
                    const uint32_t jp = (jpar >> (2 * grp)) & 3u;
                    jpar ^= 3u << (2 * grp);
                    if (!(ok = wait_bar(&ctl->t_empty[2 * grp], (jp & 1u) ^ 1u, ctl, bt.err, 12))) break;
                    if (!(ok = wait_bar(&ctl->t_empty[2 * grp + 1], (jp >> 1) ^ 1u, ctl, bt.err, 12))) break;
                    tc_fence_after();
                    mma_k128(tmem + grp * 256, kaddr, kTileBytes / 2, smem_u32(sm.q), (uint32_t)bt.rpad_max * 128,
                             idesc_bf16_f32(128, 256));
                    // one more K-step: ones (positions) x offset terms (rows) adds -offset / scale to
                    // every logit, so the epilogue needs only exp2(scale * D)
                    umma_bf16(tmem + grp * 256, ones_desc, ext_desc, idesc_bf16_f32(128, 256), 1u);
                    umma_commit(&ctl->t_full[2 * grp]);
                    umma_commit(&ctl->t_full[2 * grp + 1]);
                } else {
                    // one 128-column MMA per column half, each into its own buffer, so that each
                    // half's warps start as soon as their columns are done and release them on
                    // their own (the next chunk waits for one half, not for the whole group)
                    for (int r0 = 0; r0 < sd.R_pad && ok; r0 += 128) {
                        const int b = 2 * grp + ((r0 >> 7) & 1);
                        const uint32_t jp = (jpar >> b) & 1u;
                        jpar ^= 1u << b;
                        if (!(ok = wait_bar(&ctl->t_empty[b], jp ^ 1u, ctl, bt.err, 12))) break;
                        tc_fence_after();
                        mma_k128(tmem + b * 128, kaddr, kTileBytes / 2, smem_u32(sm.q) + r0 * 128,
                                 (uint32_t)bt.rpad_max * 128, idesc_bf16_f32(128, 128));
                        umma_bf16(tmem + b * 128, ones_desc, ext_desc + (uint64_t)((r0 * 32) >> 4),
                                  idesc_bf16_f32(128, 128), 1u);
                        umma_commit(&ctl->t_full[b]);
                    }
                }
                umma_commit(&ctl->k_empty[st]);
                if (++st == stages) { st = 0; ph ^= 1u; }
            }
            umma_commit(&ctl->drain);
            drain_wait(&ctl->drain, 0);
        }
    } else {
        // 16 warps: quad = (warp - 2) / 4; group = quad / 2 takes alternate tiles, half = quad % 2
        // takes columns half*128 .. +128 of each 256-column chunk (32 tokens when G = 4).
        const int ew = warp - 2, quad = ew >> 2, grp = quad >> 1, hf = quad & 1, sp = warp & 3;
        const uint32_t lane_addr = (uint32_t)(sp * 32) << 16;
        float2* xch = reinterpret_cast<float2*>(sm.epi);   // [parity][grp][sp][32]
        const float c = bt.sl2e;
        const uint64_t cc = pack2(c, c);
        int64_t j = 0, gt = 0;                   // chunks of this warp's buffer and tiles of this group so far
        int prev = -1;
        bool ok = true;
        // per-sender values live in registers and are refreshed when the group s changes
        // (indexed reads of the kernel-parameter block on every tile are slow)
        float* part = nullptr;                   // U partials of the current group s
        int64_t nST = 0;                         // distance between the U, N and D partials
        int64_t T = 0;
        int nch = 0, n_tile = 1, R_pad = 0;
        float inv_m = 0.f, inv_mh = 0.f;
        const int nS = bt.nL * bt.Hkv;
        Unit un = decode2(bt, ub);
        n_tile = bt.s[un.i].n_tile2;
        auto advance = [&]() {   // next unit (sender, group, tile) without parameter reads
            if (++un.c == n_tile) {
                un.c = 0;
                if (++un.s == nS) {
                    un.s = 0;
                    ++un.i;
                    if (un.i < bt.n) n_tile = bt.s[un.i].n_tile2;
                }
            }
        };
        if (grp == 1 && ub < ue) advance();
        for (int64_t u = ub + grp; u < ue && ok; u += 2, advance(), advance()) {
            const int key = un.i * 65536 + un.s;
            if (key != prev) {
                const TcSender& sd = bt.s[un.i];
                R_pad = sd.R_pad;
                nch = (sd.R_pad + 255) / 256;
                T = sd.T;
                inv_m = sd.inv_m;
                inv_mh = sd.inv_mh;
                nST = (int64_t)nS * sd.T;
                part = sd.part + (int64_t)un.s * sd.T;
                prev = key;
            }
            const int64_t pos = (int64_t)un.c * kOut2 + kOutW * sp - kMargin + lane;
            const bool valid = pos >= 0 && pos < T;
            const bool all_valid = __all_sync(0xffffffffu, valid);
            float nacc2[2] = {0.f, 0.f}, bsum2[2] = {0.f, 0.f};   // token partial sums (two chains)
            for (int ci = 0; ci < nch && ok; ++ci) {
                // this half's columns (R_pad is a multiple of 128: 0 or 128); a half with none has
                // no MMA and nothing to wait for
                const int ncol = min(128, min(256, R_pad - 256 * ci) - hf * 128);
                if (ncol <= 0) continue;
                if (!(ok = wait_bar(&ctl->t_full[2 * grp + hf], (uint32_t)(j & 1), ctl, bt.err, 13))) break;
                ++j;
                tc_fence_after();
                const uint32_t ta = tmem + lane_addr + grp * 256 + hf * 128;
                if (G == 4) {
                    // head sums of the warp's 32 tokens first, then the buffer goes back to the MMA
                    // while Pool and the token sums run from registers; each 16-column load is
                    // issued before the head sums of the one before it
                    uint64_t b[16];   // (token 2i, token 2i + 1)
                    {
                        float va[16], vb[16];
                        tmem_ld16(ta, va);
#pragma unroll
                        for (int k = 0; k < 8; k += 2) {
                            tmem_wait_ld(va);
                            tmem_ld16(ta + 16 * (k + 1), vb);
                            head_sums16(va, cc, b[2 * k], b[2 * k + 1]);
                            tmem_wait_ld(vb);
                            if (k + 2 < 8) tmem_ld16(ta + 16 * (k + 2), va);
                            head_sums16(vb, cc, b[2 * k + 2], b[2 * k + 3]);
                        }
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&ctl->t_empty[2 * grp + hf]);
                    if (!all_valid) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) b[i] = valid ? b[i] : 0ull;
                    }
                    uint64_t bs = pack2(bsum2[0], bsum2[1]), na = pack2(nacc2[0], nacc2[1]);
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        float b0, b1;
                        unpack2(b[i], b0, b1);
                        const float p0 = lane_pool<PH>(b0), p1 = lane_pool<PH>(b1);
                        bs = fadd2(bs, b[i]);
                        if (P2) {
                            const uint64_t pp = pack2(p0, p1);
                            na = ffma2(pp, pp, na);
                        } else if (bt.p_inf) {
                            nacc2[0] = fmaxf(nacc2[0], p0);
                            nacc2[1] = fmaxf(nacc2[1], p1);
                        } else {
                            nacc2[0] += pow_p<false>(p0, bt.p);
                            nacc2[1] += pow_p<false>(p1, bt.p);
                        }
                    }
                    unpack2(bs, bsum2[0], bsum2[1]);
                    if (P2) unpack2(na, nacc2[0], nacc2[1]);
                } else {
                    // 32-column steps; sixteen epilogue warps hide the TMEM load latency
#pragma unroll 1
                    for (int col = 0; col < (G == 4 ? 0 : ncol); col += 32) {
                        float v[32];
                        tmem_ld32(ta + col, v);
                        tmem_wait_ld(v);
                        accum_block<G, PH, P2>(v, cc, valid, all_valid, bt.p, bt.p_inf, nacc2, bsum2);
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&ctl->t_empty[2 * grp + hf]);
                }
            }
            if (!ok) break;
            // p = infinity keeps the largest pooled token value instead of the sum of powers
            const bool p_inf = !P2 && bt.p_inf;
            float nacc = p_inf ? fmaxf(nacc2[0], nacc2[1]) : nacc2[0] + nacc2[1];
            float bsum = bsum2[0] + bsum2[1];
            // the two column halves of the group add up their sums; half tp (the group's tile
            // parity) writes the results, so the halves take turns waiting for each other
            const int tp = (int)(gt & 1);
            float2* xs = xch + ((tp * 2 + grp) * 4 + sp) * 32;
            uint64_t* xb = &ctl->xb[tp][grp][sp];
            uint64_t* xe = &ctl->xe[tp][grp][sp];
            if ((hf ^ tp) == 1) {
                // the slot was last used two tiles ago: wait until the other half has read it
                if (!(ok = wait_bar(xe, (uint32_t)(((gt >> 1) & 1) ^ 1), ctl, bt.err, 7))) break;
                xs[lane] = make_float2(nacc, bsum);
                __syncwarp();
                if (lane == 0) mbar_arrive(xb);
            } else {
                if (!(ok = wait_bar(xb, (uint32_t)((gt >> 1) & 1), ctl, bt.err, 14))) break;
                const float2 o = xs[lane];
                __syncwarp();
                if (lane == 0) mbar_arrive(xe);
                nacc = p_inf ? fmaxf(nacc, o.x) : nacc + o.x;
                bsum += o.y;
                const float pb = lane_pool<PH>(bsum * inv_m);
                if (valid && lane >= kMargin && lane < kMargin + kOutW) {
                    part[pos] = bsum * inv_mh;
                    part[nST + pos] = p_inf ? nacc : nacc * inv_m;
                    part[2 * nST + pos] = p_inf ? pb : pow_p<P2>(pb, bt.p);
                }
            }
            ++gt;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
    std::call_once(g_encode_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
        else
            cudaGetLastError();
    });
    return g_encode;
}

// bf16 tensor map of `rank` dimensions (innermost first); strides in bytes of dims 1..rank-1.
bool encode_nd(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims, const cuuint64_t* strides_bytes,
               const cuuint32_t* box, CUtensorMapSwizzle swizzle) {
    auto fn = encoder();
    if (!fn || !base) return false;
    const cuuint32_t es[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), dims, strides_bytes, box,
              es, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_4d(CUtensorMap* m, const void* base, const cuuint64_t dims[4], const cuuint64_t strides_bytes[3],
               const cuuint32_t box[4]) {
    return encode_nd(m, base, 4, dims, strides_bytes, box, CU_TENSOR_MAP_SWIZZLE_128B);
}

size_t smem_bytes(int rpad_max, int stages) {
    return 1024 + (size_t)2 * rpad_max * 128 + (size_t)rpad_max * 32 + 128 * 32 + (size_t)stages * kTileBytes + 512 +
           2 * 2 * 4 * 32 * 8;
}

template <int G, int PH, bool P2>
cudaError_t launch_accum(const TcBatch& tb, size_t smem, int grid, cudaStream_t st) {
    cudaError_t e =
        cudaFuncSetAttribute(k_accum_tc<G, PH, P2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_accum_tc<G, PH, P2><<<grid, kThreadsTc, smem, st>>>(tb);
    return cudaGetLastError();
}

template <int G, bool P2>
cudaError_t launch_accum_gp(const TcBatch& tb, size_t smem, int grid, cudaStream_t st) {
    switch (tb.ph) {
        case 0: return launch_accum<G, 0, P2>(tb, smem, grid, st);
        case 1: return launch_accum<G, 1, P2>(tb, smem, grid, st);
        case 2: return launch_accum<G, 2, P2>(tb, smem, grid, st);
        case 3: return launch_accum<G, 3, P2>(tb, smem, grid, st);
    }
    return cudaErrorInvalidValue;
}

template <int G>
cudaError_t launch_accum_g(const TcBatch& tb, size_t smem, int grid, cudaStream_t st) {
    return tb.p_is_2 ? launch_accum_gp<G, true>(tb, smem, grid, st) : launch_accum_gp<G, false>(tb, smem, grid, st);
}

}  // namespace

bool tc_path_supported(int head_dim, int G, int pool_half, int max_query_tokens) {
    return head_dim == 128 && (G == 1 || G == 2 || G == 4) && pool_half <= 3 && max_query_tokens * G <= 512;
}

// Pass 1, combine, pass 2 on the tensor cores for senders [0, b.n) of `b`; the caller
// launches the finalize kernel.  `combine` is the shared statistics-combine launcher.
cudaError_t launch_score_tc(ScoreBatch& b, cudaStream_t st, int num_sms, uint32_t* err,
                            cudaError_t (*combine)(const ScoreBatch&, cudaStream_t)) {
    const int G = b.n_q_heads / b.n_kv_heads;
    const int nS = b.n_layers * b.n_kv_heads;
    // Encode every tensor map first: if the driver rejects one (an unusual stride
    // pattern), nothing has been launched and the caller uses the mma.sync passes.
    std::vector<TcBatch*> batches;
    auto free_all = [&] { for (TcBatch* p : batches) delete p; };
    // Sub-batches of at most kMaxTcSenders senders; paged senders are first copied into the
    // staging buffer (contiguous [nL][Hkv][T][128]), which each sub-batch reuses from its start,
    // so a sub-batch also ends where its paged senders would overflow the staging.
    std::vector<int> firsts;
    std::vector<DepageBatch*> depages;
    auto free_depages = [&] { for (DepageBatch* p : depages) delete p; };
    for (int b0 = 0; b0 < b.n;) {
        int nb = 0;
        int64_t used = 0;
        while (b0 + nb < b.n && nb < kMaxTcSenders) {
            const ScoreSender& s = b.s[b0 + nb];
            const int64_t e = s.pm.pages ? (int64_t)b.n_layers * b.n_kv_heads * s.T * 128 : 0;
            if (e > 0 && (!b.stage || e > b.stage_elems)) {   // no room: the mma.sync passes read pages
                free_all();
                free_depages();
                return cudaErrorNotSupported;
            }
            if (nb > 0 && used + e > b.stage_elems) break;
            used += e;
            ++nb;
        }
        firsts.push_back(b0);
        DepageBatch* dp = new DepageBatch();
        depages.push_back(dp);
        dp->n_layers = b.n_layers;
        dp->n_kv_heads = b.n_kv_heads;
        dp->err = err;
        TcBatch* tb = new TcBatch();
        batches.push_back(tb);
        tb->n = nb;
        b0 += nb;
        tb->nL = b.n_layers;
        tb->Hq = b.n_q_heads;
        tb->Hkv = b.n_kv_heads;
        tb->G = G;
        tb->sl2e = b.scale_log2e;
        tb->p = b.p;
        tb->p_is_2 = b.p == 2.f;
        tb->p_inf = b.p_inf;
        tb->ph = b.pool_half;
        tb->err = err;
        int rpad_max = 128;
        int64_t u1 = 0, u2 = 0, staged = 0;
        const int b_first = firsts.back();
        for (int k = 0; k < nb; ++k) {
            const ScoreSender& s = b.s[b_first + k];
            TcSender& d = tb->s[k];
            // K as the passes read it: the sender's own tensor, or its staged copy
            const uint16_t* kp = s.k;
            int64_t kl = s.ks_l, kh = s.ks_h, kpos = s.ks_p;
            if (s.pm.pages) {
                DepageSender& ds = dp->s[dp->n++];
                ds.k = s.k;
                ds.ks_l = s.ks_l;
                ds.ks_h = s.ks_h;
                ds.ks_p = s.ks_p;
                ds.pm = s.pm;
                ds.T = s.T;
                ds.out = b.stage + staged;
                kp = ds.out;
                kpos = 128;
                kh = s.T * 128;
                kl = (int64_t)b.n_kv_heads * s.T * 128;
                staged += kl * b.n_layers;
            }
            d.T = s.T;
            d.m = s.m;
            d.inv_m = 1.f / (float)s.m;
            d.inv_mh = 1.f / ((float)s.m * (float)b.n_kv_heads);
            d.R = s.m * G;
            d.R_pad = (d.R + 127) / 128 * 128;
            rpad_max = rpad_max > d.R_pad ? rpad_max : d.R_pad;
            d.n_chunk1 = (int32_t)(4 * ((s.T + kChunk1 - 1) / kChunk1));   // one partial per (chunk, group, half)
            d.n_tile2 = (int32_t)((s.T + kOut2 - 1) / kOut2);
            d.stats = b.stats + s.stats_off;
            d.offs = b.offs + s.offs_off;
            d.part = b.part + s.part_off;
            d.unit1_begin = u1;
            u1 += (int64_t)nS * (d.n_chunk1 / 4);
            d.unit2_begin = u2;
            u2 += (int64_t)nS * d.n_tile2;
            // Q arrives in boxes of at most 256 tokens that tile the padded rows exactly
            // (R_pad is a multiple of 128, so 128-token boxes always divide it for G = 1)
            const int tok_pad = d.R_pad / G;
            d.qbox_tok = tok_pad <= 256 ? tok_pad : 128;
            d.n_qbox = tok_pad / d.qbox_tok;
            if (d.n_qbox * d.qbox_tok != tok_pad) {
                free_all();
                free_depages();
                return cudaErrorNotSupported;
            }
            const cuuint64_t kd[4] = {128, (cuuint64_t)s.T, (cuuint64_t)b.n_kv_heads, (cuuint64_t)b.n_layers};
            const cuuint64_t ks[3] = {(cuuint64_t)kpos * 2, (cuuint64_t)kh * 2, (cuuint64_t)kl * 2};
            const cuuint32_t kbox[4] = {64, kTileRows, 1, 1};
            const cuuint64_t qd[4] = {128, (cuuint64_t)b.n_q_heads, (cuuint64_t)s.m, (cuuint64_t)b.n_layers};
            const cuuint64_t qs[3] = {(cuuint64_t)s.qs_h * 2, (cuuint64_t)s.qs_t * 2, (cuuint64_t)s.qs_l * 2};
            const cuuint32_t qbox[4] = {64, (cuuint32_t)G, (cuuint32_t)d.qbox_tok, 1};
            const cuuint32_t kbox32[4] = {64, 32, 1, 1};
            // offset terms [nS][R_pad][16] written by the combine kernel, boxes of at most 256 rows
            d.ebox_rows = d.R_pad <= 256 ? d.R_pad : 128;
            d.n_ebox = d.R_pad / d.ebox_rows;
            const cuuint64_t ed[3] = {(cuuint64_t)kExtCols, (cuuint64_t)d.R_pad, (cuuint64_t)nS};
            const cuuint64_t es[2] = {(cuuint64_t)kExtCols * 2, (cuuint64_t)d.R_pad * kExtCols * 2};
            const cuuint32_t ebox[3] = {(cuuint32_t)kExtCols, (cuuint32_t)d.ebox_rows, 1};
            if (!encode_4d(&d.kmap, kp, kd, ks, kbox) || !encode_4d(&d.kmap32, kp, kd, ks, kbox32) ||
                !encode_4d(&d.qmap, s.q, qd, qs, qbox) || d.n_ebox * d.ebox_rows != d.R_pad || !b.ext ||
                !encode_nd(&d.emap, b.ext + s.ext_off, 3, ed, es, ebox, CU_TENSOR_MAP_SWIZZLE_32B)) {
                free_all();
                free_depages();
                return cudaErrorNotSupported;
            }
        }
        const cuuint64_t od[2] = {(cuuint64_t)kExtCols, 128};
        const cuuint64_t os[1] = {(cuuint64_t)kExtCols * 2};
        const cuuint32_t obox[2] = {(cuuint32_t)kExtCols, 128};
        if (!encode_nd(&tb->omap, b.ones, 2, od, os, obox, CU_TENSOR_MAP_SWIZZLE_32B)) {
            free_all();
            free_depages();
            return cudaErrorNotSupported;
        }
        tb->rpad_max = rpad_max;
        tb->stages = rpad_max > 256 ? 2 : 4;
        tb->units1 = u1;
        tb->units2 = u2;
        tb->wait_ns = b.wait_ns;
        tb->stall = batches.size() == 1 ? b.stall : 0;   // the first launch only
    }
    cudaError_t e = cudaSuccess;
    for (size_t k = 0; k < batches.size() && e == cudaSuccess; ++k) {
        TcBatch* tb = batches[k];
        const int b0 = firsts[k];
        const size_t smem = smem_bytes(tb->rpad_max, tb->stages);
        e = cudaFuncSetAttribute(k_stats_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e == cudaSuccess) {
            stage_mark(b.timer, kStageStart, st);
            e = launch_depage(*depages[k], st, num_sms);   // timed with pass 1
        }
        if (e == cudaSuccess) {
            const int g1 = (int)(tb->units1 < num_sms ? tb->units1 : num_sms);
            k_stats_tc<<<g1, kThreadsTc, smem, st>>>(*tb);
            stage_mark(b.timer, kStageStats, st);
            e = cudaGetLastError();
        }
        if (e == cudaSuccess) {
            // combine reads this batch's chunk counts (512-position chunks)
            ScoreBatch* sub = new ScoreBatch(b);
            sub->n = tb->n;
            for (int j = 0; j < tb->n; ++j) {
                sub->s[j] = b.s[b0 + j];
                sub->s[j].n_chunk1 = tb->s[j].n_chunk1;
            }
            e = combine(*sub, st);
            stage_mark(b.timer, kStageCombine, st);
            delete sub;
        }
        if (e == cudaSuccess) {
            const int g2 = (int)(tb->units2 < num_sms ? tb->units2 : num_sms);
            if (G == 4) e = launch_accum_g<4>(*tb, smem, g2, st);
            else if (G == 2) e = launch_accum_g<2>(*tb, smem, g2, st);
            else e = launch_accum_g<1>(*tb, smem, g2, st);
            stage_mark(b.timer, kStageAccum, st);
        }
    }
    free_all();
    free_depages();
    return e;
}

}  // namespace cbk
