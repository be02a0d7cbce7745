// Internal interface between the C-ABI layer (cb_api.cu) and the kernels.
// Everything here is device-side or launch plumbing; no host-side validation.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace cbk {

constexpr int kMaxBatch = 64;        // senders per launch (larger calls are split)
constexpr int kStatsChunk = 256;     // positions per pass-1 block (mma.sync path)
constexpr int kStatsChunkTc = 1024;  // positions per pass-1 chunk (tcgen05 path, four partials each)

// Pass-1 partial slots a sender of T positions may need on either path.
inline int64_t stats_slots(int64_t T) {
    const int64_t a = (T + kStatsChunk - 1) / kStatsChunk;
    const int64_t b = 4 * ((T + kStatsChunkTc - 1) / kStatsChunkTc);
    return a > b ? a : b;
}
constexpr int kAccumChunk = 128;     // output positions per pass-2 block
constexpr int kHalo = 8;             // extra positions each side of a pass-2 block (>= pool_width/2)
constexpr int kMaxPoolWidth = 15;
constexpr int kMaxSpanWidth = 256;
constexpr int kFinSlices = 16;        // finalize: groups summed in 16 fixed slices
constexpr int kMaxQueryTokens = 1024;

// Device error word bits (set by kernels' own bounds checks).
constexpr uint32_t kErrCompactIndex = 1u;
constexpr uint32_t kErrSelectBudget = 2u;
constexpr uint32_t kErrTimeout = 4u;       // a bounded mbarrier wait gave up
constexpr uint32_t kErrGatherIndex = 8u;   // a message-row index outside [0, T)
constexpr uint32_t kErrPageIndex = 16u;    // a block-table entry outside [0, n_pages)

// Paged cache layout (block table): position t is row t & (2^shift - 1) of page
// pages[t >> shift].  pages == nullptr: the strided layout, position t at t * s_pos.
struct PageMap {
    const int32_t* pages;
    int64_t s_page;
    int64_t n_pages;
    int32_t shift;            // log2(page_size)
};

// Elements from the (l, g) base of a sender's cache to position t's row, or -1 when the
// block-table entry lies outside [0, n_pages) (the row must not be read).
__device__ __forceinline__ int64_t row_offset(const PageMap& pm, int64_t s_pos, int64_t t) {
    if (!pm.pages) return t * s_pos;
    const int32_t page = __ldg(pm.pages + (t >> pm.shift));
    if (page < 0 || page >= pm.n_pages) return -1;
    return (int64_t)page * pm.s_page + (t & ((int64_t(1) << pm.shift) - 1)) * s_pos;
}

// Optional per-kernel timing of the score step (owned by the context; see cb_stage_times).
struct StageTimer;
enum ScoreStage { kStageStart = 0, kStageStats = 1, kStageCombine = 2, kStageAccum = 3, kStageFinalize = 4 };
// Records an event on `st` marking the end of `stage` (no-op when timer is null).
void stage_mark(StageTimer* timer, int stage, cudaStream_t st);

struct ScoreSender {
    const uint16_t* k;        // K[l][g][t][:] at k + l*ks_l + g*ks_h + t*ks_p
    const uint16_t* q;        // Q[l][r][h][:] at q + l*qs_l + r*qs_t + h*qs_h
    float* scores;            // [T]
    int64_t T;
    int64_t ks_l, ks_h, ks_p;
    PageMap pm;               // paged layout of K, or pages == nullptr
    int64_t qs_l, qs_t, qs_h;
    const uint16_t* kself;    // the query tokens' own keys Ks[l][u][g][:] or null
    int64_t kss_l, kss_t, kss_h;
    int32_t m;
    int32_t n_chunk1;         // ceil(T / kStatsChunk)
    int32_t n_chunk2;         // ceil(T / kAccumChunk)
    int64_t stats_off;        // float2 offset of this sender's pass-1 partials
    int64_t offs_off;         // float offset of this sender's per-row softmax offsets
    int64_t ext_off;          // bf16 offset of this sender's [nS][R_pad][16] offset rows (tcgen05 passes)
    int64_t part_off;         // float offset of this sender's [3][nS][T] partials
    int64_t blk1_begin;       // first pass-1 block of this sender
    int64_t blk2_begin;       // first pass-2 block of this sender
};

struct ScoreBatch {
    int32_t n;
    int32_t n_layers, n_q_heads, n_kv_heads, head_dim;
    float scale_log2e;        // softmax_scale * log2(e)
    float p, alpha;
    int32_t p_inf;            // p = +infinity: N and D are maxima, C = N / D (App. D.2)
    int32_t pool_half;        // pool_width / 2
    int32_t use_tc;           // 1: tcgen05 passes, 0: mma.sync passes
    uint32_t* err;            // device error word
    StageTimer* timer;        // host-side; null unless stage timing is enabled
    float2* stats;            // pass-1 partial (max, sum) in log2 domain
    float* offs;              // per-row log2 offsets (max + log2(sum) + log2(G))
    uint16_t* ext;            // tcgen05 passes: -offset / scale_log2e per row as three bf16 terms
                              // (hi, mid, lo, then 13 zeros; -1e30 on padding rows), else null
    const uint16_t* ones;     // tcgen05 passes: [128][16] bf16, columns 0-2 = 1, the rest 0
    float* part;              // per-group U_s, N_s, D_s partials
    uint16_t* stage;          // tcgen05 passes: contiguous copies of paged senders' K
    int64_t stage_elems;      // its capacity (bf16 elements)
    uint64_t wait_ns;         // tcgen05 passes: limit of one bounded mbarrier wait
    int32_t stall;            // tcgen05 passes: failure-detection test (one wait nothing completes)
    ScoreSender s[kMaxBatch];
};

// Contiguous copy of paged caches: out[l][g][t][:] = K[l][g][t][:] read through the block table.
constexpr int kMaxDepage = 32;
struct DepageSender {
    const uint16_t* k;        // the paged cache
    int64_t ks_l, ks_h, ks_p;
    PageMap pm;
    int64_t T;
    uint16_t* out;            // [nL][Hkv][T][128]
};

struct DepageBatch {
    int32_t n;
    int32_t n_layers, n_kv_heads;
    uint32_t* err;
    DepageSender s[kMaxDepage];
};

constexpr int kExtCols = 16;   // one bf16 K-step: the extra contraction column block of pass 2

// Query rows padded to the 128-row granule of the tcgen05 passes.
__host__ __device__ inline int64_t rows_pad128(int64_t rows) { return (rows + 127) / 128 * 128; }

struct SelectSender {
    const float* scores;
    int32_t* idx;
    int64_t T;
    int64_t B;
    float* span_keys;         // scratch [n_spans]
};

struct SelectBatch {
    int32_t n;
    int32_t n_sink, n_latent, span_w;
    uint32_t* err;
    SelectSender s[kMaxBatch];
};

struct CompactSender {
    const uint16_t* k;
    const uint16_t* v;
    const int32_t* idx;
    int64_t T;
    int64_t ks_l, ks_h, ks_p;
    PageMap pm;               // paged layout of K and V, or pages == nullptr
    int64_t B;
    int64_t out_off;
    int64_t row_begin;        // first row (of n_layers*n_kv_heads*B*2) of this sender
};

struct CompactBatch {
    int32_t n;
    int32_t n_layers, n_kv_heads, head_dim;
    uint16_t* k_out;
    uint16_t* v_out;
    int64_t o_layer, o_head;
    int64_t total_rows;
    uint32_t* err;
    CompactSender s[kMaxBatch];
};

// Message rows (Sec. 3.1 "State Representation", App. C.3): row j of sender i's message is
// row idx[j] of its per-position table.
struct GatherSender {
    const uint8_t* src;       // row t at src + t * src_stride (bytes)
    const int32_t* idx;       // count indices into [0, T)
    int64_t T;
    int64_t src_stride;
    int64_t count;
    int64_t out_off;          // first output row of this sender
};

struct GatherBatch {
    int32_t n;
    int64_t row_bytes;        // bytes per row: a multiple of 4
    uint8_t* out;             // row r at out + r * out_stride
    int64_t out_stride;
    uint32_t* err;
    GatherSender s[kMaxBatch];
};

// Records the message cb_last_error(NULL) returns (entry points without a context).
void set_context_free_error(const char* msg);

// Finalize tiles of a sender of T positions, and the floats of its slice sums.

// True when the tcgen05 score passes handle this shape.
bool tc_path_supported(int head_dim, int G, int pool_half, int max_query_tokens);

// Launchers (return the launch error, if any).
// *path_out: 2 when the tcgen05 passes ran, 1 for the mma.sync passes.
cudaError_t launch_score(const ScoreBatch& b, cudaStream_t st, int num_sms, int* path_out);
cudaError_t launch_select(const SelectBatch& b, cudaStream_t st);
cudaError_t launch_compact(const CompactBatch& b, cudaStream_t st, int num_sms);
cudaError_t launch_gather(const GatherBatch& b, cudaStream_t st, int num_sms);
// head_dim = 128 only (the tcgen05 passes' shape).
cudaError_t launch_depage(const DepageBatch& b, cudaStream_t st, int num_sms);
// Staging elements the tcgen05 passes want for paged senders (0 when none is paged): enough
// for the largest paged sender and for paged sub-batches up to kStageBudget elements.
constexpr int64_t kStageBudget = int64_t(1) << 30;
// cb_compact with K rotated from sender position idx[j] to receiver position pos0 + out_off + j.
cudaError_t launch_compact_rope(const CompactBatch& b, double base, int style, int64_t pos0, cudaStream_t st,
                                int num_sms);

}  // namespace cbk
