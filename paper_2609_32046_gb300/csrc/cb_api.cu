// C-ABI of the CacheBack filtering path (declared in include/cacheback.h).
// Host-side validation, scratch ownership and launch plumbing; every step of
// the path itself runs in the kernels of cb_score.cu, cb_select.cu and
// cb_compact.cu.
#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "cacheback.h"
#include "cb_internal.cuh"

namespace cbk {
// Events recorded around each score kernel while stage timing is enabled.  Each mark closes
// the interval that started at the previous mark; intervals are summed per stage on read.
struct StageTimer {
    std::vector<cudaEvent_t> pool;                 // created once, reused after each read
    std::vector<std::pair<int, cudaEvent_t>> marks;
    size_t used = 0;
    int calls = 0;
    int mode = 1;   // 1: every stage; 2: the second logit pass only (two events a launch)
    ~StageTimer() {
        for (cudaEvent_t e : pool) cudaEventDestroy(e);
    }
};

void stage_mark(StageTimer* t, int stage, cudaStream_t st) {
    if (!t) return;
    if (t->mode == 2 && stage != kStageCombine && stage != kStageAccum) return;   // brackets pass 2 only
    if (t->used == t->pool.size()) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) { cudaGetLastError(); return; }
        t->pool.push_back(e);
    }
    cudaEvent_t e = t->pool[t->used++];
    // inside a stream capture the mark must become a graph node that records on every replay
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cap) != cudaSuccess) cudaGetLastError();
    const cudaError_t r = cap == cudaStreamCaptureStatusActive
                              ? cudaEventRecordWithFlags(e, st, cudaEventRecordExternal)
                              : cudaEventRecord(e, st);
    if (r != cudaSuccess) { cudaGetLastError(); return; }
    t->marks.emplace_back(stage, e);   // one call may hold several sender batches: cb_score counts calls
}
}  // namespace cbk

constexpr int64_t kDefaultWaitNs = 1000000000;   // 1 s

struct cb_ctx {
    cb_config cfg;
    int device = 0;
    int num_sms = 0;
    int G = 1;
    bool use_tc = false;
    float scale = 0.f;
    int64_t n_chunk1_max = 0;
    float2* stats = nullptr;
    float* offs = nullptr;
    uint16_t* ext = nullptr;        // tcgen05 passes: per-row offset terms [S][nS][R_pad][16] bf16
    uint16_t* ones = nullptr;       // tcgen05 passes: [128][16] bf16 block of ones columns
    float* part = nullptr;
    float* span_keys = nullptr;
    uint16_t* stage = nullptr;      // tcgen05 passes: contiguous copies of paged senders' K (on demand)
    int64_t stage_elems = 0;
    uint32_t* err = nullptr;
    int64_t keys_per_sender = 0;
    int64_t scratch_bytes = 0;
    int32_t score_path = 0;         // kernels of the last cb_score: 2 tcgen05, 1 mma.sync, 0 none yet
    int64_t wait_ns = kDefaultWaitNs;   // limit of one bounded device wait (tcgen05 passes)
    int32_t stall_next = 0;         // failure-detection test: stall the next cb_score once
    int32_t score_sms = 0;          // SMs of the persistent score kernels (0: all)
    cbk::StageTimer* timer = nullptr;
    std::string last_error;
};

namespace {

thread_local std::string g_create_error;

cb_status fail(cb_ctx* ctx, cb_status st, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (ctx)
        ctx->last_error = buf;
    else
        g_create_error = buf;
    return st;
}

// Makes ctx's device current for the duration of a call, restoring the caller's device after.
struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) { ok = false; return; }
        if (prev != dev && cudaSetDevice(dev) != cudaSuccess) ok = false;
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};


// The pointer must be device (or managed) memory on ctx's device.
cb_status check_device_ptr(cb_ctx* ctx, const void* p, const char* what, int i, int align = 16) {
    if (!p) return fail(ctx, CB_EINVAL, "%s[%d] is NULL", what, i);
    if (reinterpret_cast<uintptr_t>(p) % (uintptr_t)align != 0)
        return fail(ctx, CB_EINVAL, "%s[%d] is not %d-byte aligned", what, i, align);
    cudaPointerAttributes a;
    cudaError_t e = cudaPointerGetAttributes(&a, p);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(ctx, CB_EINVAL, "%s[%d]: cannot query pointer (%s)", what, i, cudaGetErrorString(e));
    }
    if (a.type == cudaMemoryTypeManaged) return CB_OK;
    if (a.type != cudaMemoryTypeDevice)
        return fail(ctx, CB_EINVAL, "%s[%d] is not device memory", what, i);
    if (a.device != ctx->device)
        return fail(ctx, CB_EINVAL, "%s[%d] lives on device %d, context on device %d", what, i, a.device,
                    ctx->device);
    return CB_OK;
}

// A row source the kernels may read across the host link: device memory, or pinned host memory
// mapped into the device's address space (cudaHostAlloc / cudaHostRegister).  *dev receives the
// address to use on the device.
cb_status check_source_ptr(cb_ctx* ctx, const void* p, const char* what, int i, int align, const void** dev) {
    if (!p) return fail(ctx, CB_EINVAL, "%s[%d] is NULL", what, i);
    if (reinterpret_cast<uintptr_t>(p) % (uintptr_t)align != 0)
        return fail(ctx, CB_EINVAL, "%s[%d] is not %d-byte aligned", what, i, align);
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return fail(ctx, CB_EINVAL, "%s[%d]: cannot query pointer", what, i);
    }
    if (a.type == cudaMemoryTypeHost) {
        void* d = nullptr;
        if (cudaHostGetDevicePointer(&d, const_cast<void*>(p), 0) != cudaSuccess || !d) {
            cudaGetLastError();
            return fail(ctx, CB_EINVAL, "%s[%d] is pinned host memory not mapped into the device", what, i);
        }
        if (reinterpret_cast<uintptr_t>(d) % (uintptr_t)align != 0)
            return fail(ctx, CB_EINVAL, "%s[%d]: device mapping is not %d-byte aligned", what, i, align);
        *dev = d;
        return CB_OK;
    }
    cb_status st = check_device_ptr(ctx, p, what, i, align);
    if (st == CB_OK) *dev = p;
    return st;
}

bool stride_ok(int64_t s) { return s > 0 && (s % 8) == 0; }

// The optional block table of a sender (paged layout).
cb_status check_pages(cb_ctx* ctx, const cb_kv& s, int i) {
    if (!s.pages) return CB_OK;
    if (s.page_size < 1 || s.page_size > 65536 || (s.page_size & (s.page_size - 1)) != 0)
        return fail(ctx, CB_EINVAL, "senders[%d].page_size = %d is not a power of two in [1, 65536]", i,
                    s.page_size);
    if (!stride_ok(s.s_page)) return fail(ctx, CB_EINVAL, "senders[%d].s_page must be a positive multiple of 8", i);
    if (s.n_pages < 1) return fail(ctx, CB_EINVAL, "senders[%d].n_pages must be at least 1", i);
    return check_device_ptr(ctx, s.pages, "senders.pages", i, 4);
}

cbk::PageMap page_map(const cb_kv& s) {
    cbk::PageMap pm{};
    if (s.pages) {
        pm.pages = s.pages;
        pm.s_page = s.s_page;
        pm.n_pages = s.n_pages;
        int sh = 0;
        while ((1 << sh) < s.page_size) ++sh;
        pm.shift = sh;
    }
    return pm;
}

template <typename T>
cudaError_t alloc(T** p, size_t count, int64_t* total) {
    if (count == 0) count = 1;
    *total += (int64_t)(count * sizeof(T));
    return cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T));
}

}  // namespace

namespace cbk {
// Error text of entry points that take no context (read back by cb_last_error(NULL)).
void set_context_free_error(const char* msg) { g_create_error = msg; }
}  // namespace cbk

extern "C" {

void cb_config_init(cb_config* cfg) {
    if (!cfg) return;
    std::memset(cfg, 0, sizeof *cfg);
    cfg->softmax_scale = 0.f;
    cfg->p = 2.f;
    cfg->alpha = 2.f;
    cfg->pool_width = 7;
    cfg->span_width = 16;
    cfg->n_sink = 1;
    cfg->n_latent = 40;
    cfg->max_senders = 1;
    cfg->score_kernel = 0;
}

int64_t cb_budget(int64_t T, double keep) {
    if (T <= 0 || !(keep > 0.0)) return 0;
    const double b = std::ceil(keep * (double)T);
    if (b >= (double)T) return T;
    return (int64_t)b;
}

int64_t cb_chain_budget(int64_t T_old, int64_t T_new, double keep, int32_t mode, int64_t B_max) {
    if (T_old < 0 || T_new < 0) return -1;
    const int64_t T = T_old + T_new;
    int64_t B;
    if (mode == 0) B = T_old + cb_budget(T_new, keep);
    else if (mode == 1 && B_max >= 0) B = B_max < T ? B_max : T;
    else return -1;
    return B < 0 ? 0 : (B > T ? T : B);
}

const char* cb_last_error(const cb_ctx* ctx) { return ctx ? ctx->last_error.c_str() : g_create_error.c_str(); }

int64_t cb_scratch_bytes(const cb_ctx* ctx) { return ctx ? ctx->scratch_bytes : 0; }

int32_t cb_score_path(const cb_ctx* ctx) { return ctx ? ctx->score_path : 0; }

cb_status cb_create(const cb_config* cfg, cb_ctx** out) {
    if (!out) return fail(nullptr, CB_EINVAL, "out is NULL");
    *out = nullptr;
    if (!cfg) return fail(nullptr, CB_EINVAL, "cfg is NULL");
    const cb_config& c = *cfg;
    if (c.n_layers < 1 || c.n_q_heads < 1 || c.n_kv_heads < 1)
        return fail(nullptr, CB_ESHAPE, "n_layers, n_q_heads and n_kv_heads must be >= 1");
    if (c.n_q_heads % c.n_kv_heads)
        return fail(nullptr, CB_ESHAPE, "n_q_heads (%d) is not a multiple of n_kv_heads (%d)", c.n_q_heads,
                    c.n_kv_heads);
    const int G = c.n_q_heads / c.n_kv_heads;
    if (G != 1 && G != 2 && G != 4) return fail(nullptr, CB_ESHAPE, "group size G = %d not in {1, 2, 4}", G);
    if (c.head_dim != 64 && c.head_dim != 128)
        return fail(nullptr, CB_ESHAPE, "head_dim %d not in {64, 128}", c.head_dim);
    if (c.max_query_tokens < 1 || c.max_query_tokens > cbk::kMaxQueryTokens)
        return fail(nullptr, CB_ESHAPE, "max_query_tokens %d not in [1, %d]", c.max_query_tokens,
                    cbk::kMaxQueryTokens);
    if (c.max_positions < 1 || c.max_positions > INT32_MAX)
        return fail(nullptr, CB_ESHAPE, "max_positions must be in [1, 2^31)");
    if (c.max_senders < 1 || c.max_senders > 4096)
        return fail(nullptr, CB_ESHAPE, "max_senders %d not in [1, 4096]", c.max_senders);
    if (!((std::isfinite(c.p) && c.p > 1.f) || (std::isinf(c.p) && c.p > 0.f)))
        return fail(nullptr, CB_EINVAL, "p must be > 1 (or +infinity)");
    if (!(std::isfinite(c.alpha) && c.alpha >= 0.f)) return fail(nullptr, CB_EINVAL, "alpha must be finite and >= 0");
    if (!(std::isfinite(c.softmax_scale) && c.softmax_scale >= 0.f))
        return fail(nullptr, CB_EINVAL, "softmax_scale must be finite and >= 0");
    if (c.pool_width < 1 || c.pool_width > cbk::kMaxPoolWidth || (c.pool_width % 2) == 0)
        return fail(nullptr, CB_EINVAL, "pool_width %d must be odd and in [1, %d]", c.pool_width,
                    cbk::kMaxPoolWidth);
    if (c.span_width < 1 || c.span_width > cbk::kMaxSpanWidth)
        return fail(nullptr, CB_EINVAL, "span_width %d not in [1, %d]", c.span_width, cbk::kMaxSpanWidth);
    if (c.n_sink < 0 || c.n_latent < 0) return fail(nullptr, CB_EINVAL, "n_sink and n_latent must be >= 0");
    if (c.score_kernel < 0 || c.score_kernel > 2) return fail(nullptr, CB_EINVAL, "score_kernel must be 0, 1 or 2");
    const bool tc_ok = cbk::tc_path_supported(c.head_dim, G, c.pool_width / 2, c.max_query_tokens);
    if (c.score_kernel == 2 && !tc_ok)
        return fail(nullptr, CB_ESHAPE, "tcgen05 score passes need head_dim 128, pool_width <= 7 and "
                    "max_query_tokens * G <= 512");

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(nullptr, CB_ECUDA, "no CUDA device: %s", cudaGetErrorString(e));
    cb_ctx* ctx = new cb_ctx();
    ctx->cfg = c;
    ctx->device = dev;
    ctx->G = G;
    ctx->use_tc = c.score_kernel == 2 || (c.score_kernel == 0 && tc_ok);
    ctx->scale = c.softmax_scale > 0.f ? c.softmax_scale : 1.f / std::sqrt((float)c.head_dim);
    cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, dev);

    const int64_t nS = (int64_t)c.n_layers * c.n_kv_heads;
    const int64_t S = c.max_senders;
    ctx->n_chunk1_max = cbk::stats_slots(c.max_positions);
    const int64_t rows = (int64_t)c.max_query_tokens * G;
    ctx->keys_per_sender = (c.max_positions + c.span_width - 1) / c.span_width;
    int64_t total = 0;
    e = alloc(&ctx->stats, (size_t)(S * nS * ctx->n_chunk1_max * rows), &total);
    if (e == cudaSuccess) e = alloc(&ctx->offs, (size_t)(S * nS * rows), &total);
    if (e == cudaSuccess) e = alloc(&ctx->part, (size_t)(S * 3 * nS * c.max_positions), &total);
    if (e == cudaSuccess) e = alloc(&ctx->span_keys, (size_t)(S * ctx->keys_per_sender), &total);
    if (e == cudaSuccess && ctx->use_tc) {
        e = alloc(&ctx->ext, (size_t)(S * nS * cbk::rows_pad128(rows) * cbk::kExtCols), &total);
        if (e == cudaSuccess) e = alloc(&ctx->ones, (size_t)(128 * cbk::kExtCols), &total);
        if (e == cudaSuccess) {
            std::vector<uint16_t> h(128 * cbk::kExtCols, 0);
            for (int r = 0; r < 128; ++r)
                for (int k = 0; k < 3; ++k) h[r * cbk::kExtCols + k] = 0x3F80;   // bf16 1.0
            e = cudaMemcpy(ctx->ones, h.data(), h.size() * sizeof(uint16_t), cudaMemcpyHostToDevice);
        }
    }
    if (e == cudaSuccess) e = alloc(&ctx->err, 1, &total);
    if (e == cudaSuccess) e = cudaMemset(ctx->err, 0, sizeof(uint32_t));
    ctx->scratch_bytes = total;
    if (e != cudaSuccess) {
        cudaGetLastError();
        cb_destroy(ctx);
        return fail(nullptr, CB_ENOMEM, "scratch allocation of %lld bytes failed: %s", (long long)total,
                    cudaGetErrorString(e));
    }
    *out = ctx;
    return CB_OK;
}

void cb_destroy(cb_ctx* ctx) {
    if (!ctx) return;
    {
        DeviceGuard dg(ctx->device);
        cudaDeviceSynchronize();
        cudaFree(ctx->stats);
        cudaFree(ctx->offs);
        cudaFree(ctx->ext);
        cudaFree(ctx->ones);
        cudaFree(ctx->part);
        cudaFree(ctx->span_keys);
        cudaFree(ctx->stage);
        cudaFree(ctx->err);
        delete ctx->timer;
    }
    delete ctx;
}

namespace {
// An NVTX range over one call of the C-ABI (header-only NVTX: free unless a profiler listens).
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};
}  // namespace

cb_status cb_score(cb_ctx* ctx, int32_t n, const cb_kv* senders, const cb_query* queries, float* const* scores,
                   void* stream) {
    NvtxRange nr("cb_score");
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    ctx->last_error.clear();
    const cb_config& c = ctx->cfg;
    if (n < 1 || n > c.max_senders) return fail(ctx, CB_ESHAPE, "n = %d not in [1, %d]", n, c.max_senders);
    if (!senders || !queries || !scores) return fail(ctx, CB_EINVAL, "senders, queries or scores is NULL");
    DeviceGuard dg(ctx->device);
    if (!dg.ok) return fail(ctx, CB_ECUDA, "cannot select device %d", ctx->device);
    for (int i = 0; i < n; ++i) {
        const cb_kv& s = senders[i];
        const cb_query& q = queries[i];
        if (s.T < 1 || s.T > c.max_positions)
            return fail(ctx, CB_ESHAPE, "senders[%d].T = %lld not in [1, %lld]", i, (long long)s.T,
                        (long long)c.max_positions);
        if (q.m < 1 || q.m > c.max_query_tokens)
            return fail(ctx, CB_ESHAPE, "queries[%d].m = %d not in [1, %d]", i, q.m, c.max_query_tokens);
        if (!stride_ok(s.s_layer) || !stride_ok(s.s_head) || !stride_ok(s.s_pos) || s.s_pos < c.head_dim)
            return fail(ctx, CB_EINVAL, "senders[%d]: strides must be positive multiples of 8 (s_pos >= d)", i);
        if (!stride_ok(q.s_layer) || !stride_ok(q.s_tok) || !stride_ok(q.s_head) || q.s_head < c.head_dim)
            return fail(ctx, CB_EINVAL, "queries[%d]: strides must be positive multiples of 8 (s_head >= d)", i);
        cb_status st;
        if ((st = check_device_ptr(ctx, s.k, "senders.k", i))) return st;
        if ((st = check_pages(ctx, s, i))) return st;
        if ((st = check_device_ptr(ctx, q.q, "queries.q", i))) return st;
        if (q.k_self) {
            if (!stride_ok(q.ks_layer) || !stride_ok(q.ks_tok) || !stride_ok(q.ks_head) || q.ks_head < c.head_dim)
                return fail(ctx, CB_EINVAL, "queries[%d]: k_self strides must be positive multiples of 8 "
                            "(ks_head >= d)", i);
            if ((st = check_device_ptr(ctx, q.k_self, "queries.k_self", i))) return st;
        }
        if ((st = check_device_ptr(ctx, scores[i], "scores", i))) return st;
    }
    cudaStream_t strm = reinterpret_cast<cudaStream_t>(stream);
    const int nS = c.n_layers * c.n_kv_heads;
    if (ctx->use_tc) {
        // paged senders are copied into a contiguous staging buffer for the tensor-map passes:
        // room for the largest one, and for the rest up to kStageBudget elements per sub-batch
        int64_t largest = 0, sum = 0;
        for (int i = 0; i < n; ++i)
            if (senders[i].pages) {
                const int64_t e = (int64_t)nS * senders[i].T * c.head_dim;
                largest = e > largest ? e : largest;
                sum += e;
            }
        const int64_t want = largest > (sum < cbk::kStageBudget ? sum : cbk::kStageBudget)
                                 ? largest : (sum < cbk::kStageBudget ? sum : cbk::kStageBudget);
        if (want > ctx->stage_elems) {
            cudaFree(ctx->stage);   // waits for work still using it
            ctx->scratch_bytes -= ctx->stage_elems * 2;
            ctx->stage = nullptr;
            ctx->stage_elems = 0;
            if (cudaMalloc(reinterpret_cast<void**>(&ctx->stage), (size_t)want * 2) != cudaSuccess) {
                cudaGetLastError();
                ctx->stage = nullptr;
                return fail(ctx, CB_ENOMEM, "cannot allocate %lld bytes to stage paged caches", (long long)want * 2);
            }
            ctx->stage_elems = want;
            ctx->scratch_bytes += want * 2;
        }
    }
    for (int b0 = 0; b0 < n; b0 += cbk::kMaxBatch) {
        const int nb = n - b0 < cbk::kMaxBatch ? n - b0 : cbk::kMaxBatch;
        cbk::ScoreBatch* bt = new cbk::ScoreBatch();
        bt->n = nb;
        bt->n_layers = c.n_layers;
        bt->n_q_heads = c.n_q_heads;
        bt->n_kv_heads = c.n_kv_heads;
        bt->head_dim = c.head_dim;
        bt->scale_log2e = ctx->scale * 1.4426950408889634f;
        bt->p = c.p;
        bt->p_inf = std::isinf(c.p) ? 1 : 0;
        bt->alpha = c.alpha;
        bt->pool_half = c.pool_width / 2;
        bt->use_tc = ctx->use_tc ? 1 : 0;
        bt->timer = ctx->timer;
        bt->err = ctx->err;
        bt->stats = ctx->stats;
        bt->offs = ctx->offs;
        bt->ext = ctx->use_tc ? ctx->ext : nullptr;
        bt->ones = ctx->ones;
        bt->part = ctx->part;
        bt->stage = ctx->stage;
        bt->stage_elems = ctx->stage_elems;
        bt->wait_ns = (uint64_t)ctx->wait_ns;
        bt->stall = b0 == 0 ? ctx->stall_next : 0;
        int64_t so = 0, oo = 0, eo = 0, po = 0, b1 = 0, b2 = 0;
        for (int k = 0; k < nb; ++k) {
            const cb_kv& s = senders[b0 + k];
            const cb_query& q = queries[b0 + k];
            cbk::ScoreSender& d = bt->s[k];
            d.k = static_cast<const uint16_t*>(s.k);
            d.q = static_cast<const uint16_t*>(q.q);
            d.scores = scores[b0 + k];
            d.T = s.T;
            d.ks_l = s.s_layer; d.ks_h = s.s_head; d.ks_p = s.s_pos;
            d.pm = page_map(s);
            d.qs_l = q.s_layer; d.qs_t = q.s_tok; d.qs_h = q.s_head;
            d.kself = static_cast<const uint16_t*>(q.k_self);
            d.kss_l = q.ks_layer; d.kss_t = q.ks_tok; d.kss_h = q.ks_head;
            d.m = q.m;
            d.n_chunk1 = (int32_t)((s.T + cbk::kStatsChunk - 1) / cbk::kStatsChunk);
            d.n_chunk2 = (int32_t)((s.T + cbk::kAccumChunk - 1) / cbk::kAccumChunk);
            d.stats_off = so; so += (int64_t)nS * cbk::stats_slots(s.T) * q.m * ctx->G;
            d.offs_off = oo; oo += (int64_t)nS * q.m * ctx->G;
            d.ext_off = eo; eo += (int64_t)nS * cbk::rows_pad128((int64_t)q.m * ctx->G) * cbk::kExtCols;
            d.part_off = po; po += (int64_t)3 * nS * s.T;
            d.blk1_begin = b1; b1 += (int64_t)nS * d.n_chunk1;
            d.blk2_begin = b2; b2 += (int64_t)nS * d.n_chunk2;
        }
        int path = 0;
        const int sms = ctx->score_sms > 0 && ctx->score_sms < ctx->num_sms ? ctx->score_sms : ctx->num_sms;
        cudaError_t e = cbk::launch_score(*bt, strm, sms, &path);
        ctx->score_path = path;
        delete bt;
        if (e != cudaSuccess) return fail(ctx, CB_ECUDA, "score launch failed: %s", cudaGetErrorString(e));
    }
    ctx->stall_next = 0;
    if (ctx->timer) ++ctx->timer->calls;
    return CB_OK;
}

cb_status cb_set_wait_limit(cb_ctx* ctx, int64_t limit_ns, int32_t stall_next_score) {
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    ctx->last_error.clear();
    if (limit_ns != 0 && (limit_ns < 1000 || limit_ns > 60000000000ll))
        return fail(ctx, CB_EINVAL, "limit_ns = %lld: 0 (the default, 1 s) or 1e3 .. 6e10", (long long)limit_ns);
    if (stall_next_score != 0 && stall_next_score != 1)
        return fail(ctx, CB_EINVAL, "stall_next_score must be 0 or 1");
    ctx->wait_ns = limit_ns ? limit_ns : kDefaultWaitNs;
    ctx->stall_next = stall_next_score;
    return CB_OK;
}

cb_status cb_set_score_sms(cb_ctx* ctx, int32_t n_sms) {
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    ctx->last_error.clear();
    if (n_sms < 0) return fail(ctx, CB_EINVAL, "n_sms = %d must be >= 0", n_sms);
    ctx->score_sms = n_sms;
    return CB_OK;
}

cb_status cb_select(cb_ctx* ctx, int32_t n, const float* const* scores, const int64_t* T, const int64_t* budget,
                    int32_t* const* idx, void* stream) {
    NvtxRange nr("cb_select");
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    ctx->last_error.clear();
    const cb_config& c = ctx->cfg;
    if (n < 1 || n > c.max_senders) return fail(ctx, CB_ESHAPE, "n = %d not in [1, %d]", n, c.max_senders);
    if (!scores || !T || !budget || !idx) return fail(ctx, CB_EINVAL, "scores, T, budget or idx is NULL");
    DeviceGuard dg(ctx->device);
    if (!dg.ok) return fail(ctx, CB_ECUDA, "cannot select device %d", ctx->device);
    for (int i = 0; i < n; ++i) {
        if (T[i] < 1 || T[i] > c.max_positions)
            return fail(ctx, CB_ESHAPE, "T[%d] = %lld not in [1, %lld]", i, (long long)T[i], (long long)c.max_positions);
        const int64_t a = c.n_sink < T[i] ? c.n_sink : T[i];
        const int64_t b = T[i] - c.n_latent > 0 ? T[i] - c.n_latent : 0;
        const int64_t forced = a >= b ? T[i] : a + (T[i] - b);
        if (budget[i] < forced || budget[i] > T[i])
            return fail(ctx, CB_EBUDGET, "budget[%d] = %lld outside [%lld, %lld] (forced positions count toward it)",
                        i, (long long)budget[i], (long long)forced, (long long)T[i]);
        cb_status st;
        if ((st = check_device_ptr(ctx, scores[i], "scores", i))) return st;
        if ((st = check_device_ptr(ctx, idx[i], "idx", i))) return st;
    }
    cudaStream_t strm = reinterpret_cast<cudaStream_t>(stream);
    for (int b0 = 0; b0 < n; b0 += cbk::kMaxBatch) {
        const int nb = n - b0 < cbk::kMaxBatch ? n - b0 : cbk::kMaxBatch;
        cbk::SelectBatch bt;
        std::memset(&bt, 0, sizeof bt);
        bt.n = nb;
        bt.n_sink = c.n_sink;
        bt.n_latent = c.n_latent;
        bt.span_w = c.span_width;
        bt.err = ctx->err;
        for (int k = 0; k < nb; ++k) {
            bt.s[k].scores = scores[b0 + k];
            bt.s[k].idx = idx[b0 + k];
            bt.s[k].T = T[b0 + k];
            bt.s[k].B = budget[b0 + k];
            bt.s[k].span_keys = ctx->span_keys + (int64_t)k * ctx->keys_per_sender;
        }
        cudaError_t e = cbk::launch_select(bt, strm);
        if (e != cudaSuccess) return fail(ctx, CB_ECUDA, "select launch failed: %s", cudaGetErrorString(e));
    }
    return CB_OK;
}

}  // extern "C"

namespace {

// Rotary re-index of cb_compact_rope (null for cb_compact).
struct RopeArgs {
    double base;
    int32_t style;
    int64_t pos0;
};

// Shared body of cb_compact and cb_compact_rope: validation, batching, launch.
cb_status compact_impl(cb_ctx* ctx, int32_t n, const cb_kv* senders, const int32_t* const* idx,
                       const int64_t* budget, void* k_out, void* v_out, int64_t out_capacity,
                       const int64_t* out_offset, int64_t o_layer, int64_t o_head, const RopeArgs* rope,
                       void* stream) {
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    ctx->last_error.clear();
    const cb_config& c = ctx->cfg;
    if (n < 1 || n > c.max_senders) return fail(ctx, CB_ESHAPE, "n = %d not in [1, %d]", n, c.max_senders);
    if (!senders || !idx || !budget || !out_offset) return fail(ctx, CB_EINVAL, "senders, idx, budget or out_offset is NULL");
    if (out_capacity < 0) return fail(ctx, CB_EINVAL, "out_capacity < 0");
    if (!stride_ok(o_head) || !stride_ok(o_layer) || o_head < out_capacity * c.head_dim ||
        o_layer < (int64_t)c.n_kv_heads * o_head)
        return fail(ctx, CB_EINVAL, "output strides must be multiples of 8 and not overlap rows");
    if (rope && (!(rope->base > 1.0) || !std::isfinite(rope->base) || (rope->style != 0 && rope->style != 1)))
        return fail(ctx, CB_EINVAL, "rope_base must be finite and > 1, rope_style 0 or 1");
    DeviceGuard dg(ctx->device);
    if (!dg.ok) return fail(ctx, CB_ECUDA, "cannot select device %d", ctx->device);
    cb_status st;
    if ((st = check_device_ptr(ctx, k_out, "k_out", 0))) return st;
    if ((st = check_device_ptr(ctx, v_out, "v_out", 0))) return st;
    std::vector<const void*> kdev(n), vdev(n);
    for (int i = 0; i < n; ++i) {
        const cb_kv& s = senders[i];
        if (s.T < 1 || s.T > c.max_positions)
            return fail(ctx, CB_ESHAPE, "senders[%d].T = %lld not in [1, %lld]", i, (long long)s.T,
                        (long long)c.max_positions);
        if (budget[i] < 0 || budget[i] > s.T)
            return fail(ctx, CB_EBUDGET, "budget[%d] = %lld not in [0, T]", i, (long long)budget[i]);
        if (out_offset[i] < 0 || out_offset[i] + budget[i] > out_capacity)
            return fail(ctx, CB_EBUDGET, "sender %d: rows [%lld, %lld) exceed out_capacity %lld", i,
                        (long long)out_offset[i], (long long)(out_offset[i] + budget[i]), (long long)out_capacity);
        if ((int64_t)2 * c.n_layers * c.n_kv_heads * budget[i] * (c.head_dim / 8) >= ((int64_t)1 << 31))
            return fail(ctx, CB_ESHAPE, "sender %d: too many rows for one launch", i);
        if (!stride_ok(s.s_layer) || !stride_ok(s.s_head) || !stride_ok(s.s_pos) || s.s_pos < c.head_dim)
            return fail(ctx, CB_EINVAL, "senders[%d]: strides must be positive multiples of 8 (s_pos >= d)", i);
        // K and V rows may come from mapped pinned host memory (only the selected rows cross the link)
        if ((st = check_source_ptr(ctx, s.k, "senders.k", i, 16, &kdev[i]))) return st;
        if ((st = check_source_ptr(ctx, s.v, "senders.v", i, 16, &vdev[i]))) return st;
        if ((st = check_pages(ctx, s, i))) return st;
        if (budget[i] > 0 && (st = check_device_ptr(ctx, idx[i], "idx", i))) return st;
    }
    cudaStream_t strm = reinterpret_cast<cudaStream_t>(stream);
    for (int b0 = 0; b0 < n; b0 += cbk::kMaxBatch) {
        const int nb = n - b0 < cbk::kMaxBatch ? n - b0 : cbk::kMaxBatch;
        cbk::CompactBatch bt;
        std::memset(&bt, 0, sizeof bt);
        bt.n = nb;
        bt.n_layers = c.n_layers;
        bt.n_kv_heads = c.n_kv_heads;
        bt.head_dim = c.head_dim;
        bt.k_out = static_cast<uint16_t*>(k_out);
        bt.v_out = static_cast<uint16_t*>(v_out);
        bt.o_layer = o_layer;
        bt.o_head = o_head;
        bt.err = ctx->err;
        for (int k = 0; k < nb; ++k) {
            const cb_kv& s = senders[b0 + k];
            cbk::CompactSender& d = bt.s[k];
            d.k = static_cast<const uint16_t*>(kdev[b0 + k]);
            d.v = static_cast<const uint16_t*>(vdev[b0 + k]);
            d.idx = idx[b0 + k];
            d.T = s.T;
            d.ks_l = s.s_layer; d.ks_h = s.s_head; d.ks_p = s.s_pos;
            d.pm = page_map(s);
            d.B = budget[b0 + k];
            d.out_off = out_offset[b0 + k];
        }
        cudaError_t e = rope ? cbk::launch_compact_rope(bt, rope->base, rope->style, rope->pos0, strm, ctx->num_sms)
                             : cbk::launch_compact(bt, strm, ctx->num_sms);
        if (e != cudaSuccess) return fail(ctx, CB_ECUDA, "compact launch failed: %s", cudaGetErrorString(e));
    }
    return CB_OK;
}

}  // namespace

extern "C" {

cb_status cb_compact(cb_ctx* ctx, int32_t n, const cb_kv* senders, const int32_t* const* idx, const int64_t* budget,
                     void* k_out, void* v_out, int64_t out_capacity, const int64_t* out_offset, int64_t o_layer,
                     int64_t o_head, void* stream) {
    NvtxRange nr("cb_compact");
    return compact_impl(ctx, n, senders, idx, budget, k_out, v_out, out_capacity, out_offset, o_layer, o_head,
                        nullptr, stream);
}

cb_status cb_compact_rope(cb_ctx* ctx, int32_t n, const cb_kv* senders, const int32_t* const* idx,
                          const int64_t* budget, void* k_out, void* v_out, int64_t out_capacity,
                          const int64_t* out_offset, int64_t o_layer, int64_t o_head, double rope_base,
                          int32_t rope_style, int64_t pos0, void* stream) {
    NvtxRange nr("cb_compact_rope");
    const RopeArgs r{rope_base, rope_style, pos0};
    return compact_impl(ctx, n, senders, idx, budget, k_out, v_out, out_capacity, out_offset, o_layer, o_head, &r,
                        stream);
}

cb_status cb_enable_stage_timing(cb_ctx* ctx, int32_t enable) {
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    DeviceGuard dg(ctx->device);
    if (enable < 0 || enable > 2) return fail(ctx, CB_EINVAL, "enable = %d not in {0, 1, 2}", enable);
    if (enable && !ctx->timer) ctx->timer = new cbk::StageTimer();
    if (enable) ctx->timer->mode = enable;
    if (!enable && ctx->timer) {
        cudaDeviceSynchronize();
        delete ctx->timer;
        ctx->timer = nullptr;
    }
    return CB_OK;
}

cb_status cb_stage_times(cb_ctx* ctx, float* ms, int32_t* calls) {
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    if (!ms || !calls) return fail(ctx, CB_EINVAL, "ms or calls is NULL");
    for (int k = 0; k < 4; ++k) ms[k] = 0.f;
    *calls = 0;
    cbk::StageTimer* t = ctx->timer;
    if (!t) return fail(ctx, CB_EINVAL, "stage timing is not enabled");
    DeviceGuard dg(ctx->device);
    if (!t->marks.empty()) {
        cudaError_t e = cudaEventSynchronize(t->marks.back().second);
        if (e != cudaSuccess) return fail(ctx, CB_ECUDA, "event wait failed: %s", cudaGetErrorString(e));
        for (size_t i = 1; i < t->marks.size(); ++i) {
            const int stage = t->marks[i].first;
            if (stage == cbk::kStageStart) continue;
            if (t->mode == 2 && stage != cbk::kStageAccum) continue;
            float x = 0.f;
            if (cudaEventElapsedTime(&x, t->marks[i - 1].second, t->marks[i].second) == cudaSuccess)
                ms[stage - 1] += x;
            else
                cudaGetLastError();
        }
    }
    *calls = t->calls;
    t->marks.clear();
    t->used = 0;
    t->calls = 0;
    return CB_OK;
}

cb_status cb_gather(cb_ctx* ctx, int32_t n, const void* const* src, const int64_t* T, int64_t src_stride,
                    int64_t row_bytes, const int32_t* const* idx, const int64_t* count, void* out,
                    int64_t out_capacity, const int64_t* out_offset, int64_t out_stride, void* stream) {
    NvtxRange nr("cb_gather");
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    ctx->last_error.clear();
    if (n < 1) return fail(ctx, CB_ESHAPE, "n = %d < 1", n);
    if (!src || !T || !idx || !count || !out_offset) return fail(ctx, CB_EINVAL, "src, T, idx, count or out_offset is NULL");
    if (row_bytes <= 0 || row_bytes % 4 != 0) return fail(ctx, CB_EINVAL, "row_bytes %lld must be a positive multiple of 4",
                                                          (long long)row_bytes);
    if (src_stride < row_bytes || src_stride % 4 != 0 || out_stride < row_bytes || out_stride % 4 != 0)
        return fail(ctx, CB_EINVAL, "strides must be multiples of 4 bytes and at least row_bytes");
    if (out_capacity < 0) return fail(ctx, CB_EINVAL, "out_capacity < 0");
    DeviceGuard dg(ctx->device);
    if (!dg.ok) return fail(ctx, CB_ECUDA, "cannot select device %d", ctx->device);
    cb_status st;
    if ((st = check_device_ptr(ctx, out, "out", 0, 4))) return st;
    std::vector<const void*> sdev(n);
    for (int i = 0; i < n; ++i) {
        if (T[i] < 1) return fail(ctx, CB_ESHAPE, "T[%d] = %lld < 1", i, (long long)T[i]);
        if (count[i] < 0) return fail(ctx, CB_EBUDGET, "count[%d] = %lld < 0", i, (long long)count[i]);
        if (out_offset[i] < 0 || out_offset[i] + count[i] > out_capacity)
            return fail(ctx, CB_EBUDGET, "sender %d: rows [%lld, %lld) exceed out_capacity %lld", i,
                        (long long)out_offset[i], (long long)(out_offset[i] + count[i]), (long long)out_capacity);
        if (count[i] * (row_bytes / 4) >= ((int64_t)1 << 40))
            return fail(ctx, CB_ESHAPE, "sender %d: message too large", i);
        if ((st = check_source_ptr(ctx, src[i], "src", i, 4, &sdev[i]))) return st;
        if (count[i] > 0 && (st = check_device_ptr(ctx, idx[i], "idx", i, 4))) return st;
    }
    cudaStream_t strm = reinterpret_cast<cudaStream_t>(stream);
    for (int b0 = 0; b0 < n; b0 += cbk::kMaxBatch) {
        const int nb = n - b0 < cbk::kMaxBatch ? n - b0 : cbk::kMaxBatch;
        cbk::GatherBatch bt;
        std::memset(&bt, 0, sizeof bt);
        bt.n = nb;
        bt.row_bytes = row_bytes;
        bt.out = static_cast<uint8_t*>(out);
        bt.out_stride = out_stride;
        bt.err = ctx->err;
        for (int k = 0; k < nb; ++k) {
            cbk::GatherSender& d = bt.s[k];
            d.src = static_cast<const uint8_t*>(sdev[b0 + k]);
            d.idx = idx[b0 + k];
            d.T = T[b0 + k];
            d.src_stride = src_stride;
            d.count = count[b0 + k];
            d.out_off = out_offset[b0 + k];
        }
        cudaError_t e = cbk::launch_gather(bt, strm, ctx->num_sms);
        if (e != cudaSuccess) return fail(ctx, CB_ECUDA, "gather launch failed: %s", cudaGetErrorString(e));
    }
    return CB_OK;
}

cb_status cb_sync_status(cb_ctx* ctx, void* stream) {
    if (!ctx) return fail(nullptr, CB_EINVAL, "ctx is NULL");
    DeviceGuard dg(ctx->device);
    cudaStream_t strm = reinterpret_cast<cudaStream_t>(stream);
    uint32_t word = 0;
    cudaError_t e = cudaMemcpyAsync(&word, ctx->err, sizeof word, cudaMemcpyDeviceToHost, strm);
    if (e == cudaSuccess) e = cudaStreamSynchronize(strm);
    if (e != cudaSuccess) return fail(ctx, CB_ECUDA, "device error: %s", cudaGetErrorString(e));
    if (word) {
        cudaMemsetAsync(ctx->err, 0, sizeof(uint32_t), strm);
        cudaStreamSynchronize(strm);
        if (word & cbk::kErrTimeout)
            return fail(ctx, CB_ETIMEOUT,
                        "a bounded device wait gave up (code 0x%x: bits 8+ name the wait); the results are invalid",
                        word);
        return fail(ctx, CB_EDEVICE, "kernel bounds check failed (code 0x%x:%s%s%s%s)", word,
                    (word & cbk::kErrCompactIndex) ? " compact index outside [0, T)" : "",
                    (word & cbk::kErrSelectBudget) ? " select count mismatch" : "",
                    (word & cbk::kErrGatherIndex) ? " gather index outside [0, T)" : "",
                    (word & cbk::kErrPageIndex) ? " block-table entry outside [0, n_pages)" : "");
    }
    return CB_OK;
}

}  // extern "C"
