/*
 * cacheback.h -- C-ABI of the GB300 (sm_103a) CacheBack filtering path:
 * score every cached sender position by the attention it receives from the
 * receiver's query, select positions under a keep budget, and gather the
 * selected K/V rows of every layer into one contiguous send buffer.
 *
 * Paper: receiver-conditioned communication with CacheBack.
 *   App. A (formal model): the sender cache M_S = {(K_j^l, V_j^l)}, l = 1..L, j = 1..N.
 *   App. C.1 (general scoring rule): attention a_{l,h,r,t} from the m query tokens,
 *     mean query attention Q_t, the CacheBack correction C_{p,t}, Pool_7.
 *   App. D.2 (parameter sensitivity): S_t(p, alpha) = Q_t * C_{p,t}^alpha
 *     (CacheBack: p = alpha = 2; alpha = 0 is mean query attention).
 *   App. C.2 (budgets and position selection): B_i = ceil(T_i / r), forced
 *     first and latent positions, width-16 span ranking, source-order output.
 *
 * Conventions shared by every entry point
 *   - All data pointers inside descriptors are DEVICE pointers owned by the
 *     caller; arrays of descriptors / pointers / sizes passed directly are HOST
 *     arrays read during the call only.  The library never frees caller memory.
 *   - K, V and Q are bf16 (raw 16-bit storage).  Strides are in ELEMENTS; the
 *     head-dimension stride is 1.  Every device pointer must be 16-byte aligned
 *     and every stride a multiple of 8 elements.
 *   - Calls are asynchronous on the given CUDA stream (a cudaStream_t passed
 *     as void*; NULL is the legacy default stream).  Errors found on the host
 *     are returned synchronously and nothing is enqueued.  cb_last_error()
 *     describes the most recent failure of that context.
 *   - Results are bitwise deterministic: every reduction has a fixed order.
 *   - Query head h reads KV head h / G, G = n_q_heads / n_kv_heads (App. C.1:
 *     query heads that share each KV head).
 *   - A context is not thread-safe: one host thread at a time.  Scratch is
 *     shared by calls on one context, so calls on one context must be ordered
 *     on one stream (or synchronised); use one context per concurrent stream.
 */
#ifndef CACHEBACK_H_
#define CACHEBACK_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CB_OK = 0,
    CB_EINVAL = 1,   /* null / misaligned pointer, bad parameter value */
    CB_ESHAPE = 2,   /* unsupported or inconsistent shape, above a creation limit */
    CB_EBUDGET = 3,  /* budget below the forced positions, above T, or beyond the output capacity */
    CB_ENOMEM = 4,   /* device allocation failed */
    CB_ECUDA = 5,    /* a CUDA runtime call or a kernel launch failed */
    CB_ETIMEOUT = 6, /* a bounded device wait gave up (see cb_set_wait_limit, cb_sync_status) */
    CB_EDEVICE = 7   /* a kernel's own bounds check rejected an input (see cb_sync_status) */
} cb_status;

typedef struct cb_ctx cb_ctx; /* opaque; owns device scratch only */

/*
 * Creation-time configuration (App. C.1 notation).
 *   n_layers           |L|: scored layers only (global-attention layers; App. C.1 skips
 *                      local/sliding layers, App. F lists 8/48 for Gemma, 6/62 for Nemotron)
 *   n_q_heads          Hq, query heads per layer
 *   n_kv_heads         Hkv; Hq % Hkv == 0 and G = Hq / Hkv in {1, 2, 4}
 *   head_dim           d in {64, 128}
 *   max_query_tokens   upper bound on m (1..1024)
 *   max_positions      upper bound on any sender's T (scratch is sized from it)
 *   max_senders        upper bound on senders per call
 *   softmax_scale      logit scale; 0 selects 1/sqrt(d)
 *   p, alpha           correction power p > 1 and strength alpha >= 0 (App. D.2); p = +INFINITY
 *                      takes the limit the parameter-sensitivity study names: C_t = largest pooled
 *                      per-token attention / largest pooled token mean over the groups
 *   pool_width         Pool window, odd, 1..15 (7 in the paper; 1 disables pooling)
 *   span_width         span width for selection, 1..256 (16 in the paper; 1 ranks positions)
 *   n_sink, n_latent   forced positions: the first n_sink and the last n_latent (1 and 40)
 *   score_kernel       0: automatic (tcgen05 tensor-core passes when head_dim = 128,
 *                      pool_width <= 7 and max_query_tokens * G <= 512, else the mma.sync
 *                      passes); 1: mma.sync passes; 2: tcgen05 passes (CB_ESHAPE if unsupported)
 */
typedef struct {
    int32_t n_layers, n_q_heads, n_kv_heads, head_dim;
    int32_t max_query_tokens;
    int64_t max_positions;
    int32_t max_senders;
    float softmax_scale;
    float p, alpha;
    int32_t pool_width;
    int32_t span_width;
    int32_t n_sink, n_latent;
    int32_t score_kernel;
} cb_config;

/* One sender's cache M_S (App. A): K[l][g][t][:] at k + l*s_layer + g*s_head + t*s_pos,
 * V likewise with the same strides.  T = number of cached positions (T_i = H_i + G_i, Sec. 2).
 *
 * Paged layout (optional; App. F: the agents run under vLLM, whose cache lives in fixed-size
 * pages named by a per-sequence block table).  With pages != NULL, position t is row
 * t % page_size of page pages[t / page_size], the same page in every layer and KV head:
 *   K[l][g][t][:] at k + l*s_layer + g*s_head + pages[t / page_size]*s_page + (t % page_size)*s_pos
 * and V likewise (same table, same strides).  vLLM's per-layer [n_pages][page_size][Hkv][d]
 * caches stacked over layers give s_layer = n_pages*page_size*Hkv*d, s_page = page_size*Hkv*d,
 * s_pos = Hkv*d, s_head = d.
 *   pages      device int32[ceil(T / page_size)] (4-byte aligned), read by the kernels; NULL
 *              selects the strided layout and the three fields below are ignored
 *   page_size  rows per page, a power of two in 1..65536
 *   s_page     elements between consecutive pages: a positive multiple of 8
 *   n_pages    pages in the pool; an entry outside [0, n_pages) is never dereferenced: its rows
 *              read as zero (cb_score) or are not written (cb_compact*), and the next
 *              cb_sync_status() reports CB_EDEVICE
 * cb_score, cb_compact and cb_compact_rope take either layout, sender by sender. */
typedef struct {
    const void *k, *v;
    int64_t T;
    int64_t s_layer, s_head, s_pos;
    const int32_t *pages;
    int32_t page_size;
    int64_t s_page, n_pages;
} cb_kv;

/* The receiver query's post-RoPE query vectors in the sender's scored layers (Sec. 3:
 * the sender appends q and computes only the query tokens against its cache):
 * Q[l][r][h][:] at q + l*s_layer + r*s_tok + h*s_head, r < m.  Several senders may share one.
 * k_self (optional, NULL for none): the query tokens' own post-RoPE keys, Ks[l][u][g][:] at
 * k_self + l*ks_layer + u*ks_tok + g*ks_head (u < m, g < Hkv; strides positive multiples of 8).
 * When given, query token r's softmax also runs over the keys of query tokens 0..r, as the
 * appended query attends causally in a real forward pass; the scores still cover the sender
 * positions only, whose attention then sums to less than one.  NULL keeps App. C.1's reading:
 * the softmax over the T sender positions. */
typedef struct {
    const void *q;
    int32_t m;
    int64_t s_layer, s_tok, s_head;
    const void *k_self;
    int64_t ks_layer, ks_tok, ks_head;
} cb_query;

/* Fill *cfg with the paper's defaults (p = alpha = 2, Pool_7, width-16 spans, 1 sink,
 * 40 latent positions, scale 1/sqrt(d)) and zero shapes / limits. */
void cb_config_init(cb_config *cfg);

/* Validate cfg, select the current CUDA device, and allocate the scratch the limits need.
 * On success *out owns the scratch until cb_destroy.  Errors: CB_EINVAL, CB_ESHAPE, CB_ENOMEM,
 * CB_ECUDA (then *out is NULL). */
cb_status cb_create(const cb_config *cfg, cb_ctx **out);

/*
 * Score (App. C.1, App. D.2): for each sender i, write scores[i][t], t < T_i (fp32, device):
 *   S_t = Q_t * C_{p,t}^alpha,
 *   Q_t = Pool( sum_l 1/(m Hq) sum_r sum_h a_{l,h,r,t} ),
 *   C_{p,t} = ( sum_s mean_r Pool(b_{s,r,.})_t^p / sum_s Pool(mean_r b_{s,r,.})_t^p )^(1/(p-1)),
 * a = softmax over the sender's T positions of softmax_scale * <q_{l,r,h}, k_{l,h/G,t}>,
 * b_{s,r,t} = mean of a over the G query heads of KV group s = (l, g); C = 1 where the
 * denominator is 0 (or below FLT_MIN in fp32).  Sender i is scored against queries[i].
 * Entries may repeat one sender cache with different queries: one launch then scores one
 * sender state against many receiver queries (multi-query serving: Sec. 5, Discussion, notes
 * that one completed sender state can be scored for several receiver queries), each pair
 * exactly as if it were scored alone.
 * Paged senders (cb_kv.pages) on the tcgen05 passes are first copied into a contiguous staging
 * buffer of the context (the copy is timed with pass 1).  The first call that needs more room
 * than the buffer has allocates it anew, which waits for the device: make such a call before
 * capturing cb_score in a CUDA graph.  Its size is that of the largest paged cache of the call,
 * or of all of them up to 2 GiB, whichever is larger (senders beyond it are scored in later
 * launches that reuse the buffer).
 *   n         1..max_senders;  senders, queries, scores: host arrays of n entries
 *   scores[i] device float[T_i], written; 16-byte aligned
 * Errors: CB_EINVAL (null/misaligned pointers, strides), CB_ESHAPE (T_i or m_i above the limits),
 * CB_ENOMEM (no room for the staging buffer).
 */
cb_status cb_score(cb_ctx *ctx, int32_t n, const cb_kv *senders, const cb_query *queries,
                   float *const *scores, void *stream);

/* B = ceil(keep * T) computed in double, clamped to [0, T] (App. C.2: B_i = ceil(T_i / r)
 * with keep = 1/r).  Pure host function; needs no context. */
int64_t cb_budget(int64_t T, double keep);

/* Budget of one hop of a sequential chain (App. C.2): the hop's cache holds T_old inherited
 * positions (the previous message) followed by T_new new prompt and latent positions.
 *   mode 0 (relative): B = T_old + ceil(keep * T_new)   (keep = 1/r, ceiling in double)
 *   mode 1 (fixed):    B = min(B_max, T_old + T_new)
 * clamped to [0, T_old + T_new].  Inherited and new positions are then ranked together by
 * cb_select (only the first position and the last n_latent positions are forced).  Returns -1
 * for negative sizes, an unknown mode or a negative B_max.  Pure host function. */
int64_t cb_chain_budget(int64_t T_old, int64_t T_new, double keep, int32_t mode, int64_t B_max);

/*
 * Select (App. C.2): for each sender i, write idx[i][0..budget[i]) (int32, device),
 * strictly ascending, containing the forced positions (the first n_sink and the last
 * n_latent) and filled from spans ranked by mean score after the first position's score
 * is raised to the maximum; equal means favour the earlier span; a span that does not
 * fit contributes its unselected positions nearest its highest-scoring one (ties: lower index).
 * Span means are formed in fp32 in index order and divided by the span's own length.
 *   scores[i]  device float[T[i]] (e.g. cb_score's output)
 *   T, budget  host int64 arrays of n entries; min(T, n_sink + n_latent) <= budget[i] <= T[i]
 *   idx[i]     device int32[budget[i]], written
 * Errors: CB_EINVAL, CB_ESHAPE (T above max_positions), CB_EBUDGET.
 */
cb_status cb_select(cb_ctx *ctx, int32_t n, const float *const *scores, const int64_t *T,
                    const int64_t *budget, int32_t *const *idx, void *stream);

/*
 * Compact (the message of selected positions; Sec. 3 "State Representation", App. C.3):
 * for every sender i, layer l, KV head g and j < budget[i]:
 *   k_out[l*o_layer + g*o_head + (out_offset[i] + j)*d .. +d) = K_i[l][g][idx[i][j]][:]
 * and likewise v_out from V_i -- a bit-exact copy.  Fan-in senders are concatenated by
 * giving each its own out_offset.  out_capacity is the number of position rows per
 * (l, g) in the output; out_offset[i] + budget[i] <= out_capacity is required.
 * Indices outside [0, T_i) are skipped by the kernel and reported as CB_EDEVICE by the
 * next cb_sync_status().
 * K_i and V_i may be device memory or pinned host memory mapped into the device (cudaHostAlloc,
 * cudaHostRegister): the kernel then reads only the selected rows across the host link, e.g. a
 * sender cache kept on the host whose K was copied to the device for cb_score while its V stays
 * put.  Outputs, indices and block tables are device memory.
 * Errors: CB_EINVAL, CB_ESHAPE, CB_EBUDGET (capacity overflow).
 */
cb_status cb_compact(cb_ctx *ctx, int32_t n, const cb_kv *senders, const int32_t *const *idx,
                     const int64_t *budget, void *k_out, void *v_out, int64_t out_capacity,
                     const int64_t *out_offset, int64_t o_layer, int64_t o_head, void *stream);

/*
 * cb_compact with the positional re-index that sending K rows as they are needs (App. C.3: the
 * paper re-prefills the selected rows at their new positions and notes that direct K/V transfer
 * would have to handle the sender/receiver position mismatch).  Arguments as for cb_compact,
 * plus the receiver's rotary embedding: rope_base (> 1; e.g. 1e6 for Qwen3), rope_style 0 for
 * pairs (k, k + d/2) (rotate-half layout) or 1 for pairs (2k, 2k + 1), and pos0, the receiver
 * position of send-buffer row 0.  Row r = out_offset[i] + j of the send buffer takes sender i's
 * position t = idx[i][j] to receiver position pos0 + r: every pair of K's dimensions turns by
 * (pos0 + r - t) * rope_base^(-2k/d) (rounded once to bf16); V is copied unchanged.  Errors as
 * cb_compact, plus CB_EINVAL for a bad rope_base or rope_style.
 */
cb_status cb_compact_rope(cb_ctx *ctx, int32_t n, const cb_kv *senders, const int32_t *const *idx,
                          const int64_t *budget, void *k_out, void *v_out, int64_t out_capacity,
                          const int64_t *out_offset, int64_t o_layer, int64_t o_head, double rope_base,
                          int32_t rope_style, int64_t pos0, void *stream);

/*
 * Message rows by index (Sec. 3.1 "State Representation", App. C.3 "Message encoding").  The
 * continuous-row encoding sends one row of the sender's per-position table (its hidden states:
 * 8 KiB per position for Qwen3-8B) for every selected position; the token-ID encoding sends the
 * selected source positions as token IDs (a table of 4-byte rows) and the latent positions as
 * continuous rows.  Both are this gather, for each sender i:
 *     out row (out_offset[i] + j) = row idx[i][j] of src[i],   j < count[i]
 *   src[i]       table, row t (t < T[i]) at src[i] + t * src_stride bytes: device memory, or
 *                pinned host memory mapped into the device (only the selected rows are read)
 *   row_bytes    bytes per row, a positive multiple of 4 (src_stride, out_stride likewise, >= row_bytes)
 *   idx[i]       device int32 [count[i]] (e.g. cb_select's output or a sub-range of it)
 *   out          device buffer, row r at out + r * out_stride bytes, r < out_capacity
 * Pointers need 4-byte alignment; rows of 16-byte multiples at 16-byte aligned addresses move
 * as 16-byte pieces.  Asynchronous on `stream`; the caller owns every buffer.  Host errors:
 * CB_EINVAL (NULL pointers, bad sizes or strides, unmapped host memory), CB_ESHAPE (n < 1, T < 1),
 * CB_EBUDGET (count < 0 or rows past
 * out_capacity).  An index outside [0, T[i]) skips its row and is reported by cb_sync_status as
 * CB_EDEVICE.
 */
cb_status cb_gather(cb_ctx *ctx, int32_t n, const void *const *src, const int64_t *T, int64_t src_stride,
                    int64_t row_bytes, const int32_t *const *idx, const int64_t *count, void *out,
                    int64_t out_capacity, const int64_t *out_offset, int64_t out_stride, void *stream);

/* Wait for `stream`, then report (and clear) errors the kernels recorded on the device
 * (CB_EDEVICE) or a failed launch (CB_ECUDA).  Blocks the host. */
cb_status cb_sync_status(cb_ctx *ctx, void *stream);

/*
 * Per-kernel timing of cb_score (tracing).  While enabled, every cb_score records CUDA events on
 * its stream between its internal kernels (no synchronisation, a few microseconds of overhead).
 * enable: 0 off, 1 every stage, 2 only the normalised accumulation (two events around each of
 * its launches, the least overhead).  Calls captured into a CUDA graph record their events on
 * every replay; cb_stage_times then reports the latest replay (read it once per replay).
 * cb_stage_times waits for the last recorded event and writes, into ms[0..3], the summed
 * milliseconds since the previous read of the four score kernels: row statistics (first logit
 * pass), statistics combine, normalised accumulation (second logit pass), finalize (0 for the
 * stages not timed); *calls receives the number of cb_score calls covered.  The sums are then
 * reset.  Errors: CB_EINVAL (timing not enabled, NULL arguments, enable outside 0..2), CB_ECUDA.
 */
cb_status cb_enable_stage_timing(cb_ctx *ctx, int32_t enable);
cb_status cb_stage_times(cb_ctx *ctx, float *ms, int32_t *calls);

/*
 * Bounded device waits (failure detection; the paper has no counterpart: this is a runtime
 * control).  Every mbarrier wait of the tcgen05 score passes gives up after limit_ns
 * nanoseconds (default 1 s): the kernel then records which wait gave up, sets an abort flag
 * that every role of its CTA sees, waits (bounded) for its own copies and MMAs in flight,
 * frees its tensor memory and returns, so the context stays usable; the next cb_sync_status
 * reports CB_ETIMEOUT and that call's scores are invalid.
 *   limit_ns          0 restores the default; otherwise 1e3 .. 6e10
 *   stall_next_score  1: the next cb_score that runs the tcgen05 passes makes one wait of its
 *                     first row-statistics launch (CTA 0's MMA issuer) on a barrier nothing
 *                     arrives on, so that wait runs out after limit_ns and the path above is
 *                     taken; cleared by that call.  For tests of failure detection; it faults
 *                     and hangs nothing.  The mma.sync passes have no waits and ignore it.
 * Errors: CB_EINVAL (NULL ctx, values out of range).  Host-only; affects later calls.
 */
cb_status cb_set_wait_limit(cb_ctx *ctx, int64_t limit_ns, int32_t stall_next_score);

/*
 * SMs the score kernels occupy (a runtime control; the paper has no counterpart).  The
 * tcgen05 passes run one persistent CTA per SM on at most n_sms SMs (0, the default: every SM
 * of the device), leaving the other SMs free for work on other streams: a batch's cb_select and
 * cb_compact queued beside the next batch's cb_score run there (their blocks cannot share an SM
 * with a score CTA), so selection and compaction of one wave of senders overlap the scoring of
 * the next.  Scores, indices and messages do not depend on it (every sum keeps its order).
 * The mma.sync passes ignore it.
 * Errors: CB_EINVAL (NULL ctx, n_sms < 0).  Host-only; affects later calls.
 */
cb_status cb_set_score_sms(cb_ctx *ctx, int32_t n_sms);

/* Free the context's scratch (after synchronising its device).  NULL is ignored. */
void cb_destroy(cb_ctx *ctx);

/* Text of the context's most recent error ("" if none).  NULL ctx: the last cb_create failure. */
const char *cb_last_error(const cb_ctx *ctx);

/* Device scratch bytes the context holds now (for capacity planning; grows when cb_score
 * first stages paged caches). */
int64_t cb_scratch_bytes(const cb_ctx *ctx);

/* Which implementation of the two logit passes (App. C.1) the context's last cb_score launched:
 * 2 = tcgen05 (tensor-memory) kernels, 1 = mma.sync kernels, 0 = no cb_score yet or NULL ctx.
 * With score_kernel = 0 or 2 the tcgen05 kernels run unless the driver rejects a tensor map for
 * the given strides; then the mma.sync kernels run instead and this reports 1.  Host-only. */
int32_t cb_score_path(const cb_ctx *ctx);

/*
 * Allocation-free selection.  The paper has no counterpart: this entry point exists
 * for callers that cannot allocate device memory (code running inside a memory pool or
 * arena it does not own, hosts that forbid cudaMalloc after start-up, engines whose
 * allocator is busy or not reentrant at the point of the call), which therefore cannot
 * hold a cb_ctx.  It computes exactly what cb_select computes, with the same kernel,
 * and takes the selection parameters directly instead of from a context.
 *
 * Scratch: a fixed array of 65536 span slots (256 KiB) compiled into the library, held by
 * every GPU that loads the library until the process exits.  The selection kernel keeps the
 * span means of a sender with at most 8192 spans in shared memory; only senders with more
 * spans (ceil(T[i] / span_width) > 8192, e.g. T above 131072 at width 16) take slots in the
 * array.  Senders are launched in groups of 64, each group placing its large senders from slot
 * 0, so a call is limited to 65536 such slots per group of 64 consecutive senders; a larger
 * call returns CB_ESHAPE with nothing enqueued.  The call allocates nothing: no cudaMalloc,
 * cudaFree or allocating library routine.
 *
 * Set-up: the first call on each device looks up the array's device address (with that
 * device current) and caches it; make that first call before any stream capture.
 *
 * Sharing: every call on a device uses the same array and finds the previous call's
 * contents in it (the kernel rewrites every slot it reads, and the call clears its status
 * word).  Calls whose kernels may overlap on the GPU race on the array: order them on one
 * stream or synchronise between them.  Arguments are as for cb_select; the current CUDA
 * device is used; host-side errors are returned at once and described by cb_last_error(NULL);
 * the kernel's own consistency check is read back by cb_select_noalloc_status.
 */
cb_status cb_select_noalloc(int32_t n, const float *const *scores, const int64_t *T,
                            const int64_t *budget, int32_t *const *idx, int32_t n_sink,
                            int32_t n_latent, int32_t span_width, void *stream);

/* Status of the allocation-free selection (no context, no allocation): waits for `stream`,
 * reads the status word that cb_select_noalloc's kernel keeps in the library's fixed array on
 * the current device, clears it, and returns CB_EDEVICE (text in cb_last_error(NULL)) when the
 * kernel's own check found a selected count different from the budget, CB_ECUDA when the
 * stream reported an error, else CB_OK.  It covers every cb_select_noalloc call on this device
 * since the last read.  Blocks the host. */
cb_status cb_select_noalloc_status(void *stream);

#ifdef __cplusplus
}
#endif
#endif /* CACHEBACK_H_ */
