/*
 * speechkv.h -- C ABI of the GB300 (sm_103a) SpeechKV decode hot path.
 *
 * SpeechKV ("Compress the Cache, Not the Speech Embedding", Sec. III-B)
 * compresses the speech span of a speech LLM's KV cache: from layer l0 on,
 * every window of w consecutive speech frames is replaced by one pooled key
 * and one pooled value, weighted by a softmax over a learned linear gate of
 * the keys (Eq. (pool)); text positions are kept.  Each decode step then
 * appends the new token's key/value and runs grouped-query attention of the
 * full-resolution query over the shorter cache (Eq. (attn)).  The pooling
 * runs once at prefill and its result is what the cache stores (Sec. III-C).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Pointers marked "dev" are CUDA device pointers; the caller owns every
 *   buffer, including the decode workspace.  Nothing here allocates device
 *   memory per call.
 * - Calls are asynchronous and ordered on `stream`; none synchronises the
 *   host.  Argument errors are detected on the host before any launch and
 *   returned as a status; nothing is launched then.
 * - Errors that depend on device-resident values (a cache that is full, a
 *   length beyond its capacity, inconsistent lengths, a bounded wait that
 *   ran out) set a per-device error word instead of faulting; the offending
 *   write is skipped.  speechkv_check_device_error() reads and clears it.
 * - Element types: SPEECHKV_F32 or SPEECHKV_BF16 storage for keys, values,
 *   queries and outputs; all arithmetic is fp32.  Head dim d is 64 or 128.
 * - Data pointers (keys, values, queries, outputs, caches, workspace) must be
 *   16-byte aligned.
 * - Layers are counted from 0; layer `layer` is pooled iff layer >= l0, so
 *   the paper's default "l0 = 5, first 4 layers full resolution" is l0 = 4.
 *
 * Cache layout (one buffer per layer for K and one for V)
 * -------------------------------------------------------
 * Request b owns rows [cache_off[b], cache_off[b+1]) of capacity
 * cap_b = cache_off[b+1] - cache_off[b].  Its block is head-major:
 * element (b, h, t, c) lives at ((cache_off[b] * H_kv + h * cap_b + t) * d + c)
 * for KV head h, cached row t < cap_b, channel c.  One (request, head) is thus
 * a single contiguous run of rows, which the decode kernel streams with bulk
 * asynchronous copies.  Rows are, in order: the P text tokens before the
 * speech, the n = ceil(T / w_eff) pooled speech entries, the N text tokens
 * after the speech, then the generated tokens.  len[b] (int32, dev) counts the
 * rows in use.
 */
#ifndef SPEECHKV_H_
#define SPEECHKV_H_

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    SPEECHKV_OK = 0,
    SPEECHKV_ERR_INVALID_ARG = 1,  /* bad pointer, size, shape or length   */
    SPEECHKV_ERR_UNSUPPORTED = 2,  /* valid but not built (d, group, dtype) */
    SPEECHKV_ERR_CUDA = 3,         /* a CUDA runtime call failed            */
    SPEECHKV_ERR_CAPACITY = 4,     /* a cache row would pass its capacity   */
    SPEECHKV_ERR_TIMEOUT = 5,      /* a bounded device wait ran out         */
    SPEECHKV_ERR_WORKSPACE = 6     /* decode workspace too small            */
} speechkv_status;

typedef enum { SPEECHKV_F32 = 0, SPEECHKV_BF16 = 1 } speechkv_dtype;

/* Largest batch speechkv_decode_attn / _step accept (their per-CTA tables). */
#define SPEECHKV_MAX_BATCH 512

/*
 * Flag of speechkv_decode_attn / speechkv_decode_step (and their paged and
 * allocation-free forms).  The decode kernels are launched with programmatic
 * dependent launch, so they may begin while the previous kernel on the
 * stream retires.  By default they wait for that kernel before reading
 * anything.  SPEECHKV_OVERLAP_PRIOR declares that the previous kernel on
 * `stream` writes none of this call's caches, len or cache_off (it may
 * produce q, k_new and v_new, and may use the same workspace): the call then
 * reads the lengths and starts streaming the cached rows at once, and waits
 * for the previous kernel only before reading q / k_new / v_new and before
 * any write.  Only that one kernel can still be running: a decode kernel
 * lets its successor start only after its own wait for its predecessor has
 * returned, so every kernel queued before the previous one has completed by
 * then, whatever grid sizes the calls use.  A kernel that precedes the call
 * without the launch attribute is simply waited for, as usual.
 */
#define SPEECHKV_OVERLAP_PRIOR 1u

/* Human-readable name of a status (static string, never NULL). */
const char *speechkv_status_string(speechkv_status status);

/*
 * Cached rows of one request at one layer (Sec. III-B: speech pooled in
 * windows of w from layer l0 on, text unchanged):
 *   P + ceil(T / w_eff) + N + G,  w_eff = (layer >= l0 ? w : 1).
 * P / N: text tokens before / after the speech, T: speech frames, G: tokens
 * generated so far.  A partial last window still yields one entry.  Pure host
 * function; returns -1 for negative counts, w < 1, layer < 0 or l0 < 0.
 */
int64_t speechkv_compressed_len(int32_t P, int32_t T, int32_t N, int32_t G,
                                int32_t w, int32_t layer, int32_t l0);

/*
 * speechkv_pool -- Eq. (pool), run once per request and layer at prefill.
 *
 * For every request b and KV head h, writes the cache rows described above
 * from the full-resolution prefill keys/values:
 *   - text rows are copied bit-exactly;
 *   - speech window i (frames i*w_eff .. min((i+1)*w_eff, T) - 1 of the
 *     speech span) becomes one row: logits z_j = gate[h] . k_j, weights
 *     alpha = softmax(z) over the window, k^ = sum alpha_j k_j and
 *     v^ = sum alpha_j v_j (values use the keys' weights), rounded once to the
 *     storage type (round to nearest even);
 *   - when layer < l0 (w_eff = 1) every row is copied bit-exactly.
 * Then sets len[b] = P[b] + ceil(T[b] / w_eff) + N[b].
 *
 * k_full, v_full  dev, [full_rows][H_kv][d] token-major prefill keys/values;
 *                 request b's rows are [full_off[b], full_off[b+1]), which
 *                 must hold exactly P[b] + T[b] + N[b] rows.
 * full_off        dev int64 [B+1], non-decreasing, full_off[B] <= full_rows.
 * P, T, N         dev int32 [B]: text before, speech frames, text after.
 * gate            dev fp32 [H_kv][d], 16-byte aligned: the gate vector u of
 *                 g(k) = u . k for this layer, one per KV head (no bias: a
 *                 bias is constant over a window and cancels in the softmax).
 * k_cache,v_cache dev, this layer's cache blocks (layout above).
 * cache_off       dev int64 [B+1], capacities in rows.
 * len             dev int32 [B], written.
 * full_rows       host: rows in k_full / v_full (sizes the launch).
 * w               window (>= 1); layer, l0 as above.
 * Errors: host-checked arguments return a status.  On the device, a request
 * whose rows do not match P+T+N sets SPEECHKV_ERR_INVALID_ARG; a request
 * whose pooled rows exceed its capacity sets SPEECHKV_ERR_CAPACITY (rows
 * beyond the capacity are not written and len is clamped to it).
 */
speechkv_status speechkv_pool(const void *k_full, const void *v_full,
                              const int64_t *full_off, const int32_t *P,
                              const int32_t *T, const int32_t *N,
                              const float *gate, void *k_cache, void *v_cache,
                              const int64_t *cache_off, int32_t *len,
                              int32_t B, int64_t full_rows, int32_t H_kv,
                              int32_t d, int32_t w, int32_t layer, int32_t l0,
                              speechkv_dtype dtype, cudaStream_t stream);

/*
 * speechkv_pool_hidden -- the HS-compression variant (Sec. IV-A): the
 * pooling of Eq. (pool) applied once, at layer l0, to the whole hidden
 * state instead of to each layer's keys and values, so that every later
 * layer (queries included) runs on the shorter sequence.
 *
 * For every request b: text rows are copied bit-exactly; speech window i
 * (frames i*w .. min((i+1)*w, T) - 1 of the speech span) becomes one row
 * with logits z_j = gate . h_j over the whole hidden vector, weights
 * alpha = softmax(z) over the window and h^ = sum alpha_j h_j, rounded once
 * to the storage type.  Output rows [P; pooled n; N] of request b start at
 * row out_off[b]; len[b] = P[b] + ceil(T[b] / w) + N[b].  w = 1 copies.
 *
 * h_full     dev, [full_rows][d_model] token-major hidden states; request b's
 *            rows are [full_off[b], full_off[b+1]) and must be P+T+N rows.
 * full_off   dev int64 [B+1].
 * P, T, N    dev int32 [B], as for speechkv_pool.
 * gate       dev fp32 [d_model]: the gate vector u of g(h) = u . h.
 * h_out      dev, [out_rows][d_model]; out_off dev int64 [B+1] gives each
 *            request's rows (capacity out_off[b+1] - out_off[b]).
 * len        dev int32 [B], written.
 * full_rows, out_rows  host: rows of h_full and h_out.
 * Supported: SPEECHKV_F32 or SPEECHKV_BF16 with d_model * element size a
 * multiple of 16 bytes and at most 16 KB (SPEECHKV_ERR_UNSUPPORTED
 * otherwise).  On the device, a request whose rows do not match P+T+N or
 * lie outside full_rows / out_rows sets SPEECHKV_ERR_INVALID_ARG; one whose
 * pooled rows exceed its capacity sets SPEECHKV_ERR_CAPACITY (rows beyond
 * the capacity are not written and len is clamped).
 */
speechkv_status speechkv_pool_hidden(const void *h_full,
                                     const int64_t *full_off,
                                     const int32_t *P, const int32_t *T,
                                     const int32_t *N, const float *gate,
                                     void *h_out, const int64_t *out_off,
                                     int32_t *len, int32_t B,
                                     int64_t full_rows, int64_t out_rows,
                                     int32_t d_model, int32_t w,
                                     speechkv_dtype dtype,
                                     cudaStream_t stream);

/*
 * speechkv_prefill_attn -- Eq. (attn) at prefill (Sec. III-B): every
 * full-resolution prompt query attends over the compressed cache rows that
 * precede it.
 *
 * The paper adjusts the causal mask so that a query sees only the positions
 * before it, with causality taken over the compressed sequence.  Here a
 * query at prompt position t (0 <= t < S_b = P + T + N) sits at compressed
 * position
 *     pi(t) = t                      (t < P, text before the speech)
 *           = P + (t - P) / w_eff    (speech frame: the row of its window)
 *           = t - T + n              (text after the speech)
 * and attends, with weights softmax(q . k / sqrt(d)), over rows 0 .. pi(t)
 * of its KV head (hq / (H_q / H_kv)).  With w_eff = 1 (layer < l0) this is
 * ordinary causal attention.  The cache is read as speechkv_pool leaves it:
 * rows 0 .. P + n + N - 1 of every (request, KV head).
 *
 * q           dev bf16 [q_rows][H_q][d], token-major prompt queries (after
 *             any rotary embedding); request b's positions 0 .. S_b - 1 are
 *             rows q_off[b] .. q_off[b+1] - 1.
 * q_off       dev int64 [B+1], q_off[b+1] - q_off[b] must equal P+T+N.
 * q_rows      host: rows of q and out.
 * P, T, N     dev int32 [B], as for speechkv_pool.
 * k_cache, v_cache, cache_off: this layer's cache (layout above).
 * cache_rows  host: the cache buffers hold cache_rows * H_kv * d elements
 *             (cache_off[B] <= cache_rows); reads never go past them.
 * out         dev bf16 [q_rows][H_q][d]: row q_off[b] + t of head hq is
 *             written for every t < S_b (other rows are left as they are).
 * scale       0 for 1/sqrt(d), else the logit scale.
 * w, layer, l0  w_eff = (layer >= l0 ? w : 1).
 * Supported: SPEECHKV_BF16, d = 64 or 128, B <= SPEECHKV_MAX_BATCH, H_q <= 256,
 * q_rows and cache_rows * H_kv below 2^31 (SPEECHKV_ERR_UNSUPPORTED
 * otherwise).  On the device a request whose query rows do not match P+T+N
 * (or lie outside q_rows / cache_rows) sets SPEECHKV_ERR_INVALID_ARG, one
 * whose compressed rows exceed its capacity SPEECHKV_ERR_CAPACITY; such
 * requests are skipped.
 */
speechkv_status speechkv_prefill_attn(const void *q, const int64_t *q_off,
                                      int64_t q_rows, const int32_t *P,
                                      const int32_t *T, const int32_t *N,
                                      const void *k_cache, const void *v_cache,
                                      const int64_t *cache_off,
                                      int64_t cache_rows, void *out,
                                      float scale, int32_t B, int32_t H_q,
                                      int32_t H_kv, int32_t d, int32_t w,
                                      int32_t layer, int32_t l0,
                                      speechkv_dtype dtype,
                                      cudaStream_t stream);

/*
 * speechkv_append -- one decode step's cache update (Sec. III-C: decoding
 * appends each new token to the cache uncompressed).
 *
 * For every request b: writes k_new[b], v_new[b] ([H_kv][d]) as cached row
 * len[b] of request b, then len[b] += 1.  A request whose cache is full
 * (len[b] >= cap_b, or len[b] < 0) is left untouched and sets
 * SPEECHKV_ERR_CAPACITY in the device error word.
 *
 * k_new, v_new   dev, [B][H_kv][d].
 * k_cache, v_cache, cache_off, len: as for speechkv_pool (len read+written).
 * w, layer, l0   validated only (w >= 1, layer >= 0, l0 >= 0).
 */
speechkv_status speechkv_append(const void *k_new, const void *v_new,
                                void *k_cache, void *v_cache,
                                const int64_t *cache_off, int32_t *len,
                                int32_t B, int32_t H_kv, int32_t d, int32_t w,
                                int32_t layer, int32_t l0,
                                speechkv_dtype dtype, cudaStream_t stream);

/*
 * Bytes of workspace speechkv_decode_attn needs for a batch of B requests
 * with the given heads and head dim, launched on `grid_ctas` CTAs (0 = the
 * automatic grid, sized from the current device's SM count).  The workspace
 * holds split-K partial results, one arrival counter per (request, KV head)
 * and one counter of the fused step.  Returns 0 for invalid arguments.
 */
size_t speechkv_decode_workspace_size(int32_t B, int32_t H_q, int32_t H_kv,
                                      int32_t d, int32_t grid_ctas);

/*
 * speechkv_decode_attn -- Eq. (attn) for one decode step at one layer.
 *
 * For every request b and query head hq (KV head h = hq / (H_q / H_kv)):
 *   s_j = scale * q[b][hq] . k_j  for the cached rows j < len[b],
 *   out[b][hq] = sum_j softmax(s)_j v_j,
 * rounded once to the storage type.  scale <= 0 selects 1 / sqrt(d).  A
 * request with len[b] == 0 gets a zero output.  len[b] > cap_b sets
 * SPEECHKV_ERR_CAPACITY and attends over cap_b rows.
 *
 * The work (every request's rows times its KV heads) is cut evenly over a
 * persistent grid; every CTA streams its share from HBM once, serving all
 * H_q / H_kv query heads of a KV head from one read, and pieces of a
 * (request, head) processed by several CTAs are merged with a log-sum-exp
 * combine by the CTA that finishes last (no CTA ever waits for another).
 *
 * q            dev, [B][H_q][d].
 * k_cache, v_cache, cache_off, len: as for speechkv_pool (len read only).
 * out          dev, [B][H_q][d], written.
 * H_q / H_kv   1 to 8 for bf16 (3 to 8 on tensor cores: warp-level bf16 MMA
 *              with fp32 accumulation, the weights rounded to bf16 before
 *              P.V and normalised by the sum of the rounded weights), 1, 2
 *              or 4 for fp32; d must be 64 or 128; B <= SPEECHKV_MAX_BATCH.
 * w, layer, l0 validated only.
 * grid_ctas    CTAs to launch; 0 = automatic (one per SM times the
 *              kernel's residency).  Results do not depend on it beyond
 *              floating-point summation order.
 * workspace    dev, >= speechkv_decode_workspace_size(B, H_q, H_kv, d,
 *              grid_ctas) bytes.  It must be zero-filled once before its
 *              first use; every call leaves its counters at zero again.
 *              Calls that run concurrently need separate workspaces.  After
 *              a device error, zero it again.
 * flags        0 or SPEECHKV_OVERLAP_PRIOR (see above).
 */
speechkv_status speechkv_decode_attn(const void *q, const void *k_cache,
                                     const void *v_cache,
                                     const int64_t *cache_off,
                                     const int32_t *len, void *out,
                                     float scale, int32_t B, int32_t H_q,
                                     int32_t H_kv, int32_t d, int32_t w,
                                     int32_t layer, int32_t l0,
                                     int32_t grid_ctas, void *workspace,
                                     size_t workspace_bytes,
                                     speechkv_dtype dtype, uint32_t flags,
                                     cudaStream_t stream);

/*
 * speechkv_decode_step -- one decode step at one layer with the cache update
 * fused in: speechkv_append followed by speechkv_decode_attn in a single
 * launch (Sec. III-C: the new token's key/value join the cache uncompressed;
 * Eq. (attn): the query attends over the cache including that token).
 *
 * For every request b with len[b] < cap_b: k_new[b], v_new[b] are written as
 * cached row len[b] and take part in the attention as that row, and len[b]
 * advances by one (after every CTA has read it).  A request whose cache is
 * full sets SPEECHKV_ERR_CAPACITY and attends over its cached rows only.
 * Results equal speechkv_append then speechkv_decode_attn up to summation
 * order.
 *
 * k_new, v_new   dev, [B][H_kv][d] (16-byte aligned).
 * All other arguments as for speechkv_decode_attn; len is read and written,
 * and the caches are written at the new rows.  The workspace (same size as
 * for speechkv_decode_attn) must not be shared with a concurrent call.
 */
speechkv_status speechkv_decode_step(const void *q, const void *k_new,
                                     const void *v_new, void *k_cache,
                                     void *v_cache, const int64_t *cache_off,
                                     int32_t *len, void *out, float scale,
                                     int32_t B, int32_t H_q, int32_t H_kv,
                                     int32_t d, int32_t w, int32_t layer,
                                     int32_t l0, int32_t grid_ctas,
                                     void *workspace, size_t workspace_bytes,
                                     speechkv_dtype dtype, uint32_t flags,
                                     cudaStream_t stream);

/*
 * speechkv_decode_step_noalloc -- speechkv_decode_step for callers that
 * cannot allocate device memory.  The paper has no counterpart: this entry
 * point only changes where the split-K scratch lives.
 *
 * Some callers may not allocate GPU memory at all: a plug-in running inside
 * a serving process whose memory pool owns every byte of the device, or a
 * latency-critical path that must never enter an allocator (whose calls can
 * block, synchronise the device or fail).  Such a caller passes no
 * workspace: the scratch is a fixed array of SPEECHKV_NOALLOC_SCRATCH_BYTES
 * in device memory that the library itself owns (every GPU that loads the
 * library holds it until the process exits).  This call allocates nothing.
 *
 * Arguments, results and errors are those of speechkv_decode_step, minus the
 * workspace.  A batch whose scratch (speechkv_decode_workspace_size for the
 * same shapes and grid) exceeds SPEECHKV_NOALLOC_SCRATCH_BYTES is refused with
 * SPEECHKV_ERR_WORKSPACE before anything runs.  The first call on a device
 * looks up the array's device address (a one-time set-up per device); make
 * that first call before any stream capture.  Every call shares the one
 * array, which keeps the previous call's contents: once all arguments have
 * passed the host checks, each call zeroes the counters it needs on `stream`
 * (an asynchronous memset, not an allocation) and then launches, and calls
 * that may run at the same time on one device (for example on two streams)
 * race on it.  Because that memset sits between the previous kernel and
 * the decode kernel, SPEECHKV_OVERLAP_PRIOR is accepted but gives no
 * overlap here.
 */
#define SPEECHKV_NOALLOC_SCRATCH_BYTES (8u << 20)

speechkv_status speechkv_decode_step_noalloc(
    const void *q, const void *k_new, const void *v_new, void *k_cache,
    void *v_cache, const int64_t *cache_off, int32_t *len, void *out,
    float scale, int32_t B, int32_t H_q, int32_t H_kv, int32_t d, int32_t w,
    int32_t layer, int32_t l0, int32_t grid_ctas, speechkv_dtype dtype,
    uint32_t flags, cudaStream_t stream);

/*
 * Paged caches -- the block-table layout of the paper's serving system (a
 * vLLM-style paged KV cache, Sec. V-D); the paper has no other use for it.
 * A layer's keys and values live in fixed-size pages
 *     k_pages, v_pages   dev, [num_blocks][H_kv][block_size][d]
 * and request b's logical rows t are found through its block-table row:
 *     row t -> page block_table[b * max_blocks + t / block_size],
 *              slot t % block_size of that page (every KV head's slot).
 * block_table  dev int32 [B][max_blocks]; an entry is a page index in
 *              [0, num_blocks) for every row the call reads or writes
 *              (others may hold anything, e.g. -1).
 * block_size   a power of two; each request's capacity is
 *              max_blocks * block_size rows (at most 2^31 - 1).  The
 *              decode step reads a tile in 16-row groups aligned to the
 *              rows' index (bf16: one copy per group and page, issued in
 *              parallel): measured against the contiguous layout, 64-row
 *              pages cost 4-7 %, 16-row pages (vLLM's default) 7-14 %.
 * num_blocks   host: pages in k_pages / v_pages (bounds the table entries).
 * The other arguments, the results and the errors are those of the
 * contiguous entry point of the same name (the rows and their order are the
 * same; only where they live differs).  A table entry outside [0, num_blocks)
 * where a row is needed sets SPEECHKV_ERR_INVALID_ARG on the device; that
 * row is neither written nor used (its contents in the result are
 * unspecified).
 */
speechkv_status speechkv_pool_paged(const void *k_full, const void *v_full,
                                    const int64_t *full_off, const int32_t *P,
                                    const int32_t *T, const int32_t *N,
                                    const float *gate, void *k_pages,
                                    void *v_pages, const int32_t *block_table,
                                    int32_t max_blocks, int32_t block_size,
                                    int64_t num_blocks, int32_t *len,
                                    int32_t B, int64_t full_rows, int32_t H_kv,
                                    int32_t d, int32_t w, int32_t layer,
                                    int32_t l0, speechkv_dtype dtype,
                                    cudaStream_t stream);
speechkv_status speechkv_append_paged(const void *k_new, const void *v_new,
                                      void *k_pages, void *v_pages,
                                      const int32_t *block_table,
                                      int32_t max_blocks, int32_t block_size,
                                      int64_t num_blocks, int32_t *len,
                                      int32_t B, int32_t H_kv, int32_t d,
                                      int32_t w, int32_t layer, int32_t l0,
                                      speechkv_dtype dtype,
                                      cudaStream_t stream);
speechkv_status speechkv_decode_step_paged(
    const void *q, const void *k_new, const void *v_new, void *k_pages,
    void *v_pages, const int32_t *block_table, int32_t max_blocks,
    int32_t block_size, int64_t num_blocks, int32_t *len, void *out,
    float scale, int32_t B, int32_t H_q, int32_t H_kv, int32_t d, int32_t w,
    int32_t layer, int32_t l0, int32_t grid_ctas, void *workspace,
    size_t workspace_bytes, speechkv_dtype dtype, uint32_t flags,
    cudaStream_t stream);
/*
 * speechkv_prefill_attn_paged -- speechkv_prefill_attn over a paged cache
 * (pages as above; no cache_off / cache_rows).  block_size must be at least 8
 * (a key tile is copied as one piece per page of whole 8-row swizzle atoms;
 * SPEECHKV_ERR_UNSUPPORTED below that); num_blocks * H_kv * block_size must
 * stay below 2^31.  Pages past a request's compressed rows are not read.
 * Results are bit-identical to speechkv_prefill_attn over the same rows;
 * measured against it, 16-row pages cost 2-3 %.
 */
speechkv_status speechkv_prefill_attn_paged(
    const void *q, const int64_t *q_off, int64_t q_rows, const int32_t *P,
    const int32_t *T, const int32_t *N, const void *k_pages,
    const void *v_pages, const int32_t *block_table, int32_t max_blocks,
    int32_t block_size, int64_t num_blocks, void *out, float scale,
    int32_t B, int32_t H_q, int32_t H_kv, int32_t d, int32_t w,
    int32_t layer, int32_t l0, speechkv_dtype dtype, cudaStream_t stream);

/*
 * Synchronises `stream`, then reads and clears the current device's error
 * word.  Returns SPEECHKV_OK when no kernel reported an error since the last
 * check, else the first error reported (CAPACITY, INVALID_ARG or TIMEOUT),
 * or SPEECHKV_ERR_CUDA if the synchronisation itself failed.
 */
speechkv_status speechkv_check_device_error(cudaStream_t stream);

/*
 * Self-test of the failure path shared by every kernel (no argument of the
 * paper's method is involved): launches one CTA whose single waiting thread
 * waits, through the same bounded wait the kernels use, for an mbarrier phase
 * that nothing completes.  After the wait limit (1 s of %globaltimer) it
 * gives up, records SPEECHKV_ERR_TIMEOUT in the device error word and the
 * kernel returns normally: no trap, no fault, the context stays usable.
 * Returns SPEECHKV_OK once launched (SPEECHKV_ERR_CUDA if the launch failed);
 * read the recorded status with speechkv_check_device_error.  Stream-ordered,
 * asynchronous.
 */
speechkv_status speechkv_selftest_timeout(cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SPEECHKV_H_ */
