/*
 * kvblend.h - C ABI of the GB300 selective-recompute prefill library (libkvblend.so).
 *
 * The library computes the prefill that runs after per-chunk KV caches are
 * concatenated (the CacheBlend-style selective recompute combined with a
 * concatenation-aware model in the paper "Fine-Tuning a KV Cache
 * Concatenation-Aware Model or Recomputing KV Caches? Why Not Both?"):
 * position re-alignment of each chunk's cached keys (Sec. 3.4, Sec. 4), full
 * causal recompute of layer 0 (Sec. 4), per-token key deviation and top-k
 * selection at ratio r (Sec. 2, Sec. 3.2), and, in every later layer, the
 * recompute of the selected rows with attention over the whole blended cache
 * under a causal mask (Sec. 4, Limitations).
 *
 * Conventions shared by every call
 *  - Pointers named *_host are host memory; every other data pointer is device
 *    memory of the current CUDA device.  The caller owns all buffers; the library
 *    never allocates or frees device memory.  Scratch memory comes from a caller
 *    workspace whose size kvb_workspace_size() / kvb_hkvd_workspace_size() give.
 *  - bf16 and fp16 tensors are passed as uint16_t* (raw bits); fp32 as float*.
 *  - All device pointers must be 16-byte aligned.  Matrices are row-major and dense.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *    Every call is asynchronous on that stream and enqueues no host synchronisation,
 *    except kvb_device_status(), which synchronises the stream.
 *  - Return value: KVB_OK, or an error code for argument validation (before any
 *    launch) or a CUDA launch error.  kvb_last_error() returns a message for the
 *    last failing call on the calling thread.  Errors detected on the device
 *    (a bounded wait that ran out) are recorded in the workspace status word and
 *    read with kvb_device_status().  The word is the first 4 bytes of a workspace:
 *    zero the workspace's first 256 bytes once before its first use; calls never
 *    clear it, kvb_device_status() clears it after reading.
 *
 * Model layout (Llama-3.1 decoder, Sec. 4): hidden H, Hq query heads, Hkv kv heads,
 * head dim D in {64, 128}, MLP dim F, Hq % Hkv == 0 (group sizes Hq/Hkv up to 128 in
 * the prefill, up to 8 in the decode).
 *  - KV cache of one layer: [n_rows][Hkv][D] for K and for V; a multi-layer cache
 *    is n_layers such blocks back to back.  Two formats:
 *      chunk caches (what a caller stores per document, Sec. 3.4: the inputs of
 *      kvb_rope_realign and kvb_selective_prefill*, the optional V output of
 *      kvb_full_prefill): K and V both bf16, as the paper's bf16 model writes them;
 *      the blended cache (row t holds token t of the concatenated sequence, global
 *      position t; what the attention kernels read): K bf16, V in fp16 containers
 *      holding bf16-precision values, so that the attention's P.V product runs as an
 *      fp16 MMA whose softmax weights are rounded to fp16 rather than bf16 (8x
 *      smaller rounding error, same speed).
 *    The bf16 -> fp16 conversion of V (done by the merge pass, which reads and writes
 *    every V element anyway) is exact for 2^-14 <= |v| <= 65504 and for 0; a smaller
 *    non-zero |v| is rounded to fp16's subnormal spacing 2^-24 (absolute error at most
 *    2^-25); |v| > 65504 (the largest bf16 value below it is 65280) cannot be held:
 *    it is written as +-65504, NaN stays NaN, and both record KVB_ERR_RANGE in the
 *    workspace status word.
 *  - RoPE is rotate-half (dimension i pairs with i + D/2); tables hold
 *    cos/sin(pos * w_i) in fp32, [max_pos][D/2], computed in double precision.
 */
#ifndef KVBLEND_H
#define KVBLEND_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum kvb_status {
    KVB_OK = 0,
    KVB_ERR_INVALID_ARG = 1,   /* a pointer, size or shape the call cannot accept       */
    KVB_ERR_UNSUPPORTED = 2,   /* valid in principle but not built (e.g. head_dim 96)   */
    KVB_ERR_CUDA = 3,          /* a CUDA runtime/driver call or a launch failed         */
    KVB_ERR_TIMEOUT = 4,       /* device side: a bounded wait in a kernel ran out       */
    KVB_ERR_WORKSPACE = 5,     /* workspace missing or smaller than required            */
    KVB_ERR_RANGE = 6          /* device side: a value outside the range of its storage
                                * type (a V entry beyond fp16's finite range)           */
} kvb_status;

/* Frequency scaling of the rotary embedding (kvb_config.rope_scaling). */
enum {
    KVB_ROPE_PLAIN = 0,    /* w_i = theta^(-2i/D)                                            */
    KVB_ROPE_LLAMA3 = 1,   /* Llama 3.1: factor rs_factor, low/high frequency factors
                            * rs_low/rs_high, original context rs_orig_ctx                   */
    KVB_ROPE_YARN = 2      /* YaRN (the scaling of the paper's second model, Sec. 4): NTK-by-
                            * parts interpolation with scale s = rs_factor >= 1, ramp bounds
                            * alpha = rs_low < beta = rs_high (turns of a pair over the
                            * original context rs_orig_ctx), and the attention logits
                            * multiplied by (0.1 ln s + 1)^2 (YaRN's temperature)            */
};

/* Model shape and RoPE settings.  Hq must be a multiple of Hkv; any group size
 * Hq/Hkv <= 128 runs in the prefill, group sizes up to 8 in the decode. */
typedef struct kvb_config {
    int32_t hidden, n_q_heads, n_kv_heads, head_dim, mlp_dim, n_layers, vocab;
    float rms_eps;
    float rope_theta;
    int32_t rope_scaling;                 /* KVB_ROPE_*                               */
    float rs_factor, rs_low, rs_high;
    int32_t rs_orig_ctx;
} kvb_config;

/* Device pointers of one decoder layer.  Linear weights are [out][in] bf16:
 * w_qkv [(Hq+2Hkv)D][H] (rows: q heads, then k heads, then v heads), w_o [H][Hq D],
 * w_gate and w_up [F][H], w_down [H][F]; norm gains are fp32 [H]. */
typedef struct kvb_layer_weights {
    const float* attn_norm;
    const uint16_t* w_qkv;
    const uint16_t* w_o;
    const float* mlp_norm;
    const uint16_t* w_gate;
    const uint16_t* w_up;
    const uint16_t* w_down;
    const float* b_qkv;   /* fp32 [(Hq+2Hkv)D] bias of the q/k/v projection (added before
                           * RoPE), or NULL for none                                      */
} kvb_layer_weights;

/* Whole model: `layers` is a HOST array of n_layers entries; embed is [vocab][H] bf16,
 * final_norm [H] fp32 (device). */
typedef struct kvb_model {
    const kvb_layer_weights* layers;
    const uint16_t* embed;
    const float* final_norm;
} kvb_model;

/* RoPE tables in device memory, fp32 [max_pos][D/2] each. */
typedef struct kvb_rope_table {
    const float* cos;
    const float* sin;
    int64_t max_pos;
} kvb_rope_table;

/* Multi-layer blended KV cache: k (bf16) and v (fp16 containers, bf16-precision values)
 * are [n_layers][n_rows][Hkv][D]. */
typedef struct kvb_kv_cache {
    uint16_t* k;
    uint16_t* v;
    int64_t n_rows;
    int32_t n_layers;
} kvb_kv_cache;

/* Stage and kernel times of one prefill in milliseconds (CUDA events on the call's
 * stream; kernel times are sums of per-launch event pairs). */
typedef struct kvb_timings {
    float total_ms;
    float realign_ms;     /* merge + position re-alignment of the chunk caches      */
    float dense_ms;       /* layers before the check layer, all rows (layer 0)       */
    float select_ms;      /* check-layer keys, deviation and top-k                    */
    float selective_ms;   /* selective layers over the recomputed rows                */
    float final_ms;       /* final RMSNorm of the query rows                          */
    float attn_dense_ms;  /* attention launches of the dense layers                  */
    float attn_sel_ms;    /* attention launches of the selective layers              */
    float gemm_ms;        /* all GEMM launches                                        */
    float hkvd_ms;        /* deviation + top-k launches                               */
    int32_t n_attn_dense, n_attn_sel, n_gemm;
    int32_t n_launches;   /* kernels this call launched                              */
    int64_t n_selected;   /* k = number of recomputed context rows                   */
    int64_t n_rows;       /* m = k + n_query                                          */
} kvb_timings;

/* Residual rows captured at layer boundaries, for inspection and per-layer parity checks
 * (the paper has no counterpart).  For every i < n, the fp32 residual rows that ENTER
 * layer layers[i] are copied into x_out + i * rows_cap * H just before that layer runs;
 * layers[i] == n_layers captures the rows leaving the last layer (before the final
 * RMSNorm).  Which rows: in a dense layer (every layer of kvb_full_prefill; the layers
 * before check_layer of a selective prefill, or all of them when it runs dense) all rows
 * in sequence order; from check_layer on, the m = k + n_query recomputed rows: the
 * selected context rows in ascending index order (as sel_out), then the query rows.
 * The copies run on the call's stream (device to device), outside any kernel.
 *   layers:   HOST int32 [n], each in [0, n_layers], any order, repeats allowed
 *   x_out:    DEVICE fp32 [n][rows_cap][H], 16-byte aligned
 *   rows_cap: rows per slot; a tap that needs more rows fails the call with INVALID_ARG
 *             before anything is launched
 *   rows_out: HOST int64 [n] or NULL: the number of rows captured for layers[i] */
typedef struct kvb_layer_taps {
    int32_t n;
    const int32_t* layers;
    float* x_out;
    int64_t rows_cap;
    int64_t* rows_out;
} kvb_layer_taps;

/* ------------------------------------------------------------------ status */

/* Static text for a status code. */
const char* kvb_status_string(kvb_status s);
/* Message of the last failing call on this thread ("" if none).  Thread-local. */
const char* kvb_last_error(void);
/* Library ABI version (major * 100 + minor). */
int32_t kvb_version(void);

/* ------------------------------------------------------------------ RoPE */

/* Fill HOST tables cos_host/sin_host, each [max_pos][D/2] fp32, with cos/sin of
 * pos * w_i for pos < max_pos (w_i = theta^(-2i/D) under cfg->rope_scaling;
 * Sec. 4 asks for the position adjustment in float32 - angles are formed in double
 * and rounded once).  The tables hold pure rotations: YaRN's temperature is applied
 * to the attention logits (kvb_attention_scale), not folded into cos/sin, so that the
 * re-alignment of cached keys stays a rotation.  Pure host call.  Errors: INVALID_ARG
 * for NULL pointers, max_pos < 1, an unknown scaling or bad scaling parameters,
 * UNSUPPORTED for a head_dim that is not built. */
kvb_status kvb_rope_table_fill(const kvb_config* cfg, int64_t max_pos,
                               float* cos_host, float* sin_host);

/* The factor every attention kernel applies to q.k before the softmax: 1/sqrt(D),
 * times (0.1 ln s + 1)^2 under KVB_ROPE_YARN (YaRN, Sec. 3.4 of its paper).  Pure
 * host call.  Errors: INVALID_ARG for NULL pointers or an invalid config. */
kvb_status kvb_attention_scale(const kvb_config* cfg, float* scale_out);

/* ------------------------------------------------------------------ steps */

/* Merge + position re-alignment (Sec. 3.4 "merged into one, followed by position
 * adjustment"; PIE, Sec. 2).  For layers [layer_begin, layer_end) and every context
 * row t < n_ctx in chunk c (chunk_start[c] <= t < chunk_start[c+1]):
 *   k_dst[l][t] = R(chunk_start[c]) k_src[l][t]   (rotation of every head's pairs by
 *                                                  the chunk offset, fp32 math, bf16 out)
 *   v_dst[l][t] = v_src[l][t]                     (bf16 chunk format -> fp16 container of
 *                                                  the blended cache; skipped when v_src or
 *                                                  v_dst is NULL)
 * k_src/v_src are chunk caches [n_layers][src_rows][Hkv][D] (K and V bf16) with keys
 * rotated at chunk-local positions; k_dst/v_dst are blended-cache layers
 * [n_layers][dst_rows][Hkv][D] (K bf16, V fp16).  In place is allowed (k_src == k_dst,
 * v_src == v_dst, src_rows == dst_rows: V is then converted in place).  chunk_start:
 * DEVICE int32 [n_chunks+1], ascending, chunk_start[0] == 0, chunk_start[n_chunks] ==
 * n_ctx.  The rope table must cover max_pos > chunk_start[n_chunks-1].  ws: at least 256
 * bytes whose first word is the device status word, which receives KVB_ERR_RANGE if a V
 * value lies outside fp16's range (see the layout notes above); may be NULL when V is
 * skipped.  Errors: INVALID_ARG, WORKSPACE. */
kvb_status kvb_rope_realign(const kvb_config* cfg, const kvb_rope_table* rope,
                            const uint16_t* k_src, const uint16_t* v_src, int64_t src_rows,
                            uint16_t* k_dst, uint16_t* v_dst, int64_t dst_rows,
                            int32_t layer_begin, int32_t layer_end,
                            const int32_t* chunk_start, int32_t n_chunks, int64_t n_ctx,
                            void* ws, size_t ws_bytes, void* stream);

/* Workspace bytes kvb_hkvd_select needs for n_ctx rows. */
size_t kvb_hkvd_workspace_size(int64_t n_ctx);

/* HKVD deviation and top-k (Sec. 2 on CacheBlend, Sec. 3.2: tokens whose keys
 * deviate most, by squared key difference, are recomputed):
 *   dev_out[i] = sum over kv heads and dims of (k_fresh[i] - k_cached[i])^2   (fp32)
 *   sel_out    = the k indices with the largest dev, ties to the lower index,
 *                written in ascending order.
 * k_fresh row i at k_fresh + i*ld_fresh, k_cached row i at k_cached + i*ld_cached
 * (elements), kv_dim elements per row (multiple of 8).  0 <= k <= n_ctx.
 * dev_out: [n_ctx] fp32 (required); sel_out: [k] int32.  Workspace: at least
 * kvb_hkvd_workspace_size(n_ctx) bytes, 256-byte aligned.  Errors: INVALID_ARG,
 * WORKSPACE. */
kvb_status kvb_hkvd_select(const uint16_t* k_fresh, int64_t ld_fresh,
                           const uint16_t* k_cached, int64_t ld_cached,
                           int64_t n_ctx, int32_t kv_dim, int64_t k,
                           int32_t* sel_out, float* dev_out,
                           void* ws, size_t ws_bytes, void* stream);

/* Gather + RMSNorm + QKV projection + RoPE for m rows (the per-row front half of a
 * decoder layer, Sec. 4 model):
 *   a[r]   = RMSNorm(x[row_idx[r]]) * attn_norm          (x: fp32 [*][H]; row_idx NULL = r)
 *   q[r]   = RoPE(a[r] W_q^T, rope_pos[r])  -> q_out [m][Hq D] bf16
 *   k[r]   = RoPE(a[r] W_k^T, rope_pos[r])  -> k_out row kv_dst[r] (or r), [n_kv_rows][Hkv D] bf16
 *   v[r]   = a[r] W_v^T                     -> v_out row kv_dst[r] (or r), fp16 holding
 *                                              the bf16-rounded value
 * Passing a cache layer as k_out/v_out with kv_dst = the rows' cache indices fuses the
 * KV scatter.  rope_pos: [m] int32.  Index contents are checked on the device where they
 * are used: a row whose destination kv_dst[r] (or r) lies outside [0, n_kv_rows) writes
 * no k/v row, and a rope_pos[r] outside [0, rope->max_pos) is rotated by position 0;
 * either records KVB_ERR_INVALID_ARG in the workspace status word (the results of such
 * a call are not meaningful, but no memory outside the given buffers is touched).  Uses
 * tcgen05 tensor cores (bf16 in, fp32 accumulate).  Workspace >= kvb_workspace_size(cfg,
 * m).  Errors: INVALID_ARG, WORKSPACE, UNSUPPORTED. */
kvb_status kvb_gather_rmsnorm_qkv(const kvb_config* cfg, const kvb_layer_weights* w,
                                  const kvb_rope_table* rope,
                                  const float* x, const int32_t* row_idx,
                                  const int32_t* rope_pos, int64_t m,
                                  uint16_t* q_out, uint16_t* k_out, uint16_t* v_out,
                                  const int32_t* kv_dst, int64_t n_kv_rows,
                                  void* ws, size_t ws_bytes, void* stream);

/* Allocation-free variant of kvb_gather_rmsnorm_qkv (the paper has no counterpart:
 * this serves callers, not the method).  Some callers cannot hand the library any
 * device memory of their own - e.g. a plugin inside a serving process whose memory
 * pool owns all device memory, or a hot loop that must never enter an allocator -
 * so the scratch this step needs (the m normalised bf16 rows that feed the GEMM)
 * lives in a fixed array inside the library, KVB_NOALLOC_MAX_ELEMS bf16 values
 * (8 MiB) that every GPU loading the library holds until the process exits.
 * Arguments, validation and results are those of kvb_gather_rmsnorm_qkv without the
 * workspace; status_out (DEVICE int32, zeroed by the caller, or NULL) receives what the
 * workspace status word would: KVB_ERR_TIMEOUT if a bounded wait in the GEMM runs out,
 * KVB_ERR_INVALID_ARG for an index outside its range.  m * hidden above
 * KVB_NOALLOC_MAX_ELEMS is rejected with INVALID_ARG.  No memory is allocated or freed.
 * The first call on a device looks the array's address up (cudaGetSymbolAddress) for that
 * device, so make it before any stream capture; the address is kept for the life of the
 * process, so do not use this entry point on a device after cudaDeviceReset() there.
 * Every call reuses the same array (nothing in it has to start at zero: each call
 * overwrites the rows it reads); calls whose kernels overlap on the GPU, e.g. on
 * unordered streams, race on it.  Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
#define KVB_NOALLOC_MAX_ELEMS (4 * 1024 * 1024)
kvb_status kvb_gather_rmsnorm_qkv_noalloc(const kvb_config* cfg, const kvb_layer_weights* w,
                                          const kvb_rope_table* rope,
                                          const float* x, const int32_t* row_idx,
                                          const int32_t* rope_pos, int64_t m,
                                          uint16_t* q_out, uint16_t* k_out, uint16_t* v_out,
                                          const int32_t* kv_dst, int64_t n_kv_rows,
                                          int32_t* status_out, void* stream);

/* KV scatter (Sec. 3.4: recomputed entries replace the cached ones): for r < m,
 *   k_dst[dst_idx[r]] = k_rows[r], v_dst[dst_idx[r]] = v_rows[r]   (kv_dim elements)
 * dst_idx values must be distinct and < n_dst_rows (bit copy, order irrelevant); a row
 * whose dst_idx lies outside [0, n_dst_rows) is skipped (the kernel checks each index).
 * Errors: INVALID_ARG. */
kvb_status kvb_kv_scatter(const uint16_t* k_rows, const uint16_t* v_rows,
                          const int32_t* dst_idx, int64_t m, int32_t kv_dim,
                          uint16_t* k_dst, uint16_t* v_dst, int64_t n_dst_rows,
                          void* stream);

/* Sparse-query causal GQA attention (Sec. 4: recompute with an attention mask;
 * Limitations 1: selected query rows attending the whole cache, causally):
 *   out[r, j] = sum_{t = lo_r}^{hi_r} softmax_t(q[r, j] . K[t, g] / sqrt(D)) V[t, g],
 *   g = j / (Hq/Hkv), hi_r = q_idx[r], lo_r = kv_lo ? kv_lo[r] : 0.
 * q: [m][Hq][D] bf16 (rotated); q_idx: [m] int32, ascending, < n_kv; kv_lo: [m] or
 * NULL; k_cache (bf16) / v_cache (fp16): one layer, [n_kv][Hkv][D]; out: [m][Hq D]
 * bf16.  tcgen05 tensor cores (Q.K^T bf16, P.V fp16), fp32 softmax.  ws: at least
 * 256 bytes (device status word).  Errors: INVALID_ARG, UNSUPPORTED, WORKSPACE. */
kvb_status kvb_sparse_query_attn(const kvb_config* cfg, const uint16_t* q,
                                 const int32_t* q_idx, const int32_t* kv_lo, int64_t m,
                                 const uint16_t* k_cache, const uint16_t* v_cache, int64_t n_kv,
                                 uint16_t* out, void* ws, size_t ws_bytes, void* stream);

/* Back half of a decoder layer on m rows (Sec. 4 model):
 *   x[r] += attn[r] W_o^T;  x[r] += W_down (silu(W_gate n) * (W_up n)),  n = RMSNorm(x[r]) * mlp_norm
 * attn: [m][Hq D] bf16; x: [m][H] fp32, updated in place.  Workspace >=
 * kvb_workspace_size(cfg, m).  Errors: INVALID_ARG, WORKSPACE. */
kvb_status kvb_mlp_rows(const kvb_config* cfg, const kvb_layer_weights* w,
                        const uint16_t* attn, int64_t m, float* x,
                        void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------ whole prefill */

/* Workspace bytes for a prefill (or a single step) over up to n_rows rows. */
kvb_status kvb_workspace_size(const kvb_config* cfg, int64_t n_rows, size_t* bytes);

/* Selective-recompute prefill over concatenated per-chunk caches (the whole path):
 *  1. merge + re-align the chunk caches of layers >= check_layer into `cache`
 *     (rows [0, n_ctx) of each layer);
 *  2. layers < check_layer (layer 0 at least): all n = n_ctx + n_query rows, causal;
 *  3. check layer: fresh keys of all context rows at global positions, deviation
 *     against the re-aligned cache, top-k with k = floor(r * n_ctx) (or the forced set);
 *  4. layers >= check_layer: rows S = selected context rows + the n_query query rows,
 *     K/V scattered into the cache before attention over the whole cache;
 *  5. final RMSNorm of the query rows -> final_hidden [n_query][H] fp32.
 * k_chunks/v_chunks: chunk caches [n_layers][n_ctx][Hkv][D] (K and V bf16), each chunk's
 * cache at chunk-local positions (read only).  cache: output blended cache (K bf16, V fp16)
 * with n_rows >= n_ctx + n_query.
 * token_ids: DEVICE int32 [n_ctx + n_query]; chunk_start: DEVICE int32 [n_chunks+1]
 * with chunk_start[n_chunks] == n_ctx.  r in [0, 1]; 1 <= check_layer <= n_layers
 * (check_layer == n_layers means every layer is dense).  forced_sel: DEVICE int32
 * [forced_k] ascending distinct context indices, or NULL.  sel_out: DEVICE int32 [n_ctx]
 * or NULL (receives the k chosen indices).  t: HOST timings or NULL (timing adds
 * events but no synchronisation until the call returns; with t != NULL the call
 * synchronises the stream once at the end to read the events).  r == 1 computes
 * the dense prefill of every layer.  taps: residual rows captured at layer boundaries
 * (kvb_layer_taps), or NULL.  Device-side checks: a token id outside [0, vocab) embeds
 * as a zero row and a forced_sel entry outside [0, n_ctx) is replaced by row 0; both
 * record KVB_ERR_INVALID_ARG in the workspace status word (kvb_device_status), and a V
 * value of the chunk caches outside fp16's range records KVB_ERR_RANGE; the results of
 * such a call are not meaningful.  Errors: INVALID_ARG, WORKSPACE, CUDA. */
kvb_status kvb_selective_prefill(const kvb_config* cfg, const kvb_model* model,
                                 const kvb_rope_table* rope,
                                 const uint16_t* k_chunks, const uint16_t* v_chunks,
                                 kvb_kv_cache* cache,
                                 const int32_t* token_ids, const int32_t* chunk_start,
                                 int32_t n_chunks, int64_t n_ctx, int64_t n_query,
                                 float r, int32_t check_layer,
                                 const int32_t* forced_sel, int64_t forced_k,
                                 float* final_hidden, int32_t* sel_out,
                                 kvb_timings* t, const kvb_layer_taps* taps,
                                 void* ws, size_t ws_bytes, void* stream);

/* The same prefill with the chunk caches in pinned HOST memory, ingested layer by layer
 * while the model computes (Sec. 3.4: KV caches are transferred to the GPU, merged and
 * position-adjusted layer by layer, overlapped with the recompute through CUDA streams).
 * For every cached layer l the library copies layer l of k_chunks_host / v_chunks_host
 * into one of two device staging slots on `copy_stream`, merges and re-aligns it into
 * `cache` there, and makes `stream` wait for that layer only just before it first reads
 * or writes cache layer l; layer 0 (and every layer before check_layer) needs no cache, so
 * the ingest runs under its compute.  k_chunks_host / v_chunks_host: pinned host memory
 * (cudaHostAlloc or registered), [n_layers][n_ctx][Hkv][D], K and V bf16.  copy_stream:
 * a stream other than `stream`.  Workspace: kvb_workspace_size_pipelined(cfg, n_ctx +
 * n_query, n_ctx) bytes (the staging slots follow the regular layout).  All other
 * arguments and results as kvb_selective_prefill; realign_ms in `t` is 0 here because the
 * merge runs on copy_stream.  Errors: as kvb_selective_prefill, INVALID_ARG if the chunk
 * caches are not pinned host memory or copy_stream == stream. */
kvb_status kvb_selective_prefill_host(const kvb_config* cfg, const kvb_model* model,
                                      const kvb_rope_table* rope,
                                      const uint16_t* k_chunks_host, const uint16_t* v_chunks_host,
                                      kvb_kv_cache* cache,
                                      const int32_t* token_ids, const int32_t* chunk_start,
                                      int32_t n_chunks, int64_t n_ctx, int64_t n_query,
                                      float r, int32_t check_layer,
                                      const int32_t* forced_sel, int64_t forced_k,
                                      float* final_hidden, int32_t* sel_out,
                                      kvb_timings* t, const kvb_layer_taps* taps,
                                      void* ws, size_t ws_bytes,
                                      void* stream, void* copy_stream);

/* Workspace bytes for kvb_selective_prefill_host: kvb_workspace_size(cfg, n_rows) plus two
 * staging slots of one layer of chunk K and V for n_ctx rows. */
kvb_status kvb_workspace_size_pipelined(const kvb_config* cfg, int64_t n_rows, int64_t n_ctx, size_t* bytes);

/* Dense causal prefill of n rows through every layer (the r = 1 comparator, Sec. 4;
 * also the per-chunk isolated prefill that produces chunk caches):
 *   row t attends cache rows [kv_lo[t], t] (kv_lo NULL = 0) with RoPE at rope_pos[t]
 *   (NULL = t).  With kv_lo = chunk start and rope_pos = t - chunk start every chunk
 *   is prefilled alone at chunk-local positions.
 * Writes every layer's K/V into the blended-format cache rows [0, n) and, if
 * v_chunk_out != NULL, every layer's V also in bf16 to v_chunk_out [n_layers][n][Hkv][D]
 * (so that cache->k (with n_rows == n) and v_chunk_out form a chunk cache in the format
 * kvb_selective_prefill reads).  If final_hidden != NULL, the final RMSNorm of the last
 * n_out rows goes to final_hidden [n_out][H].  taps: as for kvb_selective_prefill (every
 * layer is dense here), or NULL.  Token ids outside [0, vocab) are reported in the status
 * word as for kvb_selective_prefill.  Errors as above. */
kvb_status kvb_full_prefill(const kvb_config* cfg, const kvb_model* model,
                            const kvb_rope_table* rope, kvb_kv_cache* cache,
                            uint16_t* v_chunk_out,
                            const int32_t* token_ids, int64_t n,
                            const int32_t* rope_pos, const int32_t* kv_lo,
                            float* final_hidden, int64_t n_out,
                            kvb_timings* t, const kvb_layer_taps* taps,
                            void* ws, size_t ws_bytes, void* stream);

/* First token (the "first token" that closes time-to-first-token, Sec. 4.3): for n rows
 * of final hidden states h (fp32 [n][H], already through the final RMSNorm),
 *   logits[r][v] = h[r] . W[v]      (W: lm_head, bf16 [vocab][H]; fp32 accumulation)
 *   tokens[r]    = argmax_v logits[r][v], ties to the lower token id.
 * logits_out: fp32 [n][vocab] or NULL; tokens_out: int32 [n].  1 <= n <=
 * KVB_LMHEAD_MAX_ROWS, H <= 8192, H % 8 == 0.  Workspace: >= 256 + 8 * n bytes (the
 * status word, then one 64-bit argmax slot per row that the call clears).  Errors:
 * INVALID_ARG, WORKSPACE. */
#define KVB_LMHEAD_MAX_ROWS 4
kvb_status kvb_lm_head_argmax(const kvb_config* cfg, const uint16_t* lm_head, const float* hidden, int32_t n,
                              float* logits_out, int32_t* tokens_out, void* ws, size_t ws_bytes, void* stream);

/* Fixed-position selection of the methods the paper compares against (Sec. 2 and
 * Sec. 3.1): EPIC recomputes the 20 tokens that start at each separator position,
 * KVLink the separator tokens themselves.  Writes the union of the windows
 * [win_start[w], win_start[w] + window), cut to [0, n_ctx), as ascending context
 * indices, and their count.  The result is meant for kvb_selective_prefill's forced_sel.
 *   win_start: device int32 [n_win], any order, values may lie outside [0, n_ctx)
 *   sel_out:   device int32, room for min(n_ctx, n_win * window) indices
 *   k_out:     device int64 [1], the number of indices written
 * 0 <= n_win, 0 <= window, n_win * window < 2^31, 0 <= n_ctx < 2^31.  Workspace:
 * kvb_window_select_workspace_size bytes (the status word, then one flag byte per
 * context row).  Errors: INVALID_ARG, WORKSPACE. */
size_t kvb_window_select_workspace_size(int64_t n_ctx);
kvb_status kvb_window_select(const int32_t* win_start, int32_t n_win, int32_t window, int64_t n_ctx, int32_t* sel_out,
                             int64_t* k_out, void* ws, size_t ws_bytes, void* stream);

/* Distribution of per-token squared key differences, as in the paper's figures of the
 * deviation in the key entries (Sec. 3.2, Sec. 3.3):
 *   dev[i] = sum over the kv_dim entries of (K_a[i] - K_b[i])^2   (bf16 in, fp32 sum)
 *   hist[j] = #{ i : j == #{ e : dev[i] >= edges[e] } },  j = 0 .. n_edges
 * so for ascending edges hist[0] counts dev < edges[0], hist[j] counts
 * edges[j-1] <= dev < edges[j] and hist[n_edges] counts dev >= edges[n_edges-1].
 *   k_a, k_b: device bf16, row i at k_a + i * ld_a (ld, kv_dim multiples of 8)
 *   edges:    device fp32 [n_edges], 1 <= n_edges <= 1024
 *   dev_out:  device fp32 [n] or NULL (then the workspace holds it)
 *   hist_out: device int64 [n_edges + 1], cleared by the call
 * Workspace: >= 256 bytes, plus 4 * n rounded up to 16 when dev_out is NULL.
 * Errors: INVALID_ARG, WORKSPACE. */
kvb_status kvb_key_deviation_histogram(const uint16_t* k_a, int64_t ld_a, const uint16_t* k_b, int64_t ld_b, int64_t n,
                                       int32_t kv_dim, const float* edges, int32_t n_edges, float* dev_out,
                                       int64_t* hist_out, void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------- greedy decode
 * After the prefill, the paper generates with greedy decoding (Sec. 4): each step feeds
 * the last token through every layer at the next position, appends its K/V to the
 * cache and takes the argmax of the logits.  One step:
 *   x = embed[tokens[p]];  for each layer: the decoder block of Sec. 4's model on the
 *   single row at position p (RoPE at p; K/V written into cache row p; attention over
 *   cache rows [0, p]);  tokens[p + 1] = argmax(RMSNorm(x) * lm_head^T) (ties to the
 *   lower id);  p = p + 1.
 * `pos` (int32 [1]) and `tokens` (int32, room for max_pos + 1 ids) live in device
 * memory and are updated on the device, so consecutive steps need no host value; a
 * step needs 0 <= *pos < max_pos, otherwise it records KVB_ERR_INVALID_ARG in the
 * workspace status word (read with kvb_device_status) and writes nothing.
 * cache: rows [0, *pos) hold the prompt's blended cache (the prefill's output), at
 * least max_pos rows per layer; rope: at least max_pos positions; lm_head: bf16
 * [vocab][H]; hidden_out: fp32 [H] final hidden state of the step, or NULL.
 * Workspace: kvb_decode_workspace_size(cfg, max_pos) bytes (status word, activations,
 * per-split attention partials).  Errors: INVALID_ARG, UNSUPPORTED (hidden, mlp_dim or
 * Hq*D above 16384; head_dim 128 with 2, 4 or 8 q heads per kv head, or head_dim 64
 * with 2 or 4), WORKSPACE. */
kvb_status kvb_decode_workspace_size(const kvb_config* cfg, int64_t max_pos, size_t* bytes);
kvb_status kvb_decode_step(const kvb_config* cfg, const kvb_model* model, const kvb_rope_table* rope,
                           const kvb_kv_cache* cache, const uint16_t* lm_head, int32_t* tokens, int32_t* pos,
                           int64_t max_pos, float* hidden_out, void* ws, size_t ws_bytes, void* stream);

/* The decode step's attention alone: the new row's q (bf16 [Hq][D], RoPE applied)
 * over one layer's cache rows [0, *pos] (k_layer bf16, v_layer fp16 holding
 * bf16-precision values, both [n_rows][Hkv][D], n_rows >= max_pos); causal softmax
 * with the config's scale (kvb_attention_scale), GQA head map q head h -> kv head
 * h / (Hq/Hkv), at most 8 q heads per kv head.
 * out: bf16 [Hq][D].  Split-KV (one split per warp, all splits resident at once), merged
 * by log-sum-exp.
 * Workspace and errors as kvb_decode_step. */
kvb_status kvb_decode_attention(const kvb_config* cfg, const uint16_t* q, const uint16_t* k_layer,
                                const uint16_t* v_layer, int64_t n_rows, const int32_t* pos, int64_t max_pos,
                                uint16_t* out, void* ws, size_t ws_bytes, void* stream);

/* Synchronise `stream`, then read and clear the device status word that kernels using
 * workspace `ws` write when a bounded wait runs out or an index or value is out of range.
 * *code_out receives KVB_OK or the first device-side error code recorded
 * (KVB_ERR_TIMEOUT, KVB_ERR_INVALID_ARG, KVB_ERR_RANGE).  Errors: INVALID_ARG, CUDA. */
kvb_status kvb_device_status(void* ws, size_t ws_bytes, void* stream, int32_t* code_out);

/* Exercise the bounded-wait path (for tests; the paper has no counterpart): launch one
 * CTA that waits on an mbarrier nothing completes, giving up after limit_ns
 * (1000 <= limit_ns <= 4e9) and recording KVB_ERR_TIMEOUT in the status word of `ws`
 * exactly as a stalled pipeline in the GEMM or attention kernels would.  The CUDA
 * context stays usable.  Errors: INVALID_ARG. */
kvb_status kvb_debug_wait_timeout(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* KVBLEND_H */
