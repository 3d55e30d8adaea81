// Host-side internals shared by the translation units of libkvblend.
#pragma once

#include <atomic>

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kvblend.h"

namespace kvb {

// Record a message for kvb_last_error() and return the status.
kvb_status fail(kvb_status s, const char* fmt, ...);
// Clear the calling thread's kvb_last_error() message (every entry point does this first).
void clear_last_error();
// Argument checks shared by the entry points; each records a message when it fails.
kvb_status check_cfg(const kvb_config* c);
kvb_status check_ptr(const void* p, const char* name);
kvb_status check_weights(const kvb_layer_weights* w);
kvb_status check_rope(const kvb_rope_table* r, int64_t need_pos);
// KVB_OK, or KVB_ERR_CUDA with the CUDA error text.
kvb_status cuda_ok(cudaError_t e, const char* what);
// Raises `kernel`'s dynamic shared-memory limit to `bytes` on the current device the first time
// it is needed there (the attribute is per device); `done` is the caller's per-kernel mask of
// devices already set.  Thread-safe: a race only repeats the idempotent call.
kvb_status ensure_smem_limit(const void* kernel, int bytes, std::atomic<uint64_t>& done, const char* what);
int num_sms();
// Counts kernels the library launched (for the prefill's launch report).
void count_launch();
int64_t launch_count();
bool aligned16(const void* p);

// Tensor map for a row-major bf16 matrix [rows][cols] (row stride ld elements),
// box [box_rows][box_cols], 128-byte swizzle.
kvb_status make_tmap_2d(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld,
                        uint32_t box_cols, uint32_t box_rows,
                        CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16);
// Tensor map over [d2][d1][d0] bf16 (dense), box [b2][b1][b0], 128-byte swizzle.
kvb_status make_tmap_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                        uint32_t b0, uint32_t b1, uint32_t b2);

// ---------------------------------------------------------------- GEMM (tcgen05)

enum GemmEpi : int { EPI_QKV = 0, EPI_RESID = 1, EPI_SWIGLU = 2 };

struct GemmParams {
    int64_t M, N, K;
    int epi;
    // EPI_QKV: output column c of this GEMM is column col_base + c of [q | k | v]
    int col_base, q_dim, kv_dim, head_dim;
    uint16_t* q_out;
    uint16_t* k_out;
    uint16_t* v_out;
    const int32_t* kv_dst;
    int64_t n_kv_rows;            // rows k_out / v_out hold: a row whose destination (kv_dst[r], or r)
                                  // lies outside [0, n_kv_rows) writes no k / v and is reported
    uint16_t* v_out_bf16;         // optional second copy of v in bf16 (the chunk-cache format), same rows
    const int32_t* rope_pos;
    int64_t max_pos;              // rows of the RoPE tables: a position outside [0, max_pos) is reported
                                  // and rotated by position 0
    const float* cos_t;
    const float* sin_t;
    const float* bias;            // fp32 bias of the [q | k | v] columns (added before RoPE), or NULL
    // EPI_RESID: x[r][c] += acc
    float* x;
    int64_t ldx;
    // EPI_SWIGLU: out[r][c] = silu(gate) * up
    uint16_t* out;
    int64_t ldo;
    int* status;
};

// C = A B^T with A [M][K] (row stride lda), B [N][K] (row stride ldb); for EPI_SWIGLU
// B is the gate matrix and B2 the up matrix, both [N][K].
kvb_status launch_gemm(const GemmParams& p, const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                       const uint16_t* B2, cudaStream_t st);

// ---------------------------------------------------------------- attention (tcgen05)

struct AttnParams {
    const int32_t* q_idx;
    const int32_t* kv_lo;
    int64_t m, n_kv;
    int Hq, Hkv, D;
    uint16_t* out;
    float scale_log2;
    int* status;
};
kvb_status launch_attn(const AttnParams& p, const uint16_t* q, const uint16_t* k_cache, const uint16_t* v_cache,
                       cudaStream_t st);

// ---------------------------------------------------------------- memory-bound kernels

// K rotated by the chunk offset (bf16 -> bf16); V converted from the chunk caches' bf16 to the
// blended cache's fp16 containers (a value outside fp16's finite range records KVB_ERR_RANGE
// in *status and is written saturated to +-65504)
kvb_status launch_realign(const float* cos_t, const float* sin_t, int D, int Hkv, const uint16_t* k_src,
                          const uint16_t* v_src, int64_t src_layer_stride, uint16_t* k_dst, uint16_t* v_dst,
                          int64_t dst_layer_stride, int n_layers, const int32_t* chunk_start, int n_chunks,
                          int64_t n_ctx, int* status, cudaStream_t st);
// token ids outside [0, vocab) give a zero row and KVB_ERR_INVALID_ARG in *status
kvb_status launch_embed(const uint16_t* embed, const int32_t* tok, int64_t n, int H, int vocab, float* x,
                        int* status, cudaStream_t st);
// out_bf16[r] / out_f32[r] = RMSNorm(x[idx ? idx[r] : r]) * g   (one of the outputs may be NULL)
kvb_status launch_rmsnorm(const float* x, const int32_t* idx, int64_t m, int H, const float* g, float eps,
                          uint16_t* out_bf16, float* out_f32, cudaStream_t st);
kvb_status launch_gather_rows(const float* src, const int32_t* idx, int64_t m, int H, float* dst, cudaStream_t st);
// rows with dst_idx outside [0, n_dst) are skipped
kvb_status launch_scatter(const uint16_t* k_rows, const uint16_t* v_rows, const int32_t* dst_idx, int64_t m,
                          int kv_dim, uint16_t* k_dst, uint16_t* v_dst, int64_t n_dst, cudaStream_t st);
kvb_status launch_iota(int32_t* out, int64_t n, int32_t start, cudaStream_t st);
// sel entries outside [0, n_ctx) become row 0 and KVB_ERR_INVALID_ARG in *status
kvb_status launch_concat_rows(const int32_t* sel, int64_t k, int64_t n_ctx, int64_t n_query, int32_t* rows,
                              int* status, cudaStream_t st);

// ---------------------------------------------------------------- HKVD + top-k
size_t hkvd_ws_bytes(int64_t n_ctx);
kvb_status launch_hkvd(const uint16_t* k_fresh, int64_t ld_fresh, const uint16_t* k_cached, int64_t ld_cached,
                       int64_t n_ctx, int kv_dim, int64_t k, int32_t* sel_out, float* dev_out, void* scratch,
                       cudaStream_t st);

kvb_status launch_wait_timeout(int* status, uint64_t limit_ns, cudaStream_t st);
kvb_status launch_deviation(const uint16_t* ka, int64_t lda, const uint16_t* kb, int64_t ldb, int64_t n, int kv_dim,
                            float* dev, cudaStream_t st);
kvb_status launch_window_select(const int32_t* win_start, int32_t n_win, int32_t window, int64_t n_ctx,
                                uint8_t* flags, int32_t* sel, int64_t* k_out, cudaStream_t st);
kvb_status launch_deviation_histogram(const uint16_t* ka, int64_t lda, const uint16_t* kb, int64_t ldb, int64_t n,
                                      int kv_dim, const float* edges, int n_edges, float* dev,
                                      unsigned long long* hist, cudaStream_t st);
// ---------------------------------------------------------------- greedy decode
constexpr int KVB_DECODE_MAX_K = 16384;          // longest input row of a decode GEMV (shared memory)
enum GemvMode { GEMV_QKV = 0, GEMV_RESID = 1, GEMV_SWIGLU = 2 };
struct GemvArgs {
    const uint16_t* W;            // [N][K] bf16 (QKV: w_qkv; SwiGLU: gate rows)
    const uint16_t* W2;           // SwiGLU: up rows [N][K]
    const float* bias;            // QKV: fp32 bias per w_qkv row (added before RoPE), or NULL
    int64_t N;                    // output rows (RESID, SWIGLU)
    int K;
    const uint16_t* a;            // RESID: bf16 input row [K]
    const float* x;               // QKV, SWIGLU: fp32 residual row [K] (RMSNorm prologue)
    const float* g;               // its RMSNorm gain [K]
    float eps;
    float* y_f32;                 // RESID: x += y
    uint16_t* y_bf16;             // SWIGLU: h (bf16 [N])
    const int32_t* pos;           // QKV: position (device), 0 <= pos < max_pos
    int64_t max_pos;
    const float *cos_t, *sin_t;   // QKV: RoPE tables [max_pos][D/2]
    int D, Hq, Hkv;
    uint16_t* q_out;              // QKV: bf16 [Hq][D]
    uint16_t *k_layer, *v_layer;  // QKV: this layer's cache [n_rows][Hkv][D]
    int* status;
};
int decode_splits(int64_t max_pos, int Hkv);
kvb_status launch_decode_embed(const uint16_t* embed, const int32_t* tokens, const int32_t* pos, int64_t max_pos,
                               int64_t vocab, int H, float* x, int* status, cudaStream_t st);
kvb_status launch_gemv(int mode, const GemvArgs& p, cudaStream_t st);
kvb_status launch_decode_attn(const uint16_t* q, const uint16_t* kc, const uint16_t* vc, int Hq, int Hkv, int D,
                              const int32_t* pos, int64_t max_pos, float sl2, float* pm, float* pl, float* po,
                              uint16_t* out, int* status, cudaStream_t st);
kvb_status launch_decode_finish(const int32_t* tok, int32_t* tokens, int32_t* pos, int64_t max_pos, int* status,
                                cudaStream_t st);
kvb_status launch_lmhead(const uint16_t* W, int64_t vocab, int H, const float* x, int n, float* logits,
                         unsigned long long* keys, int32_t* tokens, cudaStream_t st);

// ---------------------------------------------------------------- workspace
// Layout of a caller workspace for up to n rows.
struct Workspace {
    int* status;       // device status word (first 256 bytes)
    float* x_all;      // [n][H] fp32 residual, all rows
    float* x_sel;      // [n][H] fp32 residual, recomputed rows
    uint16_t* a;       // [n][H] bf16 normalised rows (GEMM A operand)
    uint16_t* q;       // [n][Hq D] bf16
    uint16_t* attn;    // [n][Hq D] bf16
    uint16_t* h;       // [n][F] bf16 SwiGLU output
    uint16_t* k_fresh; // [n][Hkv D] bf16 check-layer keys
    float* dev;        // [n] fp32 deviation
    int32_t* rows;     // [n] recomputed row indices
    int32_t* ident;    // [n] 0..n-1
    int32_t* sel;      // [n] selected indices
    void* topk;        // top-k scratch
    size_t bytes;
};
size_t workspace_layout(const kvb_config* cfg, int64_t n, void* base, Workspace* w);

}  // namespace kvb
