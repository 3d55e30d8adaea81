// Allocation-free variant of kvb_gather_rmsnorm_qkv.
//
// Some callers cannot give the library any device memory of their own: a plugin
// inside a serving process whose memory pool owns all device memory and hands out
// only the tensors it manages, or a latency-critical loop that must never enter an
// allocator.  kvb_gather_rmsnorm_qkv needs scratch for the normalised rows that feed
// its GEMM; this variant keeps that scratch in a fixed array that lives in this
// file's device memory, so the caller passes only inputs and outputs.
//
// The array is sized for KVB_NOALLOC_MAX_ELEMS bf16 values (8 MiB); every GPU that
// loads the library holds it until the process exits.  All calls share it: two calls
// whose kernels overlap on the GPU (different streams without ordering) race on it.
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

// Rows x hidden of the normalised operand held in the fixed array.
constexpr size_t kNoAllocMaxElems = (size_t)KVB_NOALLOC_MAX_ELEMS;

// The fixed scratch.  In host code this name is only a stand-in for the symbol, not a
// device address; the address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) uint16_t g_noalloc_rows[kNoAllocMaxElems];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_addr[kMaxDevices] = {nullptr};

// Device address of the array on the current device, looked up once per device.
kvb_status scratch_address(void** out) {
    int dev = 0;
    kvb_status s = cuda_ok(cudaGetDevice(&dev), "no-alloc qkv: current device");
    if (s != KVB_OK) return s;
    if (dev < 0 || dev >= kMaxDevices) return fail(KVB_ERR_UNSUPPORTED, "no-alloc qkv: device id %d", dev);
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_addr[dev]) {
        void* p = nullptr;
        s = cuda_ok(cudaGetSymbolAddress(&p, g_noalloc_rows), "no-alloc qkv: scratch address");
        if (s != KVB_OK) return s;
        g_addr[dev] = p;
    }
    *out = g_addr[dev];
    return KVB_OK;
}

}  // namespace
}  // namespace kvb

using namespace kvb;

extern "C" kvb_status kvb_gather_rmsnorm_qkv_noalloc(const kvb_config* cfg, const kvb_layer_weights* w,
                                                     const kvb_rope_table* rope, const float* x,
                                                     const int32_t* row_idx, const int32_t* rope_pos, int64_t m,
                                                     uint16_t* q_out, uint16_t* k_out, uint16_t* v_out,
                                                     const int32_t* kv_dst, int32_t* status_out, void* stream) {
    if (!cfg || !w || !rope) return fail(KVB_ERR_INVALID_ARG, "no-alloc qkv: config, weights or rope table is NULL");
    if (m < 0) return fail(KVB_ERR_INVALID_ARG, "no-alloc qkv: m < 0");
    if (m == 0) return KVB_OK;
    if (cfg->hidden <= 0 || (size_t)m * (size_t)cfg->hidden > kNoAllocMaxElems)
        return fail(KVB_ERR_INVALID_ARG,
                    "no-alloc qkv: m * hidden = %lld exceeds the fixed scratch of %lld elements (use "
                    "kvb_gather_rmsnorm_qkv with a workspace, or split the rows)",
                    (long long)m * cfg->hidden, (long long)kNoAllocMaxElems);
    if (cfg->head_dim != 64 && cfg->head_dim != 128)
        return fail(KVB_ERR_UNSUPPORTED, "no-alloc qkv: head_dim %d not built", cfg->head_dim);
    if (cfg->n_kv_heads <= 0 || cfg->n_q_heads % cfg->n_kv_heads || cfg->hidden % 256)
        return fail(KVB_ERR_UNSUPPORTED, "no-alloc qkv: unsupported head counts or hidden size");
    const void* ptrs[] = {w->attn_norm, w->w_qkv, x, rope_pos, q_out, k_out, v_out, rope->cos, rope->sin};
    for (const void* p : ptrs)
        if (!p || !aligned16(p)) return fail(KVB_ERR_INVALID_ARG, "no-alloc qkv: NULL or misaligned pointer");
    if (status_out && !aligned16(status_out))
        return fail(KVB_ERR_INVALID_ARG, "no-alloc qkv: status_out not 16-byte aligned");
    if (w->b_qkv && !aligned16(w->b_qkv)) return fail(KVB_ERR_INVALID_ARG, "no-alloc qkv: b_qkv not 16-byte aligned");

    void* scratch = nullptr;
    kvb_status s = scratch_address(&scratch);
    if (s != KVB_OK) return s;
    uint16_t* a = static_cast<uint16_t*>(scratch);
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    const int H = cfg->hidden, D = cfg->head_dim;
    const int QD = cfg->n_q_heads * D, KVD = cfg->n_kv_heads * D;
    s = launch_rmsnorm(x, row_idx, m, H, w->attn_norm, cfg->rms_eps, a, nullptr, st);
    if (s != KVB_OK) return s;
    GemmParams p{};
    p.M = m; p.N = QD + 2 * KVD; p.K = H; p.epi = EPI_QKV;
    p.col_base = 0; p.q_dim = QD; p.kv_dim = KVD; p.head_dim = D;
    p.q_out = q_out; p.k_out = k_out; p.v_out = v_out; p.kv_dst = kv_dst; p.rope_pos = rope_pos;
    p.cos_t = rope->cos; p.sin_t = rope->sin; p.bias = w->b_qkv; p.status = status_out;
    return launch_gemm(p, a, H, w->w_qkv, H, nullptr, st);
}
