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
// Its device address is looked up once per device and kept for the life of the process,
// so the entry point must not be used on a device after cudaDeviceReset() there (the
// module is reloaded and the array may move).
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
                                                     const int32_t* kv_dst, int64_t n_kv_rows, int32_t* status_out,
                                                     void* stream) {
    // the same validation as kvb_gather_rmsnorm_qkv, so both entry points accept and reject the same inputs
    clear_last_error();
    kvb_status s = check_cfg(cfg);
    if (s != KVB_OK) return s;
    if ((s = check_weights(w)) != KVB_OK) return s;
    if (m < 0 || n_kv_rows < 0) return fail(KVB_ERR_INVALID_ARG, "m < 0 or n_kv_rows < 0");
    if (m == 0) return KVB_OK;
    const void* ptrs[] = {x, rope_pos, q_out, k_out, v_out};
    const char* names[] = {"x", "rope_pos", "q_out", "k_out", "v_out"};
    for (int i = 0; i < 5; ++i)
        if ((s = check_ptr(ptrs[i], names[i])) != KVB_OK) return s;
    if ((s = check_rope(rope, 1)) != KVB_OK) return s;
    if (status_out && !aligned16(status_out))
        return fail(KVB_ERR_INVALID_ARG, "no-alloc qkv: status_out not 16-byte aligned");
    // the one limit of its own: the normalised rows must fit the fixed scratch
    if ((size_t)m * (size_t)cfg->hidden > kNoAllocMaxElems)
        return fail(KVB_ERR_INVALID_ARG,
                    "no-alloc qkv: m * hidden = %lld exceeds the fixed scratch of %lld elements (use "
                    "kvb_gather_rmsnorm_qkv with a workspace, or split the rows)",
                    (long long)m * cfg->hidden, (long long)kNoAllocMaxElems);

    void* scratch = nullptr;
    s = scratch_address(&scratch);
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
    p.q_out = q_out; p.k_out = k_out; p.v_out = v_out; p.kv_dst = kv_dst; p.n_kv_rows = n_kv_rows;
    p.rope_pos = rope_pos; p.max_pos = rope->max_pos;
    p.cos_t = rope->cos; p.sin_t = rope->sin; p.bias = w->b_qkv; p.status = status_out;
    return launch_gemm(p, a, H, w->w_qkv, H, nullptr, st);
}
