// C ABI of libkvblend: argument validation, workspace layout, tensor maps, and the
// orchestration of the selective-recompute prefill (all on the caller's stream,
// no host synchronisation inside the path).
#include <cudaTypedefs.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "internal.h"

namespace kvb {

static thread_local char g_err[512] = "";

kvb_status fail(kvb_status s, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

void clear_last_error() { g_err[0] = 0; }

kvb_status cuda_ok(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return KVB_OK;
    return fail(KVB_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

int num_sms() {
    static std::atomic<int> cache[64];   // 0 = not looked up yet; callers may be on several threads
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    int n = cache[dev].load(std::memory_order_relaxed);
    if (n == 0) {
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
        cache[dev].store(n, std::memory_order_relaxed);
    }
    return n;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

static std::atomic<int64_t> g_launches{0};
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
int64_t launch_count() { return g_launches.load(std::memory_order_relaxed); }

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

kvb_status make_tmap_2d(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld,
                        uint32_t box_cols, uint32_t box_rows, CUtensorMapDataType dtype) {
    auto fn = encode_fn();
    if (!fn) return fail(KVB_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {ld * 2};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(m, dtype, 2, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(KVB_ERR_INVALID_ARG, "tensor map (2d %llu x %llu, ld %llu) rejected: CUresult %d",
                    (unsigned long long)rows, (unsigned long long)cols, (unsigned long long)ld, (int)r);
    return KVB_OK;
}

kvb_status make_tmap_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint32_t b0,
                        uint32_t b1, uint32_t b2) {
    auto fn = encode_fn();
    if (!fn) return fail(KVB_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    cuuint64_t dims[3] = {d0, d1, d2};
    cuuint64_t strides[2] = {d0 * 2, d0 * d1 * 2};
    cuuint32_t box[3] = {b0, b1, b2};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(KVB_ERR_INVALID_ARG, "tensor map (3d) rejected: CUresult %d", (int)r);
    return KVB_OK;
}

kvb_status ensure_smem_limit(const void* kernel, int bytes, std::atomic<uint64_t>& done, const char* what) {
    int dev = 0;
    kvb_status s = cuda_ok(cudaGetDevice(&dev), what);
    if (s != KVB_OK) return s;
    const uint64_t bit = 1ull << (dev & 63);
    if (done.load(std::memory_order_acquire) & bit) return KVB_OK;
    s = cuda_ok(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes), what);
    if (s == KVB_OK) done.fetch_or(bit, std::memory_order_release);
    return s;
}

static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

size_t workspace_layout(const kvb_config* c, int64_t n, void* base, Workspace* w) {
    size_t off = 0;
    char* b = static_cast<char*>(base);
    auto take = [&](size_t bytes) -> void* {
        void* p = b ? b + off : nullptr;
        off = align_up(off + bytes, 256);
        return p;
    };
    const size_t N = (size_t)(n > 0 ? n : 1);
    const size_t H = c->hidden, QD = (size_t)c->n_q_heads * c->head_dim, KVD = (size_t)c->n_kv_heads * c->head_dim;
    w->status = static_cast<int*>(take(256));
    w->x_all = static_cast<float*>(take(N * H * 4));
    w->x_sel = static_cast<float*>(take(N * H * 4));
    w->a = static_cast<uint16_t*>(take(N * H * 2));
    w->q = static_cast<uint16_t*>(take(N * QD * 2));
    w->attn = static_cast<uint16_t*>(take(N * QD * 2));
    w->h = static_cast<uint16_t*>(take(N * (size_t)c->mlp_dim * 2));
    w->k_fresh = static_cast<uint16_t*>(take(N * KVD * 2));
    w->dev = static_cast<float*>(take(N * 4));
    w->rows = static_cast<int32_t*>(take(N * 4));
    w->ident = static_cast<int32_t*>(take(N * 4));
    w->sel = static_cast<int32_t*>(take(N * 4));
    w->topk = take(hkvd_ws_bytes(n) + 256);
    w->bytes = off;
    return off;
}

kvb_status check_cfg(const kvb_config* c) {
    if (!c) return fail(KVB_ERR_INVALID_ARG, "config is NULL");
    if (c->hidden <= 0 || c->n_q_heads <= 0 || c->n_kv_heads <= 0 || c->head_dim <= 0 || c->mlp_dim <= 0 ||
        c->n_layers <= 0)
        return fail(KVB_ERR_INVALID_ARG, "config: sizes must be positive");
    if (c->head_dim != 64 && c->head_dim != 128)
        return fail(KVB_ERR_UNSUPPORTED, "config: head_dim %d not built (64 or 128)", c->head_dim);
    if (c->n_q_heads % c->n_kv_heads || c->n_q_heads / c->n_kv_heads > 128)
        return fail(KVB_ERR_UNSUPPORTED, "config: Hq must be a multiple of Hkv with Hq/Hkv <= 128");
    if (c->hidden % 256 || c->hidden > 8192)
        return fail(KVB_ERR_UNSUPPORTED, "config: hidden must be a multiple of 256, at most 8192");
    if (c->mlp_dim % 16) return fail(KVB_ERR_UNSUPPORTED, "config: mlp_dim must be a multiple of 16");
    if (!(c->rms_eps >= 0.f) || !(c->rope_theta > 0.f)) return fail(KVB_ERR_INVALID_ARG, "config: eps/theta");
    if (c->rope_scaling != KVB_ROPE_PLAIN && c->rope_scaling != KVB_ROPE_LLAMA3 && c->rope_scaling != KVB_ROPE_YARN)
        return fail(KVB_ERR_INVALID_ARG, "config: unknown rope_scaling %d", c->rope_scaling);
    if (c->rope_scaling != KVB_ROPE_PLAIN) {
        const float min_factor = c->rope_scaling == KVB_ROPE_YARN ? 1.f : 0.f;
        if (!(c->rs_factor >= min_factor) || !(c->rs_factor > 0.f) || !(c->rs_low > 0.f) ||
            !(c->rs_high > c->rs_low) || c->rs_orig_ctx < 1)
            return fail(KVB_ERR_INVALID_ARG, "config: rope scaling needs factor > 0 (>= 1 for YaRN), "
                        "0 < low < high and an original context >= 1");
    }
    return KVB_OK;
}

kvb_status check_ptr(const void* p, const char* name) {
    if (!p) return fail(KVB_ERR_INVALID_ARG, "%s is NULL", name);
    if (!aligned16(p)) return fail(KVB_ERR_INVALID_ARG, "%s is not 16-byte aligned", name);
    return KVB_OK;
}

kvb_status check_weights(const kvb_layer_weights* w) {
    if (!w) return fail(KVB_ERR_INVALID_ARG, "layer weights are NULL");
    kvb_status s;
    if ((s = check_ptr(w->attn_norm, "attn_norm")) || (s = check_ptr(w->w_qkv, "w_qkv")) ||
        (s = check_ptr(w->w_o, "w_o")) || (s = check_ptr(w->mlp_norm, "mlp_norm")) ||
        (s = check_ptr(w->w_gate, "w_gate")) || (s = check_ptr(w->w_up, "w_up")) ||
        (s = check_ptr(w->w_down, "w_down")))
        return s;
    if (w->b_qkv && !aligned16(w->b_qkv)) return fail(KVB_ERR_INVALID_ARG, "b_qkv is not 16-byte aligned");
    return KVB_OK;
}

kvb_status check_rope(const kvb_rope_table* r, int64_t need_pos) {
    if (!r) return fail(KVB_ERR_INVALID_ARG, "rope table is NULL");
    kvb_status s;
    if ((s = check_ptr(r->cos, "rope cos")) || (s = check_ptr(r->sin, "rope sin"))) return s;
    if (r->max_pos < need_pos)
        return fail(KVB_ERR_INVALID_ARG, "rope table covers %lld positions, %lld needed", (long long)r->max_pos,
                    (long long)need_pos);
    return KVB_OK;
}

}  // namespace kvb

using namespace kvb;

// ============================================================================ helpers

// q.k multiplier of the softmax, times log2(e) (the kernels exponentiate base 2)
static double attn_scale(const kvb_config* c) {
    double s = 1.0 / sqrt((double)c->head_dim);
    if (c->rope_scaling == KVB_ROPE_YARN) {
        const double m = 0.1 * log((double)c->rs_factor) + 1.0;   // YaRN: sqrt(1/t)
        s *= m * m;
    }
    return s;
}
static float attn_scale_log2(const kvb_config* c) {
    return (float)(1.4426950408889634 * attn_scale(c));
}

#define KVB_TRY(expr)                    \
    do {                                 \
        kvb_status _s = (expr);          \
        if (_s != KVB_OK) return _s;     \
    } while (0)

// Rotation frequency of every pair i < D/2 under the config's scaling.
static void inv_freq(const kvb_config* c, double* w) {
    const int D = c->head_dim;
    const double two_pi = 2.0 * 3.14159265358979323846;
    for (int i = 0; i < D / 2; ++i) {
        const double f = pow((double)c->rope_theta, -(2.0 * i) / D);
        if (c->rope_scaling == KVB_ROPE_PLAIN) { w[i] = f; continue; }
        const double lam = two_pi / f;   // wavelength in tokens
        if (c->rope_scaling == KVB_ROPE_LLAMA3) {
            const double hi_wl = c->rs_orig_ctx / (double)c->rs_high;   // shortest blended wavelength
            const double lo_wl = c->rs_orig_ctx / (double)c->rs_low;    // longest blended wavelength
            if (lam < hi_wl) w[i] = f;
            else if (lam > lo_wl) w[i] = f / c->rs_factor;
            else {
                const double s = (c->rs_orig_ctx / lam - c->rs_low) / ((double)c->rs_high - c->rs_low);
                w[i] = (1.0 - s) * f / c->rs_factor + s * f;
            }
        } else {
            // YaRN NTK-by-parts: r = turns of the pair over the original context; ramp
            // gamma(r) from interpolation (f / s, below alpha turns) to f (above beta)
            const double r = c->rs_orig_ctx / lam;
            const double a = c->rs_low, b = c->rs_high;
            const double gamma = r < a ? 0.0 : (r > b ? 1.0 : (r - a) / (b - a));
            w[i] = (1.0 - gamma) * f / c->rs_factor + gamma * f;
        }
    }
}

// ---------------------------------------------------------------- layer pieces

namespace {

// Per-launch CUDA event pairs around the tensor-core kernels (only when timings are asked for).
enum ProfKind { PK_ATTN_DENSE = 0, PK_ATTN_SEL = 1, PK_GEMM = 2, PK_HKVD = 3, PK_COUNT = 4 };
struct Prof {
    cudaStream_t st = nullptr;
    std::vector<cudaEvent_t> ev;
    std::vector<int> kind;
    int begin(int k) {
        cudaEvent_t a, b;
        if (cudaEventCreate(&a) != cudaSuccess) return -1;
        if (cudaEventCreate(&b) != cudaSuccess) { cudaEventDestroy(a); return -1; }
        cudaEventRecord(a, st);
        ev.push_back(a); ev.push_back(b); kind.push_back(k);
        return (int)kind.size() - 1;
    }
    void end(int i) {
        if (i >= 0) cudaEventRecord(ev[2 * i + 1], st);
    }
    void sums(float* ms, int* n) const {
        for (int k = 0; k < PK_COUNT; ++k) { ms[k] = 0.f; n[k] = 0; }
        for (size_t i = 0; i < kind.size(); ++i) {
            float t = 0.f;
            cudaEventElapsedTime(&t, ev[2 * i], ev[2 * i + 1]);
            ms[kind[i]] += t;
            n[kind[i]] += 1;
        }
    }
    ~Prof() {
        for (auto e : ev) cudaEventDestroy(e);
    }
};

struct Ctx {
    const kvb_config* c;
    const kvb_rope_table* rope;
    Workspace w;
    cudaStream_t st;
    int H, QD, KVD, D, Hq, Hkv, F;
    Prof* prof = nullptr;
};

// launch a GEMM, timed when profiling
kvb_status gemm(const Ctx& x, const GemmParams& p, const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                const uint16_t* B2) {
    const int i = x.prof ? x.prof->begin(PK_GEMM) : -1;
    kvb_status s = launch_gemm(p, A, lda, B, ldb, B2, x.st);
    if (x.prof) x.prof->end(i);
    return s;
}

Ctx make_ctx(const kvb_config* c, const kvb_rope_table* rope, const Workspace& w, void* stream) {
    Ctx x;
    x.c = c; x.rope = rope; x.w = w; x.st = static_cast<cudaStream_t>(stream);
    x.H = c->hidden; x.D = c->head_dim; x.Hq = c->n_q_heads; x.Hkv = c->n_kv_heads; x.F = c->mlp_dim;
    x.QD = x.Hq * x.D; x.KVD = x.Hkv * x.D;
    return x;
}

// a = RMSNorm(x[idx]) ; q, k, v = a W^T with RoPE; k / v rows kv_dst[r] (or r) < n_kv_rows
kvb_status qkv_rows(const Ctx& x, const kvb_layer_weights* lw, const float* xin, const int32_t* idx,
                    const int32_t* rope_pos, int64_t m, uint16_t* q, uint16_t* k, uint16_t* v, const int32_t* kv_dst,
                    int64_t n_kv_rows, uint16_t* v_bf16 = nullptr) {
    KVB_TRY(launch_rmsnorm(xin, idx, m, x.H, lw->attn_norm, x.c->rms_eps, x.w.a, nullptr, x.st));
    GemmParams p{};
    p.M = m; p.N = x.QD + 2 * x.KVD; p.K = x.H; p.epi = EPI_QKV;
    p.col_base = 0; p.q_dim = x.QD; p.kv_dim = x.KVD; p.head_dim = x.D;
    p.q_out = q; p.k_out = k; p.v_out = v; p.kv_dst = kv_dst; p.n_kv_rows = n_kv_rows; p.v_out_bf16 = v_bf16;
    p.rope_pos = rope_pos; p.max_pos = x.rope->max_pos;
    p.cos_t = x.rope->cos; p.sin_t = x.rope->sin; p.bias = lw->b_qkv; p.status = x.w.status;
    return gemm(x, p, x.w.a, x.H, lw->w_qkv, x.H, nullptr);
}

// x += attn W_o^T ; x += W_d(silu(W_g n) * W_u n), n = RMSNorm(x)
kvb_status mlp_rows(const Ctx& x, const kvb_layer_weights* lw, const uint16_t* attn, int64_t m, float* xio) {
    GemmParams p{};
    p.M = m; p.N = x.H; p.K = x.QD; p.epi = EPI_RESID; p.x = xio; p.ldx = x.H; p.status = x.w.status;
    KVB_TRY(gemm(x, p, attn, x.QD, lw->w_o, x.QD, nullptr));
    KVB_TRY(launch_rmsnorm(xio, nullptr, m, x.H, lw->mlp_norm, x.c->rms_eps, x.w.a, nullptr, x.st));
    GemmParams g{};
    g.M = m; g.N = x.F; g.K = x.H; g.epi = EPI_SWIGLU; g.out = x.w.h; g.ldo = x.F; g.status = x.w.status;
    KVB_TRY(gemm(x, g, x.w.a, x.H, lw->w_gate, x.H, lw->w_up));
    GemmParams d{};
    d.M = m; d.N = x.H; d.K = x.F; d.epi = EPI_RESID; d.x = xio; d.ldx = x.H; d.status = x.w.status;
    return gemm(x, d, x.w.h, x.F, lw->w_down, x.F, nullptr);
}

kvb_status attn_rows(const Ctx& x, const uint16_t* q, const int32_t* q_idx, const int32_t* kv_lo, int64_t m,
                     const uint16_t* kc, const uint16_t* vc, int64_t n_kv, uint16_t* out, bool selective = false) {
    AttnParams a{};
    a.q_idx = q_idx; a.kv_lo = kv_lo; a.m = m; a.n_kv = n_kv;
    a.Hq = x.Hq; a.Hkv = x.Hkv; a.D = x.D; a.out = out;
    a.scale_log2 = attn_scale_log2(x.c);
    a.status = x.w.status;
    const int i = x.prof ? x.prof->begin(selective ? PK_ATTN_SEL : PK_ATTN_DENSE) : -1;
    kvb_status s = launch_attn(a, q, kc, vc, x.st);
    if (x.prof) x.prof->end(i);
    return s;
}

// one decoder layer over m rows whose residual is the dense buffer xio [m][H]
//   row r: cache row kv_row[r] (NULL: r), RoPE position rope_pos[r], keys [kv_lo[r], kv_row[r]];
//   v_bf16: optional bf16 copy of the layer's V rows (chunk-cache format)
kvb_status layer(const Ctx& x, const kvb_layer_weights* lw, float* xio, int64_t m, const int32_t* kv_row,
                 const int32_t* rope_pos, const int32_t* kv_lo, uint16_t* kc, uint16_t* vc, int64_t n_kv,
                 uint16_t* v_bf16 = nullptr) {
    KVB_TRY(qkv_rows(x, lw, xio, nullptr, rope_pos, m, x.w.q, kc, vc, kv_row, n_kv, v_bf16));
    KVB_TRY(attn_rows(x, x.w.q, kv_row ? kv_row : x.w.ident, kv_lo, m, kc, vc, n_kv, x.w.attn, kv_row != nullptr));
    return mlp_rows(x, lw, x.w.attn, m, xio);
}

struct Timer {
    cudaEvent_t ev[8] = {};
    int n = 0;
    bool on = false;
    cudaStream_t st = nullptr;
    void start(bool enable, cudaStream_t s) {
        on = enable; st = s;
        if (!on) return;
        for (auto& e : ev) cudaEventCreate(&e);
        mark();
    }
    void mark() {
        if (on && n < 8) cudaEventRecord(ev[n++], st);
    }
    float ms(int a, int b) {
        float t = 0.f;
        if (on && b < n) cudaEventElapsedTime(&t, ev[a], ev[b]);
        return t;
    }
    ~Timer() {
        if (on)
            for (auto& e : ev) cudaEventDestroy(e);
    }
};

// Layer-boundary captures of the residual rows (kvb_layer_taps).
struct Taps {
    const kvb_layer_taps* t = nullptr;
    int H = 0;
    cudaStream_t st = nullptr;
    // copy `rows` residual rows entering layer l (n_layers: leaving the last one) into every slot asking for l
    kvb_status at(int l, const float* x, int64_t rows) const {
        if (!t) return KVB_OK;
        for (int i = 0; i < t->n; ++i) {
            if (t->layers[i] != l) continue;
            KVB_TRY(cuda_ok(cudaMemcpyAsync(t->x_out + (size_t)i * t->rows_cap * H, x, (size_t)rows * H * 4,
                                            cudaMemcpyDeviceToDevice, st), "layer tap copy"));
            if (t->rows_out) t->rows_out[i] = rows;
        }
        return KVB_OK;
    }
};

// Validates taps against the rows each boundary carries: layers below `first_sel` (and the
// end, when first_sel == n_layers) carry n_dense rows, the others n_sel.
kvb_status check_taps(const kvb_layer_taps* t, int n_layers, int first_sel, int64_t n_dense, int64_t n_sel) {
    if (!t || t->n == 0) return KVB_OK;
    if (t->n < 0 || !t->layers || t->rows_cap < 0) return fail(KVB_ERR_INVALID_ARG, "taps: bad count, layers or rows_cap");
    KVB_TRY(check_ptr(t->x_out, "taps x_out"));
    for (int i = 0; i < t->n; ++i) {
        const int l = t->layers[i];
        if (l < 0 || l > n_layers) return fail(KVB_ERR_INVALID_ARG, "taps: layer %d not in [0, %d]", l, n_layers);
        const int64_t need = (l < first_sel || first_sel >= n_layers) ? n_dense : n_sel;
        if (need > t->rows_cap)
            return fail(KVB_ERR_INVALID_ARG, "taps: layer %d carries %lld rows, rows_cap is %lld", l,
                        (long long)need, (long long)t->rows_cap);
    }
    return KVB_OK;
}

}  // namespace

static void fill_kernel_times(const Prof& prof, kvb_timings* t, int64_t launches) {
    float ms[PK_COUNT];
    int n[PK_COUNT];
    prof.sums(ms, n);
    t->attn_dense_ms = ms[PK_ATTN_DENSE];
    t->attn_sel_ms = ms[PK_ATTN_SEL];
    t->gemm_ms = ms[PK_GEMM];
    t->hkvd_ms = ms[PK_HKVD];
    t->n_attn_dense = n[PK_ATTN_DENSE];
    t->n_attn_sel = n[PK_ATTN_SEL];
    t->n_gemm = n[PK_GEMM];
    t->n_launches = (int32_t)launches;
}

// ============================================================================ ABI

extern "C" {

const char* kvb_status_string(kvb_status s) {
    switch (s) {
        case KVB_OK: return "ok";
        case KVB_ERR_INVALID_ARG: return "invalid argument";
        case KVB_ERR_UNSUPPORTED: return "unsupported";
        case KVB_ERR_CUDA: return "CUDA error";
        case KVB_ERR_TIMEOUT: return "device wait timed out";
        case KVB_ERR_WORKSPACE: return "workspace too small";
        case KVB_ERR_RANGE: return "value out of range";
        default: return "unknown status";
    }
}

const char* kvb_last_error(void) { return g_err; }

int32_t kvb_version(void) { return 300; }

kvb_status kvb_rope_table_fill(const kvb_config* cfg, int64_t max_pos, float* cos_host, float* sin_host) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    if (max_pos < 1 || !cos_host || !sin_host) return fail(KVB_ERR_INVALID_ARG, "rope table: bad size or pointer");
    const int half = cfg->head_dim / 2;
    double w[64];
    inv_freq(cfg, w);
    for (int64_t p = 0; p < max_pos; ++p)
        for (int i = 0; i < half; ++i) {
            const double a = (double)p * w[i];
            cos_host[p * half + i] = (float)cos(a);
            sin_host[p * half + i] = (float)sin(a);
        }
    return KVB_OK;
}

kvb_status kvb_attention_scale(const kvb_config* cfg, float* scale_out) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    if (!scale_out) return fail(KVB_ERR_INVALID_ARG, "attention scale: NULL output");
    *scale_out = (float)attn_scale(cfg);
    return KVB_OK;
}

kvb_status kvb_rope_realign(const kvb_config* cfg, const kvb_rope_table* rope, const uint16_t* k_src,
                            const uint16_t* v_src, int64_t src_rows, uint16_t* k_dst, uint16_t* v_dst,
                            int64_t dst_rows, int32_t layer_begin, int32_t layer_end, const int32_t* chunk_start,
                            int32_t n_chunks, int64_t n_ctx, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    if (layer_begin < 0 || layer_end < layer_begin || layer_end > cfg->n_layers)
        return fail(KVB_ERR_INVALID_ARG, "realign: bad layer range [%d, %d)", layer_begin, layer_end);
    if (n_ctx < 0 || src_rows < n_ctx || dst_rows < n_ctx || n_chunks < 1)
        return fail(KVB_ERR_INVALID_ARG, "realign: rows (%lld, src %lld, dst %lld) or chunks %d", (long long)n_ctx,
                    (long long)src_rows, (long long)dst_rows, n_chunks);
    if (n_ctx == 0 || layer_end == layer_begin) return KVB_OK;
    KVB_TRY(check_ptr(k_src, "k_src"));
    KVB_TRY(check_ptr(k_dst, "k_dst"));
    KVB_TRY(check_ptr(chunk_start, "chunk_start"));
    const bool with_v = v_src && v_dst;
    if (with_v) {
        KVB_TRY(check_ptr(v_src, "v_src"));
        KVB_TRY(check_ptr(v_dst, "v_dst"));
        if (!ws || ws_bytes < 256) return fail(KVB_ERR_WORKSPACE, "realign: V conversion needs a 256-byte status workspace");
    }
    if ((k_src == k_dst || (with_v && v_src == v_dst)) && src_rows != dst_rows)
        return fail(KVB_ERR_INVALID_ARG, "realign: in place needs equal strides");
    KVB_TRY(check_rope(rope, n_ctx));
    const int64_t kvd = (int64_t)cfg->n_kv_heads * cfg->head_dim;
    const int64_t lb = layer_begin;
    return launch_realign(rope->cos, rope->sin, cfg->head_dim, cfg->n_kv_heads, k_src + lb * src_rows * kvd,
                          with_v ? v_src + lb * src_rows * kvd : nullptr, src_rows * kvd, k_dst + lb * dst_rows * kvd,
                          with_v ? v_dst + lb * dst_rows * kvd : nullptr, dst_rows * kvd, layer_end - layer_begin,
                          chunk_start, n_chunks, n_ctx, with_v ? static_cast<int*>(ws) : nullptr,
                          static_cast<cudaStream_t>(stream));
}

size_t kvb_hkvd_workspace_size(int64_t n_ctx) { return hkvd_ws_bytes(n_ctx); }

kvb_status kvb_hkvd_select(const uint16_t* k_fresh, int64_t ld_fresh, const uint16_t* k_cached, int64_t ld_cached,
                           int64_t n_ctx, int32_t kv_dim, int64_t k, int32_t* sel_out, float* dev_out, void* ws,
                           size_t ws_bytes, void* stream) {
    clear_last_error();
    if (n_ctx < 0 || k < 0 || k > n_ctx) return fail(KVB_ERR_INVALID_ARG, "hkvd: need 0 <= k <= n_ctx");
    if (kv_dim <= 0 || kv_dim % 8 || ld_fresh < kv_dim || ld_cached < kv_dim || ld_fresh % 8 || ld_cached % 8)
        return fail(KVB_ERR_INVALID_ARG, "hkvd: kv_dim and leading dims must be multiples of 8");
    if (n_ctx > 0x7FFFFFFF) return fail(KVB_ERR_INVALID_ARG, "hkvd: n_ctx too large");
    if (n_ctx == 0) return KVB_OK;
    KVB_TRY(check_ptr(k_fresh, "k_fresh"));
    KVB_TRY(check_ptr(k_cached, "k_cached"));
    KVB_TRY(check_ptr(dev_out, "dev_out"));
    if (k > 0) KVB_TRY(check_ptr(sel_out, "sel_out"));
    const size_t need = hkvd_ws_bytes(n_ctx);
    if (ws_bytes < need || (need && !ws)) return fail(KVB_ERR_WORKSPACE, "hkvd: workspace %zu < %zu", ws_bytes, need);
    return launch_hkvd(k_fresh, ld_fresh, k_cached, ld_cached, n_ctx, kv_dim, k, sel_out, dev_out, ws,
                       static_cast<cudaStream_t>(stream));
}

kvb_status kvb_workspace_size(const kvb_config* cfg, int64_t n_rows, size_t* bytes) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    if (!bytes || n_rows < 0) return fail(KVB_ERR_INVALID_ARG, "workspace size: bad arguments");
    Workspace w;
    *bytes = workspace_layout(cfg, n_rows, nullptr, &w);
    return KVB_OK;
}

static kvb_status carve(const kvb_config* cfg, int64_t n, void* ws, size_t ws_bytes, Workspace* w) {
    const size_t need = workspace_layout(cfg, n, nullptr, w);
    if (!ws || ws_bytes < need) return fail(KVB_ERR_WORKSPACE, "workspace %zu bytes < %zu needed", ws_bytes, need);
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return fail(KVB_ERR_WORKSPACE, "workspace not 256-byte aligned");
    workspace_layout(cfg, n, ws, w);
    return KVB_OK;
}

kvb_status kvb_gather_rmsnorm_qkv(const kvb_config* cfg, const kvb_layer_weights* w, const kvb_rope_table* rope,
                                  const float* x, const int32_t* row_idx, const int32_t* rope_pos, int64_t m,
                                  uint16_t* q_out, uint16_t* k_out, uint16_t* v_out, const int32_t* kv_dst,
                                  int64_t n_kv_rows, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    KVB_TRY(check_weights(w));
    if (m < 0 || n_kv_rows < 0) return fail(KVB_ERR_INVALID_ARG, "m < 0 or n_kv_rows < 0");
    if (m == 0) return KVB_OK;
    KVB_TRY(check_ptr(x, "x"));
    KVB_TRY(check_ptr(rope_pos, "rope_pos"));
    KVB_TRY(check_ptr(q_out, "q_out"));
    KVB_TRY(check_ptr(k_out, "k_out"));
    KVB_TRY(check_ptr(v_out, "v_out"));
    KVB_TRY(check_rope(rope, 1));
    Workspace wsl;
    KVB_TRY(carve(cfg, m, ws, ws_bytes, &wsl));
    Ctx c = make_ctx(cfg, rope, wsl, stream);
    return qkv_rows(c, w, x, row_idx, rope_pos, m, q_out, k_out, v_out, kv_dst, n_kv_rows);
}

kvb_status kvb_kv_scatter(const uint16_t* k_rows, const uint16_t* v_rows, const int32_t* dst_idx, int64_t m,
                          int32_t kv_dim, uint16_t* k_dst, uint16_t* v_dst, int64_t n_dst_rows, void* stream) {
    clear_last_error();
    if (m < 0 || kv_dim <= 0 || kv_dim % 8 || m > n_dst_rows)
        return fail(KVB_ERR_INVALID_ARG, "scatter: bad sizes (m %lld, kv_dim %d, rows %lld)", (long long)m, kv_dim,
                    (long long)n_dst_rows);
    if (m == 0) return KVB_OK;
    KVB_TRY(check_ptr(k_rows, "k_rows"));
    KVB_TRY(check_ptr(v_rows, "v_rows"));
    KVB_TRY(check_ptr(dst_idx, "dst_idx"));
    KVB_TRY(check_ptr(k_dst, "k_dst"));
    KVB_TRY(check_ptr(v_dst, "v_dst"));
    return launch_scatter(k_rows, v_rows, dst_idx, m, kv_dim, k_dst, v_dst, n_dst_rows,
                          static_cast<cudaStream_t>(stream));
}

kvb_status kvb_sparse_query_attn(const kvb_config* cfg, const uint16_t* q, const int32_t* q_idx,
                                 const int32_t* kv_lo, int64_t m, const uint16_t* k_cache, const uint16_t* v_cache,
                                 int64_t n_kv, uint16_t* out, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    if (m < 0 || n_kv < 1 || n_kv > 0x7FFFFFFF) return fail(KVB_ERR_INVALID_ARG, "attention: bad sizes");
    if (m == 0) return KVB_OK;
    KVB_TRY(check_ptr(q, "q"));
    KVB_TRY(check_ptr(q_idx, "q_idx"));
    KVB_TRY(check_ptr(k_cache, "k_cache"));
    KVB_TRY(check_ptr(v_cache, "v_cache"));
    KVB_TRY(check_ptr(out, "out"));
    if (!ws || ws_bytes < 256) return fail(KVB_ERR_WORKSPACE, "attention: needs a 256-byte status workspace");
    Workspace wsl{};
    wsl.status = static_cast<int*>(ws);
    Ctx c = make_ctx(cfg, nullptr, wsl, stream);
    return attn_rows(c, q, q_idx, kv_lo, m, k_cache, v_cache, n_kv, out);
}

kvb_status kvb_mlp_rows(const kvb_config* cfg, const kvb_layer_weights* w, const uint16_t* attn, int64_t m, float* x,
                        void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    KVB_TRY(check_weights(w));
    if (m < 0) return fail(KVB_ERR_INVALID_ARG, "m < 0");
    if (m == 0) return KVB_OK;
    KVB_TRY(check_ptr(attn, "attn"));
    KVB_TRY(check_ptr(x, "x"));
    Workspace wsl;
    KVB_TRY(carve(cfg, m, ws, ws_bytes, &wsl));
    Ctx c = make_ctx(cfg, nullptr, wsl, stream);
    return mlp_rows(c, w, attn, m, x);
}

static kvb_status check_model(const kvb_config* cfg, const kvb_model* model) {
    if (!model || !model->layers) return fail(KVB_ERR_INVALID_ARG, "model or its layer array is NULL");
    KVB_TRY(check_ptr(model->embed, "embed"));
    KVB_TRY(check_ptr(model->final_norm, "final_norm"));
    for (int l = 0; l < cfg->n_layers; ++l) KVB_TRY(check_weights(&model->layers[l]));
    return KVB_OK;
}

static kvb_status check_cache(const kvb_config* cfg, const kvb_kv_cache* cache, int64_t need_rows) {
    if (!cache) return fail(KVB_ERR_INVALID_ARG, "cache is NULL");
    KVB_TRY(check_ptr(cache->k, "cache k"));
    KVB_TRY(check_ptr(cache->v, "cache v"));
    if (cache->n_layers < cfg->n_layers || cache->n_rows < need_rows)
        return fail(KVB_ERR_INVALID_ARG, "cache has %d layers x %lld rows, need %d x %lld", cache->n_layers,
                    (long long)cache->n_rows, cfg->n_layers, (long long)need_rows);
    return KVB_OK;
}

kvb_status kvb_full_prefill(const kvb_config* cfg, const kvb_model* model, const kvb_rope_table* rope,
                            kvb_kv_cache* cache, uint16_t* v_chunk_out, const int32_t* token_ids, int64_t n,
                            const int32_t* rope_pos, const int32_t* kv_lo, float* final_hidden, int64_t n_out,
                            kvb_timings* t, const kvb_layer_taps* taps, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    KVB_TRY(check_model(cfg, model));
    if (n < 1 || n > 0x7FFFFFFF || n_out < 0 || n_out > n) return fail(KVB_ERR_INVALID_ARG, "full prefill: bad n/n_out");
    KVB_TRY(check_cache(cfg, cache, n));
    KVB_TRY(check_ptr(token_ids, "token_ids"));
    KVB_TRY(check_rope(rope, rope_pos ? 1 : n));
    if (final_hidden && n_out > 0) KVB_TRY(check_ptr(final_hidden, "final_hidden"));
    if (v_chunk_out) KVB_TRY(check_ptr(v_chunk_out, "v_chunk_out"));
    KVB_TRY(check_taps(taps, cfg->n_layers, cfg->n_layers, n, n));
    Workspace w;
    KVB_TRY(carve(cfg, n, ws, ws_bytes, &w));
    Ctx c = make_ctx(cfg, rope, w, stream);
    Taps tap;
    tap.t = taps; tap.H = c.H; tap.st = c.st;
    Prof prof;
    prof.st = c.st;
    if (t) c.prof = &prof;
    const int64_t launches0 = launch_count();
    Timer tm;
    tm.start(t != nullptr, c.st);
    const int64_t kvd = c.KVD;
    KVB_TRY(launch_iota(w.ident, n, 0, c.st));
    KVB_TRY(launch_embed(model->embed, token_ids, n, c.H, cfg->vocab, w.x_all, w.status, c.st));
    for (int l = 0; l < cfg->n_layers; ++l) {
        uint16_t* kc = cache->k + (int64_t)l * cache->n_rows * kvd;
        uint16_t* vc = cache->v + (int64_t)l * cache->n_rows * kvd;
        KVB_TRY(tap.at(l, w.x_all, n));
        KVB_TRY(layer(c, &model->layers[l], w.x_all, n, nullptr, rope_pos ? rope_pos : w.ident, kv_lo, kc, vc, n,
                      v_chunk_out ? v_chunk_out + (int64_t)l * n * kvd : nullptr));
    }
    KVB_TRY(tap.at(cfg->n_layers, w.x_all, n));
    tm.mark();
    if (final_hidden && n_out > 0)
        KVB_TRY(launch_rmsnorm(w.x_all + (n - n_out) * c.H, nullptr, n_out, c.H, model->final_norm, cfg->rms_eps,
                               nullptr, final_hidden, c.st));
    tm.mark();
    if (t) {
        KVB_TRY(cuda_ok(cudaEventSynchronize(tm.ev[tm.n - 1]), "timing sync"));
        memset(t, 0, sizeof(*t));
        t->dense_ms = tm.ms(0, 1);
        t->final_ms = tm.ms(1, 2);
        t->total_ms = tm.ms(0, 2);
        t->n_selected = n;
        t->n_rows = n;
        fill_kernel_times(prof, t, launch_count() - launches0);
    }
    return KVB_OK;
}

}  // extern "C"

// Bytes of the two staging slots the pipelined (host-resident chunk caches) prefill needs:
// one layer of chunk K and V per slot.
static size_t staging_bytes(const kvb_config* c, int64_t n_ctx) {
    const size_t layer = (size_t)(n_ctx > 0 ? n_ctx : 0) * (size_t)c->n_kv_heads * c->head_dim * 2;
    return 2 * 2 * ((layer + 255) / 256 * 256);
}

// The selective prefill.  With host_src, k_chunks / v_chunks are pinned host memory:
// each cached layer is copied into one of two device staging slots on copy_st and merged
// + re-aligned there, and the compute stream waits for layer l's event just before it
// first reads or writes cache layer l (the per-layer overlap of Sec. 3.4).
static kvb_status selective_impl(const kvb_config* cfg, const kvb_model* model, const kvb_rope_table* rope,
                                 const uint16_t* k_chunks, const uint16_t* v_chunks, kvb_kv_cache* cache,
                                 const int32_t* token_ids, const int32_t* chunk_start, int32_t n_chunks, int64_t n_ctx,
                                 int64_t n_query, float r, int32_t check_layer_idx, const int32_t* forced_sel,
                                 int64_t forced_k, float* final_hidden, int32_t* sel_out, kvb_timings* t,
                                 const kvb_layer_taps* taps, void* ws, size_t ws_bytes, void* stream, bool host_src,
                                 void* copy_stream) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    KVB_TRY(check_model(cfg, model));
    const int L = cfg->n_layers;
    if (n_ctx < 0 || n_query < 0 || n_ctx + n_query < 1 || n_ctx + n_query > 0x7FFFFFFF)
        return fail(KVB_ERR_INVALID_ARG, "selective prefill: bad n_ctx/n_query");
    if (!(r >= 0.f && r <= 1.f)) return fail(KVB_ERR_INVALID_ARG, "selective prefill: r must be in [0, 1]");
    if (check_layer_idx < 1 || check_layer_idx > L)
        return fail(KVB_ERR_INVALID_ARG, "selective prefill: check_layer %d not in [1, %d]", check_layer_idx, L);
    const int64_t N = n_ctx + n_query;
    KVB_TRY(check_cache(cfg, cache, N));
    KVB_TRY(check_ptr(token_ids, "token_ids"));
    KVB_TRY(check_rope(rope, N));
    if (n_query > 0) KVB_TRY(check_ptr(final_hidden, "final_hidden"));
    if (forced_sel && (forced_k < 0 || forced_k > n_ctx))
        return fail(KVB_ERR_INVALID_ARG, "selective prefill: forced_k %lld not in [0, n_ctx]", (long long)forced_k);
    int64_t k = (int64_t)floor((double)r * (double)n_ctx + 1e-9);
    if (forced_sel) k = forced_k;
    const bool dense_all = check_layer_idx >= L || (!forced_sel && k >= n_ctx);
    KVB_TRY(check_taps(taps, L, dense_all ? L : check_layer_idx, N, k + n_query));
    if (!dense_all && n_ctx > 0) {
        KVB_TRY(check_ptr(k_chunks, "k_chunks"));
        KVB_TRY(check_ptr(v_chunks, "v_chunks"));
        KVB_TRY(check_ptr(chunk_start, "chunk_start"));
        if (n_chunks < 1) return fail(KVB_ERR_INVALID_ARG, "selective prefill: n_chunks < 1");
        if (host_src) {
            for (const void* hp : {static_cast<const void*>(k_chunks), static_cast<const void*>(v_chunks)}) {
                cudaPointerAttributes a;
                if (cudaPointerGetAttributes(&a, hp) != cudaSuccess || a.type != cudaMemoryTypeHost) {
                    cudaGetLastError();
                    return fail(KVB_ERR_INVALID_ARG, "pipelined prefill: chunk caches must be pinned host memory");
                }
            }
        }
    }
    Workspace w;
    const size_t ws_main = workspace_layout(cfg, N, nullptr, &w);
    const size_t ws_need = ws_main + (host_src ? staging_bytes(cfg, n_ctx) : 0);
    if (ws_bytes < ws_need)
        return fail(KVB_ERR_WORKSPACE, "workspace %zu bytes < %zu needed", ws_bytes, ws_need);
    KVB_TRY(carve(cfg, N, ws, ws_bytes, &w));
    Ctx c = make_ctx(cfg, rope, w, stream);
    Taps tap;
    tap.t = taps; tap.H = c.H; tap.st = c.st;
    Prof prof;
    prof.st = c.st;
    if (t) c.prof = &prof;
    const int64_t launches0 = launch_count();
    const int64_t kvd = c.KVD, rows_c = cache->n_rows;
    auto kc = [&](int l) { return cache->k + (int64_t)l * rows_c * kvd; };
    auto vc = [&](int l) { return cache->v + (int64_t)l * rows_c * kvd; };

    Timer tm;
    tm.start(t != nullptr, c.st);
    const int lc = dense_all ? L : check_layer_idx;
    // 1. merge + re-align the chunk caches of the layers that will be read as cached
    struct Events {
        std::vector<cudaEvent_t> ev;
        ~Events() {
            for (auto e : ev)
                if (e) cudaEventDestroy(e);
        }
    } ready;
    ready.ev.assign((size_t)L, nullptr);
    if (lc < L && n_ctx > 0 && !host_src) {
        KVB_TRY(launch_realign(rope->cos, rope->sin, c.D, c.Hkv, k_chunks + (int64_t)lc * n_ctx * kvd,
                               v_chunks + (int64_t)lc * n_ctx * kvd, n_ctx * kvd, kc(lc), vc(lc), rows_c * kvd,
                               L - lc, chunk_start, n_chunks, n_ctx, w.status, c.st));
    } else if (lc < L && n_ctx > 0) {
        cudaStream_t cs = static_cast<cudaStream_t>(copy_stream);
        cudaEvent_t go = nullptr;
        KVB_TRY(cuda_ok(cudaEventCreateWithFlags(&go, cudaEventDisableTiming), "pipelined prefill: event"));
        kvb_status st = cuda_ok(cudaEventRecord(go, c.st), "pipelined prefill: record");
        if (st == KVB_OK) st = cuda_ok(cudaStreamWaitEvent(cs, go, 0), "pipelined prefill: wait");
        cudaEventDestroy(go);
        KVB_TRY(st);
        const size_t layer_elems = (size_t)n_ctx * kvd;
        const size_t slot = staging_bytes(cfg, n_ctx) / 4;   // bytes of one K (or V) slot
        char* stage = static_cast<char*>(ws) + ws_main;
        for (int l = lc; l < L; ++l) {
            const int sl = (l - lc) & 1;
            uint16_t* sk = reinterpret_cast<uint16_t*>(stage + (size_t)(2 * sl) * slot);
            uint16_t* sv = reinterpret_cast<uint16_t*>(stage + (size_t)(2 * sl + 1) * slot);
            KVB_TRY(cuda_ok(cudaMemcpyAsync(sk, k_chunks + (size_t)l * layer_elems, layer_elems * 2,
                                            cudaMemcpyHostToDevice, cs), "pipelined prefill: K copy"));
            KVB_TRY(cuda_ok(cudaMemcpyAsync(sv, v_chunks + (size_t)l * layer_elems, layer_elems * 2,
                                            cudaMemcpyHostToDevice, cs), "pipelined prefill: V copy"));
            KVB_TRY(launch_realign(rope->cos, rope->sin, c.D, c.Hkv, sk, sv, (int64_t)layer_elems, kc(l), vc(l),
                                   rows_c * kvd, 1, chunk_start, n_chunks, n_ctx, w.status, cs));
            KVB_TRY(cuda_ok(cudaEventCreateWithFlags(&ready.ev[l], cudaEventDisableTiming), "pipelined prefill: event"));
            KVB_TRY(cuda_ok(cudaEventRecord(ready.ev[l], cs), "pipelined prefill: record"));
        }
    }
    auto wait_layer = [&](int l) -> kvb_status {
        if (l < 0 || l >= L || !ready.ev[l]) return KVB_OK;
        return cuda_ok(cudaStreamWaitEvent(c.st, ready.ev[l], 0), "pipelined prefill: layer wait");
    };
    tm.mark();
    // 2. dense layers (layer 0 at least): every row, causal
    KVB_TRY(launch_iota(w.ident, N, 0, c.st));
    KVB_TRY(launch_embed(model->embed, token_ids, N, c.H, cfg->vocab, w.x_all, w.status, c.st));
    for (int l = 0; l < lc; ++l) {
        KVB_TRY(tap.at(l, w.x_all, N));
        KVB_TRY(layer(c, &model->layers[l], w.x_all, N, nullptr, w.ident, nullptr, kc(l), vc(l), N));
    }
    tm.mark();
    float* x_final = w.x_all;
    int64_t m = N;
    if (lc < L) {
        // 3. check layer: fresh keys of every context row, deviation, top-k
        const int32_t* sel = forced_sel;
        if (!forced_sel) {
            if (n_ctx > 0) {
                const kvb_layer_weights* lw = &model->layers[lc];
                KVB_TRY(launch_rmsnorm(w.x_all, nullptr, n_ctx, c.H, lw->attn_norm, cfg->rms_eps, w.a, nullptr, c.st));
                GemmParams p{};
                p.M = n_ctx; p.N = c.KVD; p.K = c.H; p.epi = EPI_QKV;
                p.col_base = c.QD; p.q_dim = c.QD; p.kv_dim = c.KVD; p.head_dim = c.D;
                p.k_out = w.k_fresh; p.n_kv_rows = n_ctx; p.rope_pos = w.ident; p.max_pos = rope->max_pos;
                p.cos_t = rope->cos; p.sin_t = rope->sin;
                p.bias = lw->b_qkv; p.status = w.status;
                KVB_TRY(gemm(c, p, w.a, c.H, lw->w_qkv + (int64_t)c.QD * c.H, c.H, nullptr));
                KVB_TRY(wait_layer(lc));
                const int hp = c.prof ? c.prof->begin(PK_HKVD) : -1;
                KVB_TRY(launch_hkvd(w.k_fresh, kvd, kc(lc), kvd, n_ctx, (int)kvd, k, w.sel, w.dev, w.topk, c.st));
                if (c.prof) c.prof->end(hp);
            }
            sel = w.sel;
        }
        m = k + n_query;
        KVB_TRY(launch_concat_rows(sel, k, n_ctx, n_query, w.rows, w.status, c.st));
        KVB_TRY(launch_gather_rows(w.x_all, w.rows, m, c.H, w.x_sel, c.st));
        if (sel_out && k > 0)
            KVB_TRY(cuda_ok(cudaMemcpyAsync(sel_out, sel, (size_t)k * 4, cudaMemcpyDeviceToDevice, c.st), "sel copy"));
        tm.mark();
        // 4. selective layers over the recomputed rows
        for (int l = lc; l < L; ++l) {
            KVB_TRY(wait_layer(l));
            KVB_TRY(tap.at(l, w.x_sel, m));
            KVB_TRY(layer(c, &model->layers[l], w.x_sel, m, w.rows, w.rows, nullptr, kc(l), vc(l), N));
        }
        KVB_TRY(tap.at(L, w.x_sel, m));
        x_final = w.x_sel;
    } else {
        KVB_TRY(tap.at(L, w.x_all, N));
        if (sel_out && n_ctx > 0) KVB_TRY(launch_iota(sel_out, n_ctx, 0, c.st));
        k = n_ctx;
        tm.mark();
    }
    tm.mark();
    // 5. final RMSNorm of the query rows (the last n_query rows of either buffer)
    if (n_query > 0)
        KVB_TRY(launch_rmsnorm(x_final + (m - n_query) * c.H, nullptr, n_query, c.H, model->final_norm, cfg->rms_eps,
                               nullptr, final_hidden, c.st));
    tm.mark();
    if (t) {
        KVB_TRY(cuda_ok(cudaEventSynchronize(tm.ev[tm.n - 1]), "timing sync"));
        memset(t, 0, sizeof(*t));
        t->realign_ms = tm.ms(0, 1);
        t->dense_ms = tm.ms(1, 2);
        t->select_ms = tm.ms(2, 3);
        t->selective_ms = tm.ms(3, 4);
        t->final_ms = tm.ms(4, 5);
        t->total_ms = tm.ms(0, 5);
        t->n_selected = k;
        t->n_rows = m;
        fill_kernel_times(prof, t, launch_count() - launches0);
    }
    return KVB_OK;
}


extern "C" {

kvb_status kvb_selective_prefill(const kvb_config* cfg, const kvb_model* model, const kvb_rope_table* rope,
                                 const uint16_t* k_chunks, const uint16_t* v_chunks, kvb_kv_cache* cache,
                                 const int32_t* token_ids, const int32_t* chunk_start, int32_t n_chunks, int64_t n_ctx,
                                 int64_t n_query, float r, int32_t check_layer, const int32_t* forced_sel,
                                 int64_t forced_k, float* final_hidden, int32_t* sel_out, kvb_timings* t,
                                 const kvb_layer_taps* taps, void* ws, size_t ws_bytes, void* stream) {
    return selective_impl(cfg, model, rope, k_chunks, v_chunks, cache, token_ids, chunk_start, n_chunks, n_ctx,
                          n_query, r, check_layer, forced_sel, forced_k, final_hidden, sel_out, t, taps, ws, ws_bytes,
                          stream, false, nullptr);
}

kvb_status kvb_selective_prefill_host(const kvb_config* cfg, const kvb_model* model, const kvb_rope_table* rope,
                                      const uint16_t* k_chunks_host, const uint16_t* v_chunks_host,
                                      kvb_kv_cache* cache, const int32_t* token_ids, const int32_t* chunk_start,
                                      int32_t n_chunks, int64_t n_ctx, int64_t n_query, float r,
                                      int32_t check_layer, const int32_t* forced_sel, int64_t forced_k,
                                      float* final_hidden, int32_t* sel_out, kvb_timings* t,
                                      const kvb_layer_taps* taps, void* ws, size_t ws_bytes, void* stream,
                                      void* copy_stream) {
    clear_last_error();
    if (copy_stream == stream) return fail(KVB_ERR_INVALID_ARG, "pipelined prefill: copy_stream must differ from stream");
    return selective_impl(cfg, model, rope, k_chunks_host, v_chunks_host, cache, token_ids, chunk_start, n_chunks,
                          n_ctx, n_query, r, check_layer, forced_sel, forced_k, final_hidden, sel_out, t, taps, ws,
                          ws_bytes, stream, true, copy_stream);
}

kvb_status kvb_workspace_size_pipelined(const kvb_config* cfg, int64_t n_rows, int64_t n_ctx, size_t* bytes) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    if (!bytes || n_rows < 0 || n_ctx < 0) return fail(KVB_ERR_INVALID_ARG, "workspace size: bad arguments");
    Workspace w;
    *bytes = workspace_layout(cfg, n_rows, nullptr, &w) + staging_bytes(cfg, n_ctx);
    return KVB_OK;
}

static kvb_status check_ptr4(const void* p, const char* name) {
    if (!p) return fail(KVB_ERR_INVALID_ARG, "%s is NULL", name);
    if (reinterpret_cast<uintptr_t>(p) % 4) return fail(KVB_ERR_INVALID_ARG, "%s is not 4-byte aligned", name);
    return KVB_OK;
}

static size_t round16(size_t x) { return (x + 15) & ~(size_t)15; }

size_t kvb_window_select_workspace_size(int64_t n_ctx) { return 256 + round16(n_ctx > 0 ? (size_t)n_ctx : 0); }

kvb_status kvb_window_select(const int32_t* win_start, int32_t n_win, int32_t window, int64_t n_ctx, int32_t* sel_out,
                             int64_t* k_out, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    if (n_win < 0 || window < 0 || n_ctx < 0 || n_ctx > 0x7FFFFFFF || (int64_t)n_win * window > 0x7FFFFFFF)
        return fail(KVB_ERR_INVALID_ARG, "window select: need 0 <= n_win, window; n_win * window and n_ctx < 2^31");
    if (n_win > 0) KVB_TRY(check_ptr4(win_start, "win_start"));
    KVB_TRY(check_ptr4(sel_out, "sel_out"));
    if (!k_out || reinterpret_cast<uintptr_t>(k_out) % 8) return fail(KVB_ERR_INVALID_ARG, "k_out NULL or misaligned");
    const size_t need = kvb_window_select_workspace_size(n_ctx);
    if (!ws || ws_bytes < need) return fail(KVB_ERR_WORKSPACE, "window select: workspace %zu < %zu", ws_bytes, need);
    uint8_t* flags = static_cast<uint8_t*>(ws) + 256;
    return launch_window_select(win_start, n_win, window, n_ctx, flags, sel_out, k_out,
                                static_cast<cudaStream_t>(stream));
}

kvb_status kvb_key_deviation_histogram(const uint16_t* k_a, int64_t ld_a, const uint16_t* k_b, int64_t ld_b, int64_t n,
                                       int32_t kv_dim, const float* edges, int32_t n_edges, float* dev_out,
                                       int64_t* hist_out, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    if (n < 0 || n > 0x7FFFFFFF) return fail(KVB_ERR_INVALID_ARG, "deviation histogram: n out of range");
    if (kv_dim <= 0 || kv_dim % 8 || ld_a < kv_dim || ld_b < kv_dim || ld_a % 8 || ld_b % 8)
        return fail(KVB_ERR_INVALID_ARG, "deviation histogram: kv_dim and leading dims must be multiples of 8");
    if (n_edges < 1 || n_edges > 1024) return fail(KVB_ERR_INVALID_ARG, "deviation histogram: 1 <= n_edges <= 1024");
    KVB_TRY(check_ptr4(edges, "edges"));
    if (!hist_out || reinterpret_cast<uintptr_t>(hist_out) % 8)
        return fail(KVB_ERR_INVALID_ARG, "hist_out NULL or misaligned");
    if (n > 0) {
        KVB_TRY(check_ptr(k_a, "k_a"));
        KVB_TRY(check_ptr(k_b, "k_b"));
    }
    if (dev_out) KVB_TRY(check_ptr4(dev_out, "dev_out"));
    const size_t need = 256 + (dev_out ? 0 : round16((size_t)n * 4));
    if (!ws || ws_bytes < need) return fail(KVB_ERR_WORKSPACE, "deviation histogram: workspace %zu < %zu", ws_bytes, need);
    float* dev = dev_out ? dev_out : reinterpret_cast<float*>(static_cast<char*>(ws) + 256);
    return launch_deviation_histogram(k_a, ld_a, k_b, ld_b, n, kv_dim, edges, n_edges, dev,
                                      reinterpret_cast<unsigned long long*>(hist_out),
                                      static_cast<cudaStream_t>(stream));
}

kvb_status kvb_lm_head_argmax(const kvb_config* cfg, const uint16_t* lm_head, const float* hidden, int32_t n,
                              float* logits_out, int32_t* tokens_out, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_cfg(cfg));
    if (n < 1 || n > KVB_LMHEAD_MAX_ROWS || cfg->vocab < 1 || cfg->hidden > 8192 || cfg->hidden % 8)
        return fail(KVB_ERR_INVALID_ARG, "lm head: need 1 <= n <= %d rows, vocab >= 1, hidden <= 8192",
                    KVB_LMHEAD_MAX_ROWS);
    KVB_TRY(check_ptr(lm_head, "lm_head"));
    KVB_TRY(check_ptr(hidden, "hidden"));
    KVB_TRY(check_ptr(tokens_out, "tokens_out"));
    if (logits_out) KVB_TRY(check_ptr(logits_out, "logits_out"));
    if (!ws || ws_bytes < 256 + 8 * (size_t)n) return fail(KVB_ERR_WORKSPACE, "lm head: workspace too small");
    auto* keys = reinterpret_cast<unsigned long long*>(static_cast<char*>(ws) + 256);
    return launch_lmhead(lm_head, cfg->vocab, cfg->hidden, hidden, n, logits_out, keys, tokens_out,
                         static_cast<cudaStream_t>(stream));
}

// ------------------------------------------------------------------ greedy decode

struct DecodeWs {
    int* status;
    float *x, *hidden, *pm, *pl, *po;
    uint16_t *a, *attn, *h, *q;
    unsigned long long* keys;
    int32_t* tok;
};

static size_t decode_layout(const kvb_config* c, int64_t max_pos, void* base, DecodeWs* w) {
    size_t off = 0;
    char* b = static_cast<char*>(base);
    auto take = [&](size_t bytes) -> void* {
        void* p = b ? b + off : nullptr;
        off = align_up(off + bytes, 256);
        return p;
    };
    const int64_t H = c->hidden, F = c->mlp_dim, D = c->head_dim, Hq = c->n_q_heads, Hkv = c->n_kv_heads;
    const int64_t S = decode_splits(max_pos, (int)Hkv);   // CTA partials per q head
    w->status = static_cast<int*>(take(256));
    w->x = static_cast<float*>(take(H * 4));
    w->hidden = static_cast<float*>(take(H * 4));
    w->a = static_cast<uint16_t*>(take(H * 2));
    w->q = static_cast<uint16_t*>(take(Hq * D * 2));
    w->attn = static_cast<uint16_t*>(take(Hq * D * 2));
    w->h = static_cast<uint16_t*>(take(F * 2));
    w->keys = static_cast<unsigned long long*>(take(8));
    w->tok = static_cast<int32_t*>(take(4));
    w->pm = static_cast<float*>(take(S * Hq * 4));
    w->pl = static_cast<float*>(take(S * Hq * 4));
    w->po = static_cast<float*>(take(S * Hq * D * 4));
    return off;
}

static kvb_status check_decode(const kvb_config* cfg, int64_t max_pos) {
    KVB_TRY(check_cfg(cfg));
    if (max_pos < 1 || max_pos > 0x7FFFFFFE) return fail(KVB_ERR_INVALID_ARG, "decode: max_pos out of range");
    const int64_t qd = (int64_t)cfg->n_q_heads * cfg->head_dim;
    if (cfg->hidden > KVB_DECODE_MAX_K || cfg->mlp_dim > KVB_DECODE_MAX_K || qd > KVB_DECODE_MAX_K)
        return fail(KVB_ERR_UNSUPPORTED, "decode: hidden, mlp_dim and Hq*D must be at most %d", KVB_DECODE_MAX_K);
    if (cfg->n_q_heads / cfg->n_kv_heads > 8)
        return fail(KVB_ERR_UNSUPPORTED, "decode: at most 8 q heads per kv head (%d)", cfg->n_q_heads / cfg->n_kv_heads);
    return KVB_OK;
}

kvb_status kvb_decode_workspace_size(const kvb_config* cfg, int64_t max_pos, size_t* bytes) {
    clear_last_error();
    KVB_TRY(check_decode(cfg, max_pos));
    if (!bytes) return fail(KVB_ERR_INVALID_ARG, "decode workspace size: bytes is NULL");
    DecodeWs w;
    *bytes = decode_layout(cfg, max_pos, nullptr, &w);
    return KVB_OK;
}

kvb_status kvb_decode_attention(const kvb_config* cfg, const uint16_t* q, const uint16_t* k_layer,
                                const uint16_t* v_layer, int64_t n_rows, const int32_t* pos, int64_t max_pos,
                                uint16_t* out, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_decode(cfg, max_pos));
    if (n_rows < max_pos) return fail(KVB_ERR_INVALID_ARG, "decode attention: n_rows %lld < max_pos %lld",
                                      (long long)n_rows, (long long)max_pos);
    KVB_TRY(check_ptr(q, "q"));
    KVB_TRY(check_ptr(k_layer, "k_layer"));
    KVB_TRY(check_ptr(v_layer, "v_layer"));
    KVB_TRY(check_ptr(pos, "pos"));
    KVB_TRY(check_ptr(out, "out"));
    DecodeWs w;
    const size_t need = decode_layout(cfg, max_pos, nullptr, &w);
    if (!ws || ws_bytes < need) return fail(KVB_ERR_WORKSPACE, "decode attention: workspace %zu < %zu", ws_bytes, need);
    decode_layout(cfg, max_pos, ws, &w);
    const float sl2 = attn_scale_log2(cfg);
    return launch_decode_attn(q, k_layer, v_layer, cfg->n_q_heads, cfg->n_kv_heads, cfg->head_dim, pos, max_pos, sl2,
                              w.pm, w.pl, w.po, out, w.status, static_cast<cudaStream_t>(stream));
}

kvb_status kvb_decode_step(const kvb_config* cfg, const kvb_model* model, const kvb_rope_table* rope,
                           const kvb_kv_cache* cache, const uint16_t* lm_head, int32_t* tokens, int32_t* pos,
                           int64_t max_pos, float* hidden_out, void* ws, size_t ws_bytes, void* stream) {
    clear_last_error();
    KVB_TRY(check_decode(cfg, max_pos));
    if (cfg->vocab < 1 || cfg->hidden > 8192) return fail(KVB_ERR_UNSUPPORTED, "decode: vocab >= 1, hidden <= 8192");
    KVB_TRY(check_model(cfg, model));
    KVB_TRY(check_rope(rope, max_pos));
    KVB_TRY(check_cache(cfg, cache, max_pos));
    KVB_TRY(check_ptr(lm_head, "lm_head"));
    KVB_TRY(check_ptr(tokens, "tokens"));
    KVB_TRY(check_ptr(pos, "pos"));
    if (hidden_out) KVB_TRY(check_ptr(hidden_out, "hidden_out"));
    DecodeWs w;
    const size_t need = decode_layout(cfg, max_pos, nullptr, &w);
    if (!ws || ws_bytes < need) return fail(KVB_ERR_WORKSPACE, "decode: workspace %zu < %zu", ws_bytes, need);
    decode_layout(cfg, max_pos, ws, &w);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int H = cfg->hidden, F = cfg->mlp_dim, D = cfg->head_dim, Hq = cfg->n_q_heads, Hkv = cfg->n_kv_heads;
    const int QD = Hq * D, KVD = Hkv * D;
    const float eps = cfg->rms_eps;
    const float sl2 = attn_scale_log2(cfg);
    float* hidden = hidden_out ? hidden_out : w.hidden;
    KVB_TRY(launch_decode_embed(model->embed, tokens, pos, max_pos, cfg->vocab, H, w.x, w.status, st));
    GemvArgs ga{};
    ga.eps = eps;
    ga.pos = pos;
    ga.max_pos = max_pos;
    ga.cos_t = rope->cos;
    ga.sin_t = rope->sin;
    ga.D = D; ga.Hq = Hq; ga.Hkv = Hkv;
    ga.status = w.status;
    for (int l = 0; l < cfg->n_layers; ++l) {
        const kvb_layer_weights& lw = model->layers[l];
        uint16_t* kc = cache->k + (int64_t)l * cache->n_rows * KVD;
        uint16_t* vc = cache->v + (int64_t)l * cache->n_rows * KVD;
        GemvArgs qkv = ga;                     // RMSNorm + QKV + RoPE + K/V append
        qkv.W = lw.w_qkv; qkv.bias = lw.b_qkv; qkv.K = H; qkv.x = w.x; qkv.g = lw.attn_norm;
        qkv.q_out = w.q; qkv.k_layer = kc; qkv.v_layer = vc;
        KVB_TRY(launch_gemv(GEMV_QKV, qkv, st));
        KVB_TRY(launch_decode_attn(w.q, kc, vc, Hq, Hkv, D, pos, max_pos, sl2, w.pm, w.pl, w.po, w.attn, w.status, st));
        GemvArgs o = ga;                       // x += O-proj(attention)
        o.W = lw.w_o; o.N = H; o.K = QD; o.a = w.attn; o.y_f32 = w.x;
        KVB_TRY(launch_gemv(GEMV_RESID, o, st));
        GemvArgs mlp = ga;                     // h = SwiGLU(RMSNorm(x))
        mlp.W = lw.w_gate; mlp.W2 = lw.w_up; mlp.N = F; mlp.K = H; mlp.x = w.x; mlp.g = lw.mlp_norm; mlp.y_bf16 = w.h;
        KVB_TRY(launch_gemv(GEMV_SWIGLU, mlp, st));
        GemvArgs down = ga;                    // x += down(h)
        down.W = lw.w_down; down.N = H; down.K = F; down.a = w.h; down.y_f32 = w.x;
        KVB_TRY(launch_gemv(GEMV_RESID, down, st));
    }
    KVB_TRY(launch_rmsnorm(w.x, nullptr, 1, H, model->final_norm, eps, nullptr, hidden, st));
    KVB_TRY(launch_lmhead(lm_head, cfg->vocab, H, hidden, 1, nullptr, w.keys, w.tok, st));
    return launch_decode_finish(w.tok, tokens, pos, max_pos, w.status, st);
}

kvb_status kvb_debug_wait_timeout(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream) {
    clear_last_error();
    if (!ws || ws_bytes < 256 || limit_ns < 1000 || limit_ns > 4000000000ll)
        return fail(KVB_ERR_INVALID_ARG, "debug wait: bad workspace or limit");
    return launch_wait_timeout(static_cast<int*>(ws), (uint64_t)limit_ns, static_cast<cudaStream_t>(stream));
}

kvb_status kvb_device_status(void* ws, size_t ws_bytes, void* stream, int32_t* code_out) {
    clear_last_error();
    if (!ws || ws_bytes < 256 || !code_out) return fail(KVB_ERR_INVALID_ARG, "device status: bad arguments");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    KVB_TRY(cuda_ok(cudaStreamSynchronize(st), "device status sync"));
    int v = 0;
    KVB_TRY(cuda_ok(cudaMemcpy(&v, ws, sizeof(int), cudaMemcpyDeviceToHost), "device status read"));
    if (v != 0) KVB_TRY(cuda_ok(cudaMemset(ws, 0, sizeof(int)), "device status clear"));
    *code_out = v;
    return KVB_OK;
}

}  // extern "C"
