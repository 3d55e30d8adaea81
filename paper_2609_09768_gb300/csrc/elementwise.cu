// Memory-bound kernels of the prefill: chunk-cache merge + RoPE re-alignment,
// embedding gather, (gathered) RMSNorm, row gather/scatter.  All move data in
// 16-byte vectors with consecutive threads on consecutive addresses.
#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

// ------------------------------------------------------------------ re-alignment
// bf16 pair (chunk-cache V) -> fp16 pair (blended-cache V container).  Exact for
// 2^-14 <= |v| <= 65504 and 0 (a bf16 value has 8 significant bits, fp16 11); smaller
// magnitudes round to fp16's subnormal spacing.  |v| > 65504 cannot be held: it is
// written as +-65504 and `bad` is set; NaN stays NaN and also sets `bad`.
KVB_DEV uint32_t v_bf16x2_to_f16x2(uint32_t v, bool& bad) {
    const float a = bf16_lo(v), b = bf16_hi(v);
    bad |= !(fabsf(a) <= 65504.f) || !(fabsf(b) <= 65504.f);
    const float ca = (a != a) ? a : fminf(fmaxf(a, -65504.f), 65504.f);
    const float cb = (b != b) ? b : fminf(fmaxf(b, -65504.f), 65504.f);
    return pack_f16(ca, cb);
}
KVB_DEV uint4 v_convert16(uint4 u, bool& bad) {
    return make_uint4(v_bf16x2_to_f16x2(u.x, bad), v_bf16x2_to_f16x2(u.y, bad), v_bf16x2_to_f16x2(u.z, bad),
                      v_bf16x2_to_f16x2(u.w, bad));
}

// Thread item = (context row t, head h, group of 8 rotation pairs); the chunk
// offset and its cos/sin are looked up once and reused for every layer.  K is rotated
// (bf16 in and out), V converted from bf16 to its fp16 container in the same pass.
template <int D>
__global__ void __launch_bounds__(256)
realign_kernel(const float* __restrict__ cos_t, const float* __restrict__ sin_t, int Hkv,
               const uint16_t* k_src, const uint16_t* v_src, int64_t src_ls,   // may alias k_dst / v_dst
               uint16_t* k_dst, uint16_t* v_dst, int64_t dst_ls, int n_layers,
               const int32_t* __restrict__ chunk_start, int n_chunks, int64_t n_ctx, bool copy_v, int* status) {
    bool bad = false;
    constexpr int GPH = D / 16;   // groups of 8 pairs per head
    const int64_t per_row = (int64_t)Hkv * GPH;
    const int64_t items = n_ctx * per_row;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < items;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t t = it / per_row;
        const int w = (int)(it - t * per_row);
        const int h = w / GPH, gi = w - h * GPH;
        // chunk c with chunk_start[c] <= t < chunk_start[c+1]
        int lo = 0, hi = n_chunks;   // invariant: chunk_start[lo] <= t < chunk_start[hi]
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (__ldg(chunk_start + mid) <= t) lo = mid; else hi = mid;
        }
        const int64_t o = __ldg(chunk_start + lo);
        const float4* cp = reinterpret_cast<const float4*>(cos_t + o * (D / 2) + gi * 8);
        const float4* sp = reinterpret_cast<const float4*>(sin_t + o * (D / 2) + gi * 8);
        const float4 c0 = __ldg(cp), c1 = __ldg(cp + 1), s0 = __ldg(sp), s1 = __ldg(sp + 1);
        const float cs[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
        const float sn[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
        const int64_t off = t * Hkv * D + h * D + gi * 8;
        // four layers' loads in flight before any store (memory-level parallelism)
        constexpr int U = 4;
        for (int l0 = 0; l0 < n_layers; l0 += U) {
            uint4 ka[U], kb[U], va[U], vb[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (l0 + u < n_layers) {
                    const int64_t o = (int64_t)(l0 + u) * src_ls + off;
                    ka[u] = __ldcs(reinterpret_cast<const uint4*>(k_src + o));
                    kb[u] = __ldcs(reinterpret_cast<const uint4*>(k_src + o + D / 2));
                    if (copy_v) {
                        va[u] = __ldcs(reinterpret_cast<const uint4*>(v_src + o));
                        vb[u] = __ldcs(reinterpret_cast<const uint4*>(v_src + o + D / 2));
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                if (l0 + u < n_layers) {
                    const uint32_t av[4] = {ka[u].x, ka[u].y, ka[u].z, ka[u].w};
                    const uint32_t bv[4] = {kb[u].x, kb[u].y, kb[u].z, kb[u].w};
                    uint32_t ra[4], rb[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float a0 = bf16_lo(av[e]), a1 = bf16_hi(av[e]);
                        const float b0 = bf16_lo(bv[e]), b1 = bf16_hi(bv[e]);
                        const float c_0 = cs[2 * e], c_1 = cs[2 * e + 1], s_0 = sn[2 * e], s_1 = sn[2 * e + 1];
                        ra[e] = pack_bf16(a0 * c_0 - b0 * s_0, a1 * c_1 - b1 * s_1);
                        rb[e] = pack_bf16(b0 * c_0 + a0 * s_0, b1 * c_1 + a1 * s_1);
                    }
                    const int64_t o = (int64_t)(l0 + u) * dst_ls + off;
                    __stcs(reinterpret_cast<uint4*>(k_dst + o), make_uint4(ra[0], ra[1], ra[2], ra[3]));
                    __stcs(reinterpret_cast<uint4*>(k_dst + o + D / 2), make_uint4(rb[0], rb[1], rb[2], rb[3]));
                    if (copy_v) {
                        __stcs(reinterpret_cast<uint4*>(v_dst + o), v_convert16(va[u], bad));
                        __stcs(reinterpret_cast<uint4*>(v_dst + o + D / 2), v_convert16(vb[u], bad));
                    }
                }
            }
        }
    }
    if (bad) set_status(status, KVB_ERR_RANGE);
}

// ------------------------------------------------------------------ embedding
__global__ void __launch_bounds__(256)
embed_kernel(const uint16_t* __restrict__ embed, const int32_t* __restrict__ tok, int64_t n, int H, int vocab,
             float* __restrict__ x, int* status) {
    const int vec = H / 8;
    const int64_t items = n * vec;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < items;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = it / vec;
        const int c = (int)(it - r * vec);
        const int32_t t = __ldg(tok + r);
        float4* dst = reinterpret_cast<float4*>(x + r * H) + 2 * c;
        if ((uint32_t)t >= (uint32_t)vocab) {   // outside the table: a zero row, reported
            if (c == 0) set_status(status, KVB_ERR_INVALID_ARG);
            dst[0] = dst[1] = make_float4(0.f, 0.f, 0.f, 0.f);
            continue;
        }
        const uint4 e = __ldg(reinterpret_cast<const uint4*>(embed + (int64_t)t * H) + c);
        dst[0] = make_float4(bf16_lo(e.x), bf16_hi(e.x), bf16_lo(e.y), bf16_hi(e.y));
        dst[1] = make_float4(bf16_lo(e.z), bf16_hi(e.z), bf16_lo(e.w), bf16_hi(e.w));
    }
}

// ------------------------------------------------------------------ RMSNorm
// One CTA of T threads per row; thread t holds float4 t, t + T, ... (at most V of them)
// of the row's H/4 float4.
template <int T, int V>
__global__ void __launch_bounds__(T)
rmsnorm_kernel(const float* __restrict__ x, const int32_t* __restrict__ idx, int64_t m, int H,
               const float* __restrict__ g, float eps, uint16_t* __restrict__ out_bf16, float* __restrict__ out_f32) {
    __shared__ float red[T / 32];
    const int64_t r = blockIdx.x;
    const int64_t src = idx ? (int64_t)__ldg(idx + r) : r;
    const float4* xr = reinterpret_cast<const float4*>(x + src * H);
    const int H4 = H / 4;
    float4 v[V];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * T;
        v[i] = c < H4 ? xr[c] : make_float4(0.f, 0.f, 0.f, 0.f);
        ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < T / 32; ++w) tot += red[w];
    const float inv = rsqrtf(tot / (float)H + eps);
    const float4* gr = reinterpret_cast<const float4*>(g);
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const int c = threadIdx.x + i * T;
        if (c >= H4) break;
        const float4 gg = __ldg(gr + c);
        const float4 y = make_float4(v[i].x * inv * gg.x, v[i].y * inv * gg.y, v[i].z * inv * gg.z, v[i].w * inv * gg.w);
        if (out_bf16) {
            uint2 pk = make_uint2(pack_bf16(y.x, y.y), pack_bf16(y.z, y.w));
            reinterpret_cast<uint2*>(out_bf16 + r * H)[c] = pk;
        }
        if (out_f32) reinterpret_cast<float4*>(out_f32 + r * H)[c] = y;
    }
}

// ------------------------------------------------------------------ row gather / scatter
__global__ void __launch_bounds__(256)
gather_rows_kernel(const float* __restrict__ src, const int32_t* __restrict__ idx, int64_t m, int H,
                   float* __restrict__ dst) {
    const int vec = H / 4;
    const int64_t items = m * vec;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < items;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = it / vec;
        const int c = (int)(it - r * vec);
        reinterpret_cast<float4*>(dst + r * H)[c] =
            reinterpret_cast<const float4*>(src + (int64_t)__ldg(idx + r) * H)[c];
    }
}

__global__ void __launch_bounds__(256)
scatter_kernel(const uint16_t* __restrict__ k_rows, const uint16_t* __restrict__ v_rows,
               const int32_t* __restrict__ dst_idx, int64_t m, int kv_dim, uint16_t* __restrict__ k_dst,
               uint16_t* __restrict__ v_dst, int64_t n_dst) {
    const int vec = kv_dim / 8;
    const int64_t items = m * vec;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < items;
         it += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = it / vec;
        const int c = (int)(it - r * vec);
        const int64_t d = __ldg(dst_idx + r);
        if (d < 0 || d >= n_dst) continue;   // outside the destination: skipped
        reinterpret_cast<uint4*>(k_dst + d * kv_dim)[c] = reinterpret_cast<const uint4*>(k_rows + r * kv_dim)[c];
        reinterpret_cast<uint4*>(v_dst + d * kv_dim)[c] = reinterpret_cast<const uint4*>(v_rows + r * kv_dim)[c];
    }
}

__global__ void iota_kernel(int32_t* out, int64_t n, int32_t start) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = start + (int32_t)i;
}

// rows = [sel[0..k) , n_ctx .. n_ctx + n_query); a selected index outside [0, n_ctx) is
// reported and replaced by row 0, so that no later gather or scatter leaves the buffers
__global__ void concat_rows_kernel(const int32_t* sel, int64_t k, int64_t n_ctx, int64_t n_query, int32_t* rows,
                                   int* status) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < k + n_query;
         i += (int64_t)gridDim.x * blockDim.x) {
        int32_t v = (int32_t)(n_ctx + (i - k));
        if (i < k) {
            v = sel[i];
            if (v < 0 || v >= n_ctx) {
                set_status(status, KVB_ERR_INVALID_ARG);
                v = 0;
            }
        }
        rows[i] = v;
    }
}

unsigned grid_for(int64_t items, int threads) {
    const int64_t want = (items + threads - 1) / threads;
    const int64_t cap = (int64_t)num_sms() * 16;
    return (unsigned)(want < 1 ? 1 : (want < cap ? want : cap));
}

}  // namespace

kvb_status launch_realign(const float* cos_t, const float* sin_t, int D, int Hkv, const uint16_t* k_src,
                          const uint16_t* v_src, int64_t src_ls, uint16_t* k_dst, uint16_t* v_dst, int64_t dst_ls,
                          int n_layers, const int32_t* chunk_start, int n_chunks, int64_t n_ctx, int* status,
                          cudaStream_t st) {
    if (n_layers <= 0 || n_ctx <= 0) return KVB_OK;
    const bool copy_v = v_src && v_dst;
    const int64_t items = n_ctx * Hkv * (D / 16);
    const unsigned grid = grid_for(items, 256);
    if (D == 128)
        realign_kernel<128><<<grid, 256, 0, st>>>(cos_t, sin_t, Hkv, k_src, v_src, src_ls, k_dst, v_dst, dst_ls,
                                                  n_layers, chunk_start, n_chunks, n_ctx, copy_v, status);
    else if (D == 64)
        realign_kernel<64><<<grid, 256, 0, st>>>(cos_t, sin_t, Hkv, k_src, v_src, src_ls, k_dst, v_dst, dst_ls,
                                                 n_layers, chunk_start, n_chunks, n_ctx, copy_v, status);
    else
        return fail(KVB_ERR_UNSUPPORTED, "realign: head_dim %d not built", D);
    count_launch();
    return cuda_ok(cudaGetLastError(), "realign launch");
}

kvb_status launch_embed(const uint16_t* embed, const int32_t* tok, int64_t n, int H, int vocab, float* x,
                        int* status, cudaStream_t st) {
    if (n <= 0) return KVB_OK;
    if (vocab < 1) return fail(KVB_ERR_INVALID_ARG, "embedding: vocab %d < 1", vocab);
    embed_kernel<<<grid_for(n * (H / 8), 256), 256, 0, st>>>(embed, tok, n, H, vocab, x, status);
    count_launch();
    return cuda_ok(cudaGetLastError(), "embed launch");
}

kvb_status launch_rmsnorm(const float* x, const int32_t* idx, int64_t m, int H, const float* g, float eps,
                          uint16_t* out_bf16, float* out_f32, cudaStream_t st) {
    if (m <= 0) return KVB_OK;
    if (m > 0x7FFFFFFF) return fail(KVB_ERR_INVALID_ARG, "rmsnorm: too many rows");
    const unsigned grid = (unsigned)m;
    // 128 threads, each holding at most V float4 of the row (64 threads for H = 256)
    if (H <= 0 || H % 4 || H > 8192) return fail(KVB_ERR_UNSUPPORTED, "rmsnorm: hidden %d not built", H);
    if (H == 256) rmsnorm_kernel<64, 1><<<grid, 64, 0, st>>>(x, idx, m, H, g, eps, out_bf16, out_f32);
    else if (H <= 512) rmsnorm_kernel<128, 1><<<grid, 128, 0, st>>>(x, idx, m, H, g, eps, out_bf16, out_f32);
    else if (H <= 1024) rmsnorm_kernel<128, 2><<<grid, 128, 0, st>>>(x, idx, m, H, g, eps, out_bf16, out_f32);
    else if (H <= 2048) rmsnorm_kernel<128, 4><<<grid, 128, 0, st>>>(x, idx, m, H, g, eps, out_bf16, out_f32);
    else if (H <= 4096) rmsnorm_kernel<128, 8><<<grid, 128, 0, st>>>(x, idx, m, H, g, eps, out_bf16, out_f32);
    else rmsnorm_kernel<128, 16><<<grid, 128, 0, st>>>(x, idx, m, H, g, eps, out_bf16, out_f32);
    count_launch();
    return cuda_ok(cudaGetLastError(), "rmsnorm launch");
}

kvb_status launch_gather_rows(const float* src, const int32_t* idx, int64_t m, int H, float* dst, cudaStream_t st) {
    if (m <= 0) return KVB_OK;
    gather_rows_kernel<<<grid_for(m * (H / 4), 256), 256, 0, st>>>(src, idx, m, H, dst);
    count_launch();
    return cuda_ok(cudaGetLastError(), "gather launch");
}

kvb_status launch_scatter(const uint16_t* k_rows, const uint16_t* v_rows, const int32_t* dst_idx, int64_t m,
                          int kv_dim, uint16_t* k_dst, uint16_t* v_dst, int64_t n_dst, cudaStream_t st) {
    if (m <= 0) return KVB_OK;
    scatter_kernel<<<grid_for(m * (kv_dim / 8), 256), 256, 0, st>>>(k_rows, v_rows, dst_idx, m, kv_dim, k_dst, v_dst,
                                                                   n_dst);
    count_launch();
    return cuda_ok(cudaGetLastError(), "scatter launch");
}

kvb_status launch_iota(int32_t* out, int64_t n, int32_t start, cudaStream_t st) {
    if (n <= 0) return KVB_OK;
    iota_kernel<<<grid_for(n, 256), 256, 0, st>>>(out, n, start);
    count_launch();
    return cuda_ok(cudaGetLastError(), "iota launch");
}

kvb_status launch_concat_rows(const int32_t* sel, int64_t k, int64_t n_ctx, int64_t n_query, int32_t* rows,
                              int* status, cudaStream_t st) {
    if (k + n_query <= 0) return KVB_OK;
    concat_rows_kernel<<<grid_for(k + n_query, 256), 256, 0, st>>>(sel, k, n_ctx, n_query, rows, status);
    count_launch();
    return cuda_ok(cudaGetLastError(), "rows launch");
}

}  // namespace kvb
