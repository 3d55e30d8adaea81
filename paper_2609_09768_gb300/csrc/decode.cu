// Greedy decode on the blended cache: one new token per step through every layer.
//
// Everything here is bound by HBM traffic (each step reads all weights once, ~15 GB
// for Llama-3.1-8B, and every layer's cache up to the current position), so the
// kernels are CUDA-core kernels built for streaming, not tensor-core tiles:
//   decode_embed      - x = embed[tokens[pos]] (fp32)
//   gemv_kernel       - y = W a for one bf16 activation row held in shared memory;
//                       warp per output row, eight 16-byte weight loads per lane in
//                       flight; epilogues: fp32 out, residual add, SwiGLU (gate and up
//                       rows in the same warp)
//   qkv_finish        - RoPE at `pos` on q and k (fp32, then bf16), K and V written
//                       into cache row `pos` (V as bf16-rounded fp16, like the prefill)
//   decode_attn       - split-KV attention of the new row over cache rows [0, pos]:
//                       one warp per split of 128 keys and kv head, lanes over head
//                       dims; the G q heads sharing the kv head and 32/G keys give 32
//                       partial dot products per step, summed with one 31-shuffle
//                       reduce-scatter; online softmax per head in fp32; the next
//                       step's K/V loads are issued before this step's arithmetic; the 8
//                       warps of a CTA merge their (max, sum, O) in shared memory
//   decode_combine    - log-sum-exp merge of the CTA partials -> bf16 attention output
//   decode_finish     - tokens[pos + 1] = argmax, pos += 1
// The position and the token live in device memory, so a step needs no host value that
// changes from one step to the next.  Kernels that read `pos` check 0 <= pos < max_pos
// and record KVB_ERR_INVALID_ARG in the status word instead of touching memory otherwise.
#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

constexpr int GEMV_THREADS = 256;
constexpr int GEMV_BATCH = 8;
constexpr int ATT_THREADS = 256;             // 8 warps = 8 splits of one kv head

KVB_DEV bool pos_ok(const int32_t* pos_ptr, int64_t max_pos, int* status, int& pos) {
    pos = *pos_ptr;
    if (pos < 0 || (int64_t)pos >= max_pos) {
        if (threadIdx.x == 0) set_status(status, KVB_ERR_INVALID_ARG);
        return false;
    }
    return true;
}

__global__ void decode_embed_kernel(const uint16_t* __restrict__ embed, const int32_t* __restrict__ tokens,
                                    const int32_t* __restrict__ pos_ptr, int64_t max_pos, int64_t vocab, int H,
                                    float* __restrict__ x, int* status) {
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    const int tok = tokens[pos];
    if (tok < 0 || (int64_t)tok >= vocab) {
        if (threadIdx.x == 0) set_status(status, KVB_ERR_INVALID_ARG);
        return;
    }
    const uint16_t* row = embed + (int64_t)tok * H;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < H; i += gridDim.x * blockDim.x) x[i] = bf16_to_f(row[i]);
}

template <int MODE>
__global__ void __launch_bounds__(GEMV_THREADS)
gemv_kernel(const uint16_t* __restrict__ W, const uint16_t* __restrict__ W2, int64_t N, int K,
            const uint16_t* __restrict__ a, float* __restrict__ y_f32, uint16_t* __restrict__ y_bf16) {
    extern __shared__ float av[];   // [K]
    for (int i = threadIdx.x; i < K; i += blockDim.x) av[i] = bf16_to_f(a[i]);
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
    const int vec = K / 8;
    for (int64_t n = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); n < N; n += warps) {
        const uint4* wr = reinterpret_cast<const uint4*>(W + n * K);
        const uint4* wr2 = reinterpret_cast<const uint4*>((MODE == GEMV_SWIGLU ? W2 : W) + n * K);
        float acc = 0.f, acc2 = 0.f;
        for (int c0 = lane; c0 < vec; c0 += 32 * GEMV_BATCH) {
            uint4 w[GEMV_BATCH], w2[GEMV_BATCH];
#pragma unroll
            for (int u = 0; u < GEMV_BATCH; ++u) {
                const int c = c0 + 32 * u;
                w[u] = c < vec ? __ldcs(wr + c) : make_uint4(0u, 0u, 0u, 0u);
                if (MODE == GEMV_SWIGLU) w2[u] = c < vec ? __ldcs(wr2 + c) : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < GEMV_BATCH; ++u) {
                const int c = c0 + 32 * u;
                if (c >= vec) break;
                const float4* xr = reinterpret_cast<const float4*>(av + c * 8);
                const float4 x0 = xr[0], x1 = xr[1];
                const float xs[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
                const uint32_t ww[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc = fmaf(bf16_lo(ww[e]), xs[2 * e], acc);
                    acc = fmaf(bf16_hi(ww[e]), xs[2 * e + 1], acc);
                }
                if (MODE == GEMV_SWIGLU) {
                    const uint32_t w2w[4] = {w2[u].x, w2[u].y, w2[u].z, w2[u].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        acc2 = fmaf(bf16_lo(w2w[e]), xs[2 * e], acc2);
                        acc2 = fmaf(bf16_hi(w2w[e]), xs[2 * e + 1], acc2);
                    }
                }
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (MODE == GEMV_SWIGLU) acc2 += __shfl_xor_sync(0xffffffffu, acc2, o);
        }
        if (lane == 0) {
            if (MODE == GEMV_F32) y_f32[n] = acc;
            if (MODE == GEMV_RESID) y_f32[n] += acc;
            if (MODE == GEMV_SWIGLU)
                y_bf16[n] = __bfloat16_as_ushort(__float2bfloat16_rn(acc / (1.0f + __expf(-acc)) * acc2));
        }
    }
}

// Threads: (Hq + Hkv) * D/2 rotation pairs, then Hkv * D values of V.
__global__ void qkv_finish_kernel(const float* __restrict__ qkv, const int32_t* __restrict__ pos_ptr, int64_t max_pos,
                                  const float* __restrict__ cos_t, const float* __restrict__ sin_t, int D, int Hq,
                                  int Hkv, uint16_t* __restrict__ q_out, uint16_t* __restrict__ k_layer,
                                  uint16_t* __restrict__ v_layer, int* status) {
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    const int half = D / 2;
    const int n_rot = (Hq + Hkv) * half;
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t < n_rot) {
        const int h = t / half, i = t % half;
        const float a = qkv[h * D + i], b = qkv[h * D + i + half];
        const float c = cos_t[(int64_t)pos * half + i], s = sin_t[(int64_t)pos * half + i];
        const float y1 = a * c - b * s;
        const float y2 = b * c + a * s;
        uint16_t* dst = h < Hq ? q_out + h * D : k_layer + ((int64_t)pos * Hkv + (h - Hq)) * D;
        dst[i] = __bfloat16_as_ushort(__float2bfloat16_rn(y1));
        dst[i + half] = __bfloat16_as_ushort(__float2bfloat16_rn(y2));
    } else if (t < n_rot + Hkv * D) {
        const int j = t - n_rot;
        const float v = __bfloat162float(__float2bfloat16_rn(qkv[(Hq + Hkv) * D + j]));
        v_layer[(int64_t)pos * Hkv * D + j] = __half_as_ushort(__float2half_rn(v));
    }
}

// Unpack one lane's DPL head dims of a key (bf16) or value (fp16) row from raw words.
template <int DPL>
struct RowBits {
    uint32_t w[DPL / 2];
};
template <int DPL>
KVB_DEV RowBits<DPL> load_row(const uint16_t* p) {
    RowBits<DPL> r;
    if constexpr (DPL == 4) {
        const uint2 u = __ldcs(reinterpret_cast<const uint2*>(p));
        r.w[0] = u.x; r.w[1] = u.y;
    } else {
        r.w[0] = __ldcs(reinterpret_cast<const unsigned int*>(p));
    }
    return r;
}

// One CTA = eight consecutive splits of KVB_DECODE_KEYS_PER_SPLIT cache rows for kv head
// blockIdx.y, one warp per split; the warps' partial results are merged in shared memory
// and the CTA writes one partial (max, sum, O) per q head.
template <int D, int G>
__global__ void __launch_bounds__(ATT_THREADS, 2)
decode_attn_kernel(const uint16_t* __restrict__ q, const uint16_t* __restrict__ kc, const uint16_t* __restrict__ vc,
                   int Hkv, const int32_t* __restrict__ pos_ptr, int64_t max_pos, int n_blocks, float scale_log2,
                   float* __restrict__ pm, float* __restrict__ pl, float* __restrict__ po, int* status) {
    constexpr int DPL = D / 32;      // head dims per lane
    constexpr int KS = 32 / G;       // keys per step: KS * G = 32 partial dot products
    constexpr int WARPS = ATT_THREADS / 32;
    __shared__ float sm_m[WARPS][G], sm_l[WARPS][G];
    __shared__ float sm_o[WARPS][G][D];
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    if ((int)blockIdx.x >= n_blocks) return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = blockIdx.y;
    const int Hq = Hkv * G;
    const int64_t start = ((int64_t)blockIdx.x * WARPS + warp) * KVB_DECODE_KEYS_PER_SPLIT;
    int64_t end = start + KVB_DECODE_KEYS_PER_SPLIT;
    if (end > (int64_t)pos + 1) end = (int64_t)pos + 1;

    float qv[G][DPL];
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
        for (int e = 0; e < DPL; ++e) qv[h][e] = bf16_to_f(q[(g * G + h) * D + lane * DPL + e]);
    float o[G][DPL];
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
        for (int e = 0; e < DPL; ++e) o[h][e] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;    // of head lane % G

    const int64_t row_stride = (int64_t)Hkv * D;
    const uint16_t* kbase = kc + (int64_t)g * D + lane * DPL;
    const uint16_t* vbase = vc + (int64_t)g * D + lane * DPL;
    RowBits<DPL> ck[KS], cv[KS], nk[KS], nv[KS];
    auto fetch = [&](int64_t k0, RowBits<DPL>* kr, RowBits<DPL>* vr) {
#pragma unroll
        for (int k = 0; k < KS; ++k) {
            if (k0 + k < end) {
                kr[k] = load_row<DPL>(kbase + (k0 + k) * row_stride);
                vr[k] = load_row<DPL>(vbase + (k0 + k) * row_stride);
            } else {
#pragma unroll
                for (int i = 0; i < DPL / 2; ++i) { kr[k].w[i] = 0u; vr[k].w[i] = 0u; }
            }
        }
    };
    if (start < end) fetch(start, ck, cv);
    for (int64_t k0 = start; k0 < end; k0 += KS) {
        // loads of the next step go out before this step's arithmetic
        if (k0 + KS < end) fetch(k0 + KS, nk, nv);
        float sc[32];
#pragma unroll
        for (int k = 0; k < KS; ++k) {
            float kf[DPL];
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i) { kf[2 * i] = bf16_lo(ck[k].w[i]); kf[2 * i + 1] = bf16_hi(ck[k].w[i]); }
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float acc = 0.f;
#pragma unroll
                for (int e = 0; e < DPL; ++e) acc = fmaf(qv[h][e], kf[e], acc);
                sc[k * G + h] = acc;
            }
        }
        // reduce-scatter: afterwards lane L holds the full dot product of index L
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) {
#pragma unroll
            for (int i = 0; i < off; ++i) {
                const bool upper = (lane & off) != 0;
                const float send = upper ? sc[i] : sc[i + off];
                const float keep = upper ? sc[i + off] : sc[i];
                sc[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
            }
        }
        float t = sc[0] * scale_log2;
        if (k0 + lane / G >= end) t = -INFINITY;
        // online softmax of head lane % G over this step's keys
        float mx = t;
#pragma unroll
        for (int off = G; off < 32; off <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        const float m_new = fmaxf(m_run, mx);
        const float alpha = (m_new == -INFINITY) ? 1.f : exp2f(m_run - m_new);
        const float pv = (t == -INFINITY) ? 0.f : exp2f(t - m_new);
        float ps = pv;
#pragma unroll
        for (int off = G; off < 32; off <<= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
        l_run = l_run * alpha + ps;
        m_run = m_new;
#pragma unroll
        for (int h = 0; h < G; ++h) {
            const float ah = __shfl_sync(0xffffffffu, alpha, h);
#pragma unroll
            for (int e = 0; e < DPL; ++e) o[h][e] *= ah;
        }
#pragma unroll
        for (int k = 0; k < KS; ++k) {
            float vf[DPL];
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i) {
                const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&cv[k].w[i]));
                vf[2 * i] = f.x; vf[2 * i + 1] = f.y;
            }
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float pk = __shfl_sync(0xffffffffu, pv, k * G + h);
#pragma unroll
                for (int e = 0; e < DPL; ++e) o[h][e] = fmaf(pk, vf[e], o[h][e]);
            }
        }
#pragma unroll
        for (int k = 0; k < KS; ++k) { ck[k] = nk[k]; cv[k] = nv[k]; }
    }
    // merge the warps of this CTA
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
        for (int e = 0; e < DPL; ++e) sm_o[warp][h][lane * DPL + e] = o[h][e];
    if (lane < G) { sm_m[warp][lane] = m_run; sm_l[warp][lane] = l_run; }
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * Hq + g * G;
    for (int i = threadIdx.x; i < G * D; i += ATT_THREADS) {
        const int h = i / D, d = i % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) M = fmaxf(M, sm_m[w][h]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) {
            const float c = (sm_m[w][h] == -INFINITY) ? 0.f : exp2f(sm_m[w][h] - M);
            L += c * sm_l[w][h];
            O += c * sm_o[w][h][d];
        }
        po[(base + h) * D + d] = O;
        if (d == 0) { pm[base + h] = M; pl[base + h] = L; }
    }
}

// One block per q head: COMB_GROUPS groups of D threads, each over every COMB_GROUPS-th CTA
// partial, then merged in shared memory.
constexpr int COMB_GROUPS = 4;
__global__ void decode_combine_kernel(const float* __restrict__ pm, const float* __restrict__ pl,
                                      const float* __restrict__ po, const int32_t* __restrict__ pos_ptr,
                                      int64_t max_pos, int keys_per_block, int Hq, int D, uint16_t* __restrict__ out,
                                      int* status) {
    __shared__ float s_m[COMB_GROUPS], s_l[COMB_GROUPS];
    __shared__ float s_o[COMB_GROUPS][128];
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    const int hq = blockIdx.x, d = threadIdx.x % D, grp = threadIdx.x / D;
    const int n = (pos + keys_per_block) / keys_per_block;   // CTA partials holding keys [0, pos]
    float M = -INFINITY;
    for (int s = grp; s < n; s += COMB_GROUPS) M = fmaxf(M, pm[(int64_t)s * Hq + hq]);
    float L = 0.f, O = 0.f;
#pragma unroll 4
    for (int s = grp; s < n; s += COMB_GROUPS) {
        const float ms = pm[(int64_t)s * Hq + hq];
        const float w = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
        L += w * pl[(int64_t)s * Hq + hq];
        O += w * po[((int64_t)s * Hq + hq) * D + d];
    }
    if (d == 0) { s_m[grp] = M; s_l[grp] = L; }
    s_o[grp][d] = O;
    __syncthreads();
    if (grp == 0) {
        float MM = -INFINITY;
#pragma unroll
        for (int q2 = 0; q2 < COMB_GROUPS; ++q2) MM = fmaxf(MM, s_m[q2]);
        float LL = 0.f, OO = 0.f;
#pragma unroll
        for (int q2 = 0; q2 < COMB_GROUPS; ++q2) {
            const float w = (s_m[q2] == -INFINITY) ? 0.f : exp2f(s_m[q2] - MM);
            LL += w * s_l[q2];
            OO += w * s_o[q2][d];
        }
        out[hq * D + d] = __bfloat16_as_ushort(__float2bfloat16_rn(LL > 0.f ? OO / LL : 0.f));
    }
}

__global__ void decode_finish_kernel(const int32_t* __restrict__ tok, int32_t* __restrict__ tokens,
                                     int32_t* __restrict__ pos_ptr, int64_t max_pos, int* status) {
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    tokens[pos + 1] = tok[0];
    *pos_ptr = pos + 1;
}

template <int D, int G>
kvb_status run_attn(const uint16_t* q, const uint16_t* kc, const uint16_t* vc, int Hkv, const int32_t* pos,
                    int64_t max_pos, int n_blocks, float sl2, float* pm, float* pl, float* po, int* status,
                    cudaStream_t st) {
    const dim3 grid((unsigned)n_blocks, (unsigned)Hkv);
    decode_attn_kernel<D, G><<<grid, ATT_THREADS, 0, st>>>(q, kc, vc, Hkv, pos, max_pos, n_blocks, sl2, pm, pl, po,
                                                           status);
    count_launch();
    return cuda_ok(cudaGetLastError(), "decode attention launch");
}

}  // namespace

kvb_status launch_decode_embed(const uint16_t* embed, const int32_t* tokens, const int32_t* pos, int64_t max_pos,
                               int64_t vocab, int H, float* x, int* status, cudaStream_t st) {
    decode_embed_kernel<<<(H + 255) / 256, 256, 0, st>>>(embed, tokens, pos, max_pos, vocab, H, x, status);
    count_launch();
    return cuda_ok(cudaGetLastError(), "decode embed launch");
}

kvb_status launch_gemv(int mode, const uint16_t* W, const uint16_t* W2, int64_t N, int K, const uint16_t* a,
                       float* y_f32, uint16_t* y_bf16, cudaStream_t st) {
    if (N <= 0) return KVB_OK;
    if (K <= 0 || K % 8 || K > KVB_DECODE_MAX_K)
        return fail(KVB_ERR_UNSUPPORTED, "gemv: K = %d must be a positive multiple of 8 up to %d", K, KVB_DECODE_MAX_K);
    const size_t smem = (size_t)K * sizeof(float);
    static bool attr[3] = {false, false, false};
    auto set = [&](auto kern) -> kvb_status {
        if (!attr[mode]) {
            kvb_status s = cuda_ok(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                        KVB_DECODE_MAX_K * (int)sizeof(float)),
                                   "gemv smem");
            if (s != KVB_OK) return s;
            attr[mode] = true;
        }
        int per_sm = 0;
        kvb_status s = cuda_ok(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, GEMV_THREADS, smem),
                               "gemv occupancy");
        if (s != KVB_OK) return s;
        int64_t blocks = (N + GEMV_THREADS / 32 - 1) / (GEMV_THREADS / 32);
        const int64_t cap = (int64_t)num_sms() * (per_sm > 0 ? per_sm : 1);
        if (blocks > cap) blocks = cap;
        kern<<<(unsigned)blocks, GEMV_THREADS, smem, st>>>(W, W2, N, K, a, y_f32, y_bf16);
        count_launch();
        return cuda_ok(cudaGetLastError(), "gemv launch");
    };
    switch (mode) {
        case GEMV_F32: return set(gemv_kernel<GEMV_F32>);
        case GEMV_RESID: return set(gemv_kernel<GEMV_RESID>);
        case GEMV_SWIGLU: return set(gemv_kernel<GEMV_SWIGLU>);
        default: return fail(KVB_ERR_INVALID_ARG, "gemv: unknown mode %d", mode);
    }
}

kvb_status launch_qkv_finish(const float* qkv, const int32_t* pos, int64_t max_pos, const float* cos_t,
                             const float* sin_t, int D, int Hq, int Hkv, uint16_t* q_out, uint16_t* k_layer,
                             uint16_t* v_layer, int* status, cudaStream_t st) {
    const int n = (Hq + Hkv) * (D / 2) + Hkv * D;
    qkv_finish_kernel<<<(n + 255) / 256, 256, 0, st>>>(qkv, pos, max_pos, cos_t, sin_t, D, Hq, Hkv, q_out, k_layer,
                                                       v_layer, status);
    count_launch();
    return cuda_ok(cudaGetLastError(), "qkv finish launch");
}

// CTA partials of the decode attention for positions below max_pos
int decode_splits(int64_t max_pos) {
    const int64_t per_block = (int64_t)KVB_DECODE_KEYS_PER_SPLIT * (ATT_THREADS / 32);
    return (int)((max_pos + per_block - 1) / per_block);
}

kvb_status launch_decode_attn(const uint16_t* q, const uint16_t* kc, const uint16_t* vc, int Hq, int Hkv, int D,
                              const int32_t* pos, int64_t max_pos, float sl2, float* pm, float* pl, float* po,
                              uint16_t* out, int* status, cudaStream_t st) {
    const int G = Hq / Hkv;
    const int n_splits = decode_splits(max_pos);
    kvb_status s;
    if (D == 128 && G == 4) s = run_attn<128, 4>(q, kc, vc, Hkv, pos, max_pos, n_splits, sl2, pm, pl, po, status, st);
    else if (D == 128 && G == 8) s = run_attn<128, 8>(q, kc, vc, Hkv, pos, max_pos, n_splits, sl2, pm, pl, po, status, st);
    else if (D == 128 && G == 2) s = run_attn<128, 2>(q, kc, vc, Hkv, pos, max_pos, n_splits, sl2, pm, pl, po, status, st);
    else if (D == 64 && G == 2) s = run_attn<64, 2>(q, kc, vc, Hkv, pos, max_pos, n_splits, sl2, pm, pl, po, status, st);
    else if (D == 64 && G == 4) s = run_attn<64, 4>(q, kc, vc, Hkv, pos, max_pos, n_splits, sl2, pm, pl, po, status, st);
    else return fail(KVB_ERR_UNSUPPORTED, "decode attention: head_dim %d with %d q heads per kv head not built", D, G);
    if (s != KVB_OK) return s;
    decode_combine_kernel<<<(unsigned)Hq, (unsigned)(D * COMB_GROUPS), 0, st>>>(
        pm, pl, po, pos, max_pos, KVB_DECODE_KEYS_PER_SPLIT * (ATT_THREADS / 32), Hq, D, out, status);
    count_launch();
    return cuda_ok(cudaGetLastError(), "decode combine launch");
}

kvb_status launch_decode_finish(const int32_t* tok, int32_t* tokens, int32_t* pos, int64_t max_pos, int* status,
                                cudaStream_t st) {
    decode_finish_kernel<<<1, 1, 0, st>>>(tok, tokens, pos, max_pos, status);
    count_launch();
    return cuda_ok(cudaGetLastError(), "decode finish launch");
}

}  // namespace kvb
