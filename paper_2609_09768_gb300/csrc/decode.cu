// Greedy decode on the blended cache: one new token per step through every layer.
//
// Everything here is bound by HBM traffic (each step reads all weights once, ~15 GB
// for Llama-3.1-8B, and every layer's cache up to the current position), so the
// kernels are CUDA-core kernels built for streaming, not tensor-core tiles:
//   decode_embed      - x = embed[tokens[pos]] (fp32)
//   gemv_kernel       - y = W a for one activation row held in shared memory as bf16;
//                       warp per output row (or row pair), 16-byte weight loads, 8-16 per
//                       lane in flight.  QKV and SwiGLU normalise the residual row
//                       themselves (RMSNorm prologue in every block); QKV computes the two
//                       rows of a rotation pair in one warp, applies RoPE at `pos` and writes
//                       q and the cache's K/V row `pos` (V as bf16-rounded fp16, like the
//                       prefill); the residual mode adds into x; SwiGLU computes gate and
//                       up rows in one warp
//   decode_attn       - split-KV attention of the new row over cache rows [0, pos]:
//                       one warp per split of 128 keys and kv head, lanes over head
//                       dims; the G q heads sharing the kv head (padded to a power of
//                       two GP) and 32/GP keys give 32 partial dot products per step, summed with one 31-shuffle
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

// Dot products of one or two bf16 weight rows with the bf16 activation row in shared memory,
// BATCH 16-byte loads per lane per row in flight; every lane returns the full sums.
template <bool TWO, int BATCH>
KVB_DEV void dot_rows(const uint16_t* __restrict__ w1, const uint16_t* __restrict__ w2, const uint16_t* act, int K,
                      int lane, float& s1, float& s2) {
    const uint4* r1 = reinterpret_cast<const uint4*>(w1);
    const uint4* r2 = reinterpret_cast<const uint4*>(w2);
    const uint4* av = reinterpret_cast<const uint4*>(act);
    const int vec = K / 8;
    float acc = 0.f, acc2 = 0.f;
    for (int c0 = lane; c0 < vec; c0 += 32 * BATCH) {
        uint4 wa[BATCH], wb[TWO ? BATCH : 1];
#pragma unroll
        for (int u = 0; u < BATCH; ++u) {
            const int c = c0 + 32 * u;
            wa[u] = c < vec ? __ldcs(r1 + c) : make_uint4(0u, 0u, 0u, 0u);
            if constexpr (TWO) wb[u] = c < vec ? __ldcs(r2 + c) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < BATCH; ++u) {
            const int c = c0 + 32 * u;
            if (c >= vec) break;
            const uint4 xv = av[c];
            const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
            const uint32_t ww[4] = {wa[u].x, wa[u].y, wa[u].z, wa[u].w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                acc = fmaf(bf16_lo(ww[e]), bf16_lo(xw[e]), acc);
                acc = fmaf(bf16_hi(ww[e]), bf16_hi(xw[e]), acc);
            }
            if constexpr (TWO) {
                const uint32_t vw[4] = {wb[u].x, wb[u].y, wb[u].z, wb[u].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc2 = fmaf(bf16_lo(vw[e]), bf16_lo(xw[e]), acc2);
                    acc2 = fmaf(bf16_hi(vw[e]), bf16_hi(xw[e]), acc2);
                }
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if constexpr (TWO) acc2 += __shfl_xor_sync(0xffffffffu, acc2, o);
    }
    s1 = acc;
    s2 = acc2;
}

// One GEMV of a decode step.  The activation row is put in shared memory as bf16:
//   GEMV_QKV, GEMV_SWIGLU: RMSNorm(x) * gain of the fp32 residual row x (each block
//                          normalises it itself: no separate norm launch);
//   GEMV_RESID:            the bf16 row `a` as given.
// Work units per warp:
//   GEMV_QKV    - a rotation pair (rows i and i + D/2 of a q or k head): bias, RoPE at
//                 `pos`, bf16 q or cache K row `pos`; or one V row (+ bias): cache V row `pos`
//   GEMV_RESID  - one row: x[n] += y
//   GEMV_SWIGLU - gate row n and up row n: h[n] = bf16(silu(gate) * up)
template <int MODE>
__global__ void __launch_bounds__(GEMV_THREADS)
gemv_kernel(const GemvArgs p) {
    extern __shared__ __align__(16) uint16_t act[];   // [K]
    __shared__ float red[GEMV_THREADS / 32];
    const int K = p.K;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int pos = 0;
    if constexpr (MODE == GEMV_QKV) {
        if (!pos_ok(p.pos, p.max_pos, p.status, pos)) return;
    }
    if constexpr (MODE == GEMV_RESID) {
        for (int i = threadIdx.x; i < K / 8; i += blockDim.x)
            reinterpret_cast<uint4*>(act)[i] = reinterpret_cast<const uint4*>(p.a)[i];
    } else {
        const float4* x4 = reinterpret_cast<const float4*>(p.x);
        float ss = 0.f;
        for (int i = threadIdx.x; i < K / 4; i += blockDim.x) {
            const float4 v = x4[i];
            ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) red[warp] = ss;
        __syncthreads();
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < GEMV_THREADS / 32; ++w) tot += red[w];
        const float inv = rsqrtf(tot / (float)K + p.eps);
        const float4* g4 = reinterpret_cast<const float4*>(p.g);
        for (int i = threadIdx.x; i < K / 4; i += blockDim.x) {
            const float4 v = x4[i], gg = __ldg(g4 + i);
            reinterpret_cast<uint2*>(act)[i] =
                make_uint2(pack_bf16(v.x * inv * gg.x, v.y * inv * gg.y), pack_bf16(v.z * inv * gg.z, v.w * inv * gg.w));
        }
    }
    __syncthreads();
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
    const int64_t first = (int64_t)blockIdx.x * (blockDim.x / 32) + warp;
    if constexpr (MODE == GEMV_QKV) {
        const int D = p.D, half = D / 2, Hq = p.Hq, Hkv = p.Hkv;
        const int64_t n_pairs = (int64_t)(Hq + Hkv) * half, n_units = n_pairs + (int64_t)Hkv * D;
        for (int64_t u = first; u < n_units; u += warps) {
            if (u < n_pairs) {
                const int h = (int)(u / half), i = (int)(u % half);
                float a, b;
                dot_rows<true, 8>(p.W + ((int64_t)h * D + i) * K, p.W + ((int64_t)h * D + i + half) * K, act, K, lane,
                                  a, b);
                if (lane == 0) {
                    if (p.bias) {
                        a += p.bias[(int64_t)h * D + i];
                        b += p.bias[(int64_t)h * D + i + half];
                    }
                    const float c = p.cos_t[(int64_t)pos * half + i], sn = p.sin_t[(int64_t)pos * half + i];
                    const float y1 = a * c - b * sn;
                    const float y2 = b * c + a * sn;
                    uint16_t* dst = h < Hq ? p.q_out + h * D : p.k_layer + ((int64_t)pos * Hkv + (h - Hq)) * D;
                    dst[i] = __bfloat16_as_ushort(__float2bfloat16_rn(y1));
                    dst[i + half] = __bfloat16_as_ushort(__float2bfloat16_rn(y2));
                }
            } else {
                const int j = (int)(u - n_pairs);
                float a, unused;
                dot_rows<false, 16>(p.W + ((int64_t)(Hq + Hkv) * D + j) * K, nullptr, act, K, lane, a, unused);
                if (lane == 0) {
                    if (p.bias) a += p.bias[(int64_t)(Hq + Hkv) * D + j];
                    const float v = __bfloat162float(__float2bfloat16_rn(a));
                    p.v_layer[(int64_t)pos * Hkv * D + j] = __half_as_ushort(__float2half_rn(v));
                }
            }
        }
    } else {
        for (int64_t n = first; n < p.N; n += warps) {
            float a, b;
            if constexpr (MODE == GEMV_SWIGLU) {
                dot_rows<true, 8>(p.W + n * K, p.W2 + n * K, act, K, lane, a, b);
                if (lane == 0) p.y_bf16[n] = __bfloat16_as_ushort(__float2bfloat16_rn(a / (1.0f + __expf(-a)) * b));
            } else {
                dot_rows<false, 16>(p.W + n * K, nullptr, act, K, lane, a, b);
                if (lane == 0) p.y_f32[n] += a;
            }
        }
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

// Head slots per kv head: the lane layout pads a group of G q heads to GP slots, a power
// of two and at least 4 (so that a step covers at most 8 keys and the K/V prefetch fits in
// registers); the padding heads have q = 0 and are never written out.
__host__ __device__ constexpr int pad_pow2(int g) { return g <= 4 ? 4 : 8; }

// One CTA = eight consecutive splits of KVB_DECODE_KEYS_PER_SPLIT cache rows for kv head
// blockIdx.y, one warp per split; the warps' partial results are merged in shared memory
// and the CTA writes one partial (max, sum, O) per q head.
template <int D, int G>
__global__ void __launch_bounds__(ATT_THREADS, 2)
decode_attn_kernel(const uint16_t* __restrict__ q, const uint16_t* __restrict__ kc, const uint16_t* __restrict__ vc,
                   int Hkv, const int32_t* __restrict__ pos_ptr, int64_t max_pos, int n_blocks, float scale_log2,
                   float* __restrict__ pm, float* __restrict__ pl, float* __restrict__ po, int* status) {
    constexpr int DPL = D / 32;      // head dims per lane
    constexpr int GP = pad_pow2(G);  // head slots
    static_assert(G >= 1 && G <= 8, "group size");
    constexpr int KS = 32 / GP;      // keys per step: KS * GP = 32 partial dot products
    constexpr int WARPS = ATT_THREADS / 32;
    __shared__ float sm_m[WARPS][GP], sm_l[WARPS][GP];
    __shared__ float sm_o[WARPS][GP][D];
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    if ((int)blockIdx.x >= n_blocks) return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = blockIdx.y;
    const int Hq = Hkv * G;
    const int64_t start = ((int64_t)blockIdx.x * WARPS + warp) * KVB_DECODE_KEYS_PER_SPLIT;
    int64_t end = start + KVB_DECODE_KEYS_PER_SPLIT;
    if (end > (int64_t)pos + 1) end = (int64_t)pos + 1;

    // q of the G heads (zero for the padding slots) in shared memory (registers go to the
    // K/V prefetch)
    __shared__ __align__(16) float qs[GP][D];
    __shared__ __align__(16) float sp[ATT_THREADS / 32][32];   // per warp: this step's weights
    __shared__ float sa[ATT_THREADS / 32][GP];                  // per warp: rescale factor per head
    for (int i = threadIdx.x; i < GP * D; i += ATT_THREADS)
        qs[i / D][i % D] = i < G * D ? bf16_to_f(q[(g * G) * D + i]) : 0.f;
    __syncthreads();
    float o[GP][DPL];
#pragma unroll
    for (int h = 0; h < GP; ++h)
#pragma unroll
        for (int e = 0; e < DPL; ++e) o[h][e] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;    // of head slot lane % GP

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
        {
            float qv[GP][DPL];   // this lane's head dims of q, once per step
#pragma unroll
            for (int h = 0; h < GP; ++h) {
                if constexpr (DPL == 4) {
                    const float4 t4 = *reinterpret_cast<const float4*>(&qs[h][lane * 4]);
                    qv[h][0] = t4.x; qv[h][1] = t4.y; qv[h][2] = t4.z; qv[h][3] = t4.w;
                } else {
                    const float2 t2 = *reinterpret_cast<const float2*>(&qs[h][lane * 2]);
                    qv[h][0] = t2.x; qv[h][1] = t2.y;
                }
            }
#pragma unroll
            for (int k = 0; k < KS; ++k) {
                float kf[DPL];
#pragma unroll
                for (int i = 0; i < DPL / 2; ++i) { kf[2 * i] = bf16_lo(ck[k].w[i]); kf[2 * i + 1] = bf16_hi(ck[k].w[i]); }
#pragma unroll
                for (int h = 0; h < GP; ++h) {
                    float acc = 0.f;
#pragma unroll
                    for (int e = 0; e < DPL; ++e) acc = fmaf(qv[h][e], kf[e], acc);
                    sc[k * GP + h] = acc;
                }
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
        if (k0 + lane / GP >= end) t = -INFINITY;
        // online softmax of head slot lane % GP over this step's keys
        float mx = t;
#pragma unroll
        for (int off = GP; off < 32; off <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        const float m_new = fmaxf(m_run, mx);
        const float alpha = (m_new == -INFINITY) ? 1.f : fast_exp2(m_run - m_new);
        const float pv = (t == -INFINITY) ? 0.f : fast_exp2(t - m_new);
        float ps = pv;
#pragma unroll
        for (int off = GP; off < 32; off <<= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
        l_run = l_run * alpha + ps;
        m_run = m_new;
        // this step's weights (index key * GP + head) and the heads' rescale factors to every lane
        __syncwarp();
        sp[warp][lane] = pv;
        if (lane < GP) sa[warp][lane] = alpha;
        __syncwarp();
#pragma unroll
        for (int h = 0; h < GP; ++h) {
            const float ah = sa[warp][h];
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
            float pk[GP];   // weights of key k for the GP head slots, vector loads (broadcast)
            if constexpr (GP % 4 == 0) {
#pragma unroll
                for (int h4 = 0; h4 < GP; h4 += 4) {
                    const float4 t = *reinterpret_cast<const float4*>(&sp[warp][k * GP + h4]);
                    pk[h4] = t.x; pk[h4 + 1] = t.y; pk[h4 + 2] = t.z; pk[h4 + 3] = t.w;
                }
            } else if constexpr (GP == 2) {
                const float2 t = *reinterpret_cast<const float2*>(&sp[warp][k * GP]);
                pk[0] = t.x; pk[1] = t.y;
            } else {
                pk[0] = sp[warp][k];
            }
#pragma unroll
            for (int h = 0; h < GP; ++h) {
#pragma unroll
                for (int e = 0; e < DPL; ++e) o[h][e] = fmaf(pk[h], vf[e], o[h][e]);
            }
        }
#pragma unroll
        for (int k = 0; k < KS; ++k) { ck[k] = nk[k]; cv[k] = nv[k]; }
    }
    // merge the warps of this CTA (the G real heads)
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

// Block (q head, 32 head dims): COMB_GROUPS groups of 32 threads, group q over CTA partials
// q, q + COMB_GROUPS, ..., then merged in shared memory.
constexpr int COMB_GROUPS = 32;
__global__ void __launch_bounds__(32 * COMB_GROUPS)
decode_combine_kernel(const float* __restrict__ pm, const float* __restrict__ pl, const float* __restrict__ po,
                      const int32_t* __restrict__ pos_ptr, int64_t max_pos, int keys_per_block, int Hq, int D,
                      uint16_t* __restrict__ out, int* status) {
    __shared__ float s_m[COMB_GROUPS], s_l[COMB_GROUPS];
    __shared__ float s_o[COMB_GROUPS][32];
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    const int hq = blockIdx.x, d = blockIdx.y * 32 + (threadIdx.x & 31), grp = threadIdx.x >> 5;
    const int n = (pos + keys_per_block) / keys_per_block;   // CTA partials holding keys [0, pos]
    float M = -INFINITY;
    for (int s = grp; s < n; s += COMB_GROUPS) M = fmaxf(M, pm[(int64_t)s * Hq + hq]);
    float L = 0.f, O = 0.f;
    for (int s = grp; s < n; s += COMB_GROUPS) {
        const float ms = pm[(int64_t)s * Hq + hq];
        const float w = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
        L += w * pl[(int64_t)s * Hq + hq];
        O += w * po[((int64_t)s * Hq + hq) * D + d];
    }
    if ((threadIdx.x & 31) == 0) { s_m[grp] = M; s_l[grp] = L; }
    s_o[grp][threadIdx.x & 31] = O;
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
            OO += w * s_o[q2][threadIdx.x];
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

kvb_status launch_gemv(int mode, const GemvArgs& p, cudaStream_t st) {
    if (p.K <= 0 || p.K % 8 || p.K > KVB_DECODE_MAX_K)
        return fail(KVB_ERR_UNSUPPORTED, "gemv: K = %d must be a positive multiple of 8 up to %d", p.K,
                    KVB_DECODE_MAX_K);
    const size_t smem = (size_t)p.K * sizeof(uint16_t);
    static std::atomic<uint64_t> smem_set[3];
    int64_t units = p.N;
    if (mode == GEMV_QKV) units = (int64_t)(p.Hq + p.Hkv) * (p.D / 2) + (int64_t)p.Hkv * p.D;
    if (units <= 0) return KVB_OK;
    auto go = [&](auto kern) -> kvb_status {
        kvb_status s = ensure_smem_limit((const void*)kern, KVB_DECODE_MAX_K * (int)sizeof(uint16_t), smem_set[mode],
                                         "gemv smem");
        if (s != KVB_OK) return s;
        int per_sm = 0;
        s = cuda_ok(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, GEMV_THREADS, smem),
                               "gemv occupancy");
        if (s != KVB_OK) return s;
        int64_t blocks = (units + GEMV_THREADS / 32 - 1) / (GEMV_THREADS / 32);
        const int64_t cap = (int64_t)num_sms() * (per_sm > 0 ? per_sm : 1);
        if (blocks > cap) blocks = cap;
        kern<<<(unsigned)blocks, GEMV_THREADS, smem, st>>>(p);
        count_launch();
        return cuda_ok(cudaGetLastError(), "gemv launch");
    };
    switch (mode) {
        case GEMV_QKV: return go(gemv_kernel<GEMV_QKV>);
        case GEMV_RESID: return go(gemv_kernel<GEMV_RESID>);
        case GEMV_SWIGLU: return go(gemv_kernel<GEMV_SWIGLU>);
        default: return fail(KVB_ERR_INVALID_ARG, "gemv: unknown mode %d", mode);
    }
}

// CTA partials of the decode attention for positions below max_pos
int decode_splits(int64_t max_pos, int) {
    const int64_t per_block = (int64_t)KVB_DECODE_KEYS_PER_SPLIT * (ATT_THREADS / 32);
    return (int)((max_pos + per_block - 1) / per_block);
}

kvb_status launch_decode_attn(const uint16_t* q, const uint16_t* kc, const uint16_t* vc, int Hq, int Hkv, int D,
                              const int32_t* pos, int64_t max_pos, float sl2, float* pm, float* pl, float* po,
                              uint16_t* out, int* status, cudaStream_t st) {
    const int G = Hq / Hkv;
    const int n_splits = decode_splits(max_pos, Hkv);
    kvb_status s;
#define KVB_DECODE_CASE(DD, GG) \
    else if (D == DD && G == GG) s = run_attn<DD, GG>(q, kc, vc, Hkv, pos, max_pos, n_splits, sl2, pm, pl, po, status, st);
    if (false) {}
    KVB_DECODE_CASE(128, 1) KVB_DECODE_CASE(128, 2) KVB_DECODE_CASE(128, 4) KVB_DECODE_CASE(128, 7) KVB_DECODE_CASE(128, 8)
    KVB_DECODE_CASE(64, 1) KVB_DECODE_CASE(64, 2) KVB_DECODE_CASE(64, 4) KVB_DECODE_CASE(64, 7) KVB_DECODE_CASE(64, 8)
#undef KVB_DECODE_CASE
    else return fail(KVB_ERR_UNSUPPORTED, "decode attention: head_dim %d with %d q heads per kv head not built", D, G);
    if (s != KVB_OK) return s;
    decode_combine_kernel<<<dim3((unsigned)Hq, (unsigned)(D / 32)), 32 * COMB_GROUPS, 0, st>>>(
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
