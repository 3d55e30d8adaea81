// Greedy decode on the blended cache: one new token per step through every layer.
//
// Everything here is bound by HBM traffic (each step reads all weights once, ~15 GB
// for Llama-3.1-8B, and every layer's cache up to the current position), so the
// kernels are CUDA-core kernels built for streaming, not tensor-core tiles:
//   decode_embed      - x = embed[tokens[pos]] (fp32)
//   gemv_kernel       - y = W a for one activation row held in shared memory as bf16;
//                       warp per output row (or row pair), 16-byte weight loads, 8 per
//                       lane in flight, all warps resident at once.  QKV and SwiGLU normalise the residual row
//                       themselves (RMSNorm prologue in every block); QKV computes the two
//                       rows of a rotation pair in one warp, applies RoPE at `pos` and writes
//                       q and the cache's K/V row `pos` (V as bf16-rounded fp16, like the
//                       prefill); the residual mode adds into x; SwiGLU computes gate and
//                       up rows in one warp
//   decode_attn       - split-KV attention of the new row over cache rows [0, pos]: one
//                       warp per split of 128 rows of one kv head, K/V tiles of 16 rows
//                       streamed by TMA into a per-warp ring, S^T = K Q^T and O^T += V^T P^T
//                       on mma.sync tiles with the group's q heads as the 8 columns, online
//                       softmax per head in fp32; the 4 warps of a CTA merge their
//                       (max, sum, O) in shared memory
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
// Four blocks per SM (<= 64 registers a thread): 32 warps per SM hold every row of the
// 4096-row GEMVs at once, so no warp takes a second row while others idle.
template <int MODE>
__global__ void __launch_bounds__(GEMV_THREADS, 4)
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
                dot_rows<true, 4>(p.W + ((int64_t)h * D + i) * K, p.W + ((int64_t)h * D + i + half) * K, act, K, lane,
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
                dot_rows<false, 8>(p.W + ((int64_t)(Hq + Hkv) * D + j) * K, nullptr, act, K, lane, a, unused);
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
                dot_rows<true, 4>(p.W + n * K, p.W2 + n * K, act, K, lane, a, b);
                if (lane == 0) p.y_bf16[n] = __bfloat16_as_ushort(__float2bfloat16_rn(a / (1.0f + __expf(-a)) * b));
            } else {
                dot_rows<false, 8>(p.W + n * K, nullptr, act, K, lane, a, b);
                if (lane == 0) p.y_f32[n] += a;
            }
        }
    }
}

// ---------------------------------------------------------------- decode attention
//
// One CTA = DA_WARPS warps of one kv head; warp w takes the split of `split` cache rows
// starting at (blockIdx.x * DA_WARPS + w) * split and streams it through its own ring of
// DA_STAGES stages of 16 rows (K and V tiles loaded by TMA, 128-byte swizzle).  The host
// sizes the splits so that all CTAs are resident at once (one wave: two CTAs per SM), so
// every warp pays the pipeline start-up once.  Per stage, with the G <= 8 q heads of the group as the 8
// columns of mma.sync m16n8k16 tiles (columns G..7 are zero q heads, never written out):
//   S^T [16 keys x 8 heads] = K [16 x D] . Q^T            (bf16, fp32 accumulate)
//   online softmax per head (column) in the log2 domain;
//   P^T as the B operand: fp16 pairs of the accumulator rows transposed by movmatrix,
//       as an fp16 head plus an fp16 remainder (~22-bit weights);
//   O^T [D x 8 heads] += V^T [D x 16 keys] . P^T          (fp16, V^T via ldmatrix.trans)
// so a stage costs about 60 warp instructions for 8 KB of K/V (D = 128), and the kernel is
// bound by the TMA stream.  The warps' (max, sum, O) are merged in shared memory and the
// CTA writes one partial per q head for decode_combine_kernel.

constexpr int DA_WARPS = 4;
constexpr int DA_THREADS = 32 * DA_WARPS;
constexpr int DA_STAGE_KEYS = 16;
constexpr int DA_STAGES = 3;
constexpr int DA_CTAS_PER_SM = 2;
constexpr int DA_MAX_SLOTS = 384;            // bound on resident CTAs (2 per SM, up to 192 SMs)
constexpr float DA_P_SHIFT = 15.f;           // softmax weights carried as p * 2^15

template <int D>
struct DaSmem {
    static constexpr int NB = D / 64;                    // 64-column (128-byte) boxes per row
    static constexpr int BOX = DA_STAGE_KEYS * 128;      // one box: 16 rows x 128 bytes
    static constexpr int STAGE = 2 * NB * BOX;           // K boxes, then V boxes
    static constexpr int RING = DA_WARPS * DA_STAGES * STAGE;
    static constexpr int OFF_BAR = RING;
    static constexpr int TOTAL = RING + 256 + 1024;      // barriers + flag, 1024-byte alignment slack
    // merge buffers (o [W][8][D], m and l [W][8], fp32) reuse the ring after the loop
    static_assert(DA_WARPS * 8 * D * 4 + 2 * DA_WARPS * 8 * 4 <= RING, "merge buffers");
};

// byte offset of the 16-byte unit `unit` (dims [8 unit, 8 unit + 8)) of row r in a set of
// 128-byte-swizzled boxes
template <int D>
KVB_DEV uint32_t da_off(int r, int unit) {
    return (uint32_t)((unit >> 3) * DaSmem<D>::BOX + r * 128 + (((unit & 7) ^ (r & 7)) << 4));
}

KVB_DEV void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr)
                 : "memory");
}
KVB_DEV void ldsm_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr)
                 : "memory");
}
KVB_DEV void mma16816_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                           uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
KVB_DEV void mma16816_f16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                          uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
KVB_DEV uint32_t movmatrix_trans(uint32_t a) {
    uint32_t d;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
    return d;
}

template <int D>
__global__ void __launch_bounds__(DA_THREADS, 2)
decode_attn_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                   const uint16_t* __restrict__ q, int G, int Hkv, const int32_t* __restrict__ pos_ptr,
                   int64_t max_pos, int n_blocks, int split, float sl2, float* __restrict__ pm,
                   float* __restrict__ pl, float* __restrict__ po, int* status) {
    using S = DaSmem<D>;
    constexpr int NB = S::NB;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);          // [DA_WARPS][DA_STAGES]
    volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + DA_WARPS * DA_STAGES);
    int pos;
    if (!pos_ok(pos_ptr, max_pos, status, pos)) return;
    if ((int)blockIdx.x >= n_blocks) return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int kvh = blockIdx.y;
    const int g8 = lane >> 2, t4 = lane & 3;
    if (threadIdx.x == 0) {
        for (int i = 0; i < DA_WARPS * DA_STAGES; ++i) mbar_init(&bars[i], 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (threadIdx.x == 32) { prefetch_tmap(&tmK); prefetch_tmap(&tmV); }
    __syncthreads();

    const int64_t start = ((int64_t)blockIdx.x * DA_WARPS + warp) * split;
    int64_t end = start + split;
    if (end > (int64_t)pos + 1) end = (int64_t)pos + 1;
    const int n_st = start < end ? (int)((end - start + DA_STAGE_KEYS - 1) / DA_STAGE_KEYS) : 0;
    uint8_t* ring = smem + warp * DA_STAGES * S::STAGE;
    uint64_t* wbar = bars + warp * DA_STAGES;
    auto issue = [&](int st) {            // lane 0: K and V rows of stage st into its slot
        uint8_t* dst = ring + (st % DA_STAGES) * S::STAGE;
        uint64_t* b = wbar + st % DA_STAGES;
        const int y = (int)(start + (int64_t)st * DA_STAGE_KEYS);
        mbar_expect_tx(b, S::STAGE);
#pragma unroll
        for (int c = 0; c < NB; ++c) tma_load_2d(dst + c * S::BOX, &tmK, b, kvh * D + c * 64, y);
#pragma unroll
        for (int c = 0; c < NB; ++c) tma_load_2d(dst + (NB + c) * S::BOX, &tmV, b, kvh * D + c * 64, y);
    };
    int issued = n_st < DA_STAGES ? n_st : DA_STAGES;
    if (lane == 0)
        for (int st = 0; st < issued; ++st) issue(st);

    // B operand of S^T = K Q^T: q head g8 of the group (zero columns for g8 >= G), dims
    // 16 ks + 2 t4 (+1) and 16 ks + 8 + 2 t4 (+1)
    uint32_t qb[D / 16][2];
    {
        const uint32_t* qrow = reinterpret_cast<const uint32_t*>(q + ((int64_t)kvh * G + g8) * D);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            qb[ks][0] = g8 < G ? __ldg(qrow + 8 * ks + t4) : 0u;
            qb[ks][1] = g8 < G ? __ldg(qrow + 8 * ks + 4 + t4) : 0u;
        }
    }
    float o[D / 16][4];
#pragma unroll
    for (int m = 0; m < D / 16; ++m) o[m][0] = o[m][1] = o[m][2] = o[m][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;     // heads 2 t4 and 2 t4 + 1
    // this lane's ldmatrix rows: K (A of S^T) and V (A of O^T, transposed)
    const int mm = lane >> 3;
    const int rk = ((mm & 1) << 3) | (lane & 7), uk = mm >> 1;
    const int rv = ((mm >> 1) << 3) | (lane & 7), uv = mm & 1;

    int st = 0;
    bool ok = true;
    for (; st < n_st; ++st) {
        const int slot = st % DA_STAGES;
        if (!mbar_wait_warp(wbar + slot, (uint32_t)(st / DA_STAGES) & 1, abort_flag, status)) {
            ok = false;
            break;
        }
        uint8_t* sp = ring + slot * S::STAGE;
        const uint32_t kb = smem_u32(sp), vb = kb + NB * S::BOX;
        const int64_t key0 = start + (int64_t)st * DA_STAGE_KEYS;
        const int nvalid = (int)((end - key0) < DA_STAGE_KEYS ? (end - key0) : DA_STAGE_KEYS);
        if (nvalid < DA_STAGE_KEYS) {
            // rows past the current position: zero their V (the cache may hold anything there)
            uint4* vz = reinterpret_cast<uint4*>(sp + NB * S::BOX);
            for (int i = lane; i < NB * DA_STAGE_KEYS * 8; i += 32)
                if (((i >> 3) & (DA_STAGE_KEYS - 1)) >= nvalid) vz[i] = make_uint4(0u, 0u, 0u, 0u);
            __syncwarp();
        }
        // S^T: rows = keys g8 and g8 + 8, columns = heads 2 t4 and 2 t4 + 1.  Every 16-dim
        // slice gets its own accumulator (one MMA from zero: the tensor core's sum of 16 exact
        // bf16 products) and the slices are added in fp32 afterwards, instead of chaining the
        // MMAs through one accumulator whose running sum the tensor core rounds at every step.
        float sk[D / 16][4];
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(kb + da_off<D>(rk, 2 * ks + uk), a0, a1, a2, a3);
            sk[ks][0] = sk[ks][1] = sk[ks][2] = sk[ks][3] = 0.f;
            mma16816_bf16(sk[ks], a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
        }
        float sacc[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
#pragma unroll
            for (int w = 1; w < D / 16; w <<= 1)
#pragma unroll
                for (int ks = 0; ks + w < D / 16; ks += 2 * w) sk[ks][i] += sk[ks + w][i];
            sacc[i] = sk[0][i];
        }
        const bool v0 = g8 < nvalid, v1 = g8 + 8 < nvalid;
        const float x00 = v0 ? sacc[0] * sl2 : -INFINITY, x01 = v0 ? sacc[1] * sl2 : -INFINITY;
        const float x10 = v1 ? sacc[2] * sl2 : -INFINITY, x11 = v1 ? sacc[3] * sl2 : -INFINITY;
        float mx0 = fmaxf(x00, x10), mx1 = fmaxf(x01, x11);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
        }
        // key 0 of every stage is valid, so the new maxima are finite
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        const float al0 = mn0 != m0 ? fast_exp2(m0 - mn0) : 1.f;   // 0 when m0 = -inf
        const float al1 = mn1 != m1 ? fast_exp2(m1 - mn1) : 1.f;
        m0 = mn0;
        m1 = mn1;
        // weights scaled by 2^15 (<= 32768, inside fp16's range): the fp16 head and remainder
        // below then stay normal numbers down to weights of 2^-17; l and O carry the same
        // factor, so O / l is unchanged
        const float r0 = mn0 - DA_P_SHIFT, r1 = mn1 - DA_P_SHIFT;
        const float p00 = fast_exp2(x00 - r0), p01 = fast_exp2(x01 - r1);
        const float p10 = fast_exp2(x10 - r0), p11 = fast_exp2(x11 - r1);
        l0 = l0 * al0 + (p00 + p10);
        l1 = l1 * al1 + (p01 + p11);
        // P^T as B: rows = keys, columns = heads.  Each weight is split into an fp16 head and
        // an fp16 remainder, both multiplied into the same accumulator, so the weights keep ~22
        // bits: a single fp16 rounding (11 bits) moved the output of a decode step by more
        // than fp32-vs-fp64 accumulation does.
        uint32_t ph0 = pack_f16(p00, p01), ph1 = pack_f16(p10, p11);
        const float2 h0 = __half22float2(*reinterpret_cast<const __half2*>(&ph0));
        const float2 h1 = __half22float2(*reinterpret_cast<const __half2*>(&ph1));
        const uint32_t pl0 = pack_f16(p00 - h0.x, p01 - h0.y), pl1 = pack_f16(p10 - h1.x, p11 - h1.y);
        const uint32_t pb0 = movmatrix_trans(ph0), pb1 = movmatrix_trans(ph1);
        const uint32_t pr0 = movmatrix_trans(pl0), pr1 = movmatrix_trans(pl1);
        // O^T: rows = dims 16 m + g8 (+8), columns = heads 2 t4 (+1); this stage's sum in its
        // own accumulator, folded into the running O with the rescale in fp32
#pragma unroll
        for (int m = 0; m < D / 16; ++m) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4_trans(vb + da_off<D>(rv, 2 * m + uv), a0, a1, a2, a3);
            float so[4] = {0.f, 0.f, 0.f, 0.f};
            mma16816_f16(so, a0, a1, a2, a3, pb0, pb1);
            mma16816_f16(so, a0, a1, a2, a3, pr0, pr1);
            o[m][0] = fmaf(o[m][0], al0, so[0]);
            o[m][1] = fmaf(o[m][1], al1, so[1]);
            o[m][2] = fmaf(o[m][2], al0, so[2]);
            o[m][3] = fmaf(o[m][3], al1, so[3]);
        }
        if (st + DA_STAGES < n_st) {
            // every lane is done with this slot: order its reads before the async-proxy refill
            fence_async_smem();
            __syncwarp();
            if (lane == 0) issue(st + DA_STAGES);
            ++issued;
        }
    }
    if (!ok && lane == 0) {
        // let the loads already issued land before the CTA's shared memory goes away
        const uint64_t t0 = globaltimer();
        for (int j = st; j < issued; ++j)
            while (!mbar_try_wait(wbar + j % DA_STAGES, (uint32_t)(j / DA_STAGES) & 1) &&
                   globaltimer() - t0 < 1000000ull) {}
    }
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, off);
        l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }
    __syncthreads();
    if (*abort_flag) return;
    // merge the warps of this CTA (buffers reuse the ring: every load has landed)
    float* sm_o = reinterpret_cast<float*>(smem);                 // [W][8][D]
    float* sm_m = sm_o + DA_WARPS * 8 * D;                        // [W][8]
    float* sm_l = sm_m + DA_WARPS * 8;
    {
        float* w0 = sm_o + (warp * 8 + 2 * t4) * D;
        float* w1 = w0 + D;
#pragma unroll
        for (int m = 0; m < D / 16; ++m) {
            w0[16 * m + g8] = o[m][0];
            w1[16 * m + g8] = o[m][1];
            w0[16 * m + g8 + 8] = o[m][2];
            w1[16 * m + g8 + 8] = o[m][3];
        }
        if (g8 == 0) {
            sm_m[warp * 8 + 2 * t4] = m0; sm_m[warp * 8 + 2 * t4 + 1] = m1;
            sm_l[warp * 8 + 2 * t4] = l0; sm_l[warp * 8 + 2 * t4 + 1] = l1;
        }
    }
    __syncthreads();
    const int Hq = Hkv * G;
    const int64_t base = (int64_t)blockIdx.x * Hq + (int64_t)kvh * G;
    for (int i = threadIdx.x; i < G * D; i += DA_THREADS) {
        const int h = i / D, d = i % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < DA_WARPS; ++w) M = fmaxf(M, sm_m[w * 8 + h]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < DA_WARPS; ++w) {
            const float mw = sm_m[w * 8 + h];
            const float c = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
            L += c * sm_l[w * 8 + h];
            O += c * sm_o[(w * 8 + h) * D + d];
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

template <int D>
kvb_status run_attn(const CUtensorMap& tk, const CUtensorMap& tv, const uint16_t* q, int G, int Hkv,
                    const int32_t* pos, int64_t max_pos, int n_blocks, int split, float sl2, float* pm, float* pl,
                    float* po, int* status, cudaStream_t st) {
    static std::atomic<uint64_t> smem_set{0};
    auto kern = decode_attn_kernel<D>;
    kvb_status s = ensure_smem_limit((const void*)kern, DaSmem<D>::TOTAL, smem_set, "decode attention smem");
    if (s != KVB_OK) return s;
    const dim3 grid((unsigned)n_blocks, (unsigned)Hkv);
    kern<<<grid, DA_THREADS, DaSmem<D>::TOTAL, st>>>(tk, tv, q, G, Hkv, pos, max_pos, n_blocks, split, sl2, pm, pl,
                                                     po, status);
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

// Bound on the CTA partials (per kv head) of the decode attention for positions below
// max_pos: the workspace is laid out with it, whatever device runs the kernel.
int decode_splits(int64_t max_pos, int Hkv) {
    const int64_t by_rows = (max_pos + DA_WARPS * DA_STAGE_KEYS - 1) / (DA_WARPS * DA_STAGE_KEYS);
    const int64_t by_slots = Hkv > 0 && DA_MAX_SLOTS / Hkv > 0 ? DA_MAX_SLOTS / Hkv : 1;
    return (int)(by_rows < by_slots ? by_rows : by_slots);
}

kvb_status launch_decode_attn(const uint16_t* q, const uint16_t* kc, const uint16_t* vc, int Hq, int Hkv, int D,
                              const int32_t* pos, int64_t max_pos, float sl2, float* pm, float* pl, float* po,
                              uint16_t* out, int* status, cudaStream_t st) {
    if (Hkv <= 0 || Hq % Hkv || Hq / Hkv > 8)
        return fail(KVB_ERR_UNSUPPORTED, "decode attention: at most 8 q heads per kv head (Hq %d, Hkv %d)", Hq, Hkv);
    if (D != 64 && D != 128) return fail(KVB_ERR_UNSUPPORTED, "decode attention: head_dim %d not built", D);
    const int G = Hq / Hkv;
    const uint64_t kvd = (uint64_t)Hkv * D;
    CUtensorMap tk, tv;
    kvb_status s = make_tmap_2d(&tk, kc, kvd, (uint64_t)max_pos, kvd, 64, DA_STAGE_KEYS);
    if (s != KVB_OK) return s;
    s = make_tmap_2d(&tv, vc, kvd, (uint64_t)max_pos, kvd, 64, DA_STAGE_KEYS, CU_TENSOR_MAP_DATA_TYPE_FLOAT16);
    if (s != KVB_OK) return s;
    // one wave: at most DA_CTAS_PER_SM CTAs per SM over all kv heads, each warp's split a
    // multiple of the 16-row stage, the splits covering rows [0, max_pos)
    int64_t n_blocks = (int64_t)DA_CTAS_PER_SM * num_sms() / Hkv;
    const int cap = decode_splits(max_pos, Hkv);
    if (n_blocks > cap) n_blocks = cap;
    if (n_blocks < 1) n_blocks = 1;
    int64_t split = (max_pos + n_blocks * DA_WARPS - 1) / (n_blocks * DA_WARPS);
    split = (split + DA_STAGE_KEYS - 1) / DA_STAGE_KEYS * DA_STAGE_KEYS;
    n_blocks = (max_pos + split * DA_WARPS - 1) / (split * DA_WARPS);
    if (split > 0x7FFFFFFF / DA_WARPS) return fail(KVB_ERR_INVALID_ARG, "decode attention: max_pos too large");
    s = D == 128 ? run_attn<128>(tk, tv, q, G, Hkv, pos, max_pos, (int)n_blocks, (int)split, sl2, pm, pl, po, status, st)
                 : run_attn<64>(tk, tv, q, G, Hkv, pos, max_pos, (int)n_blocks, (int)split, sl2, pm, pl, po, status, st);
    if (s != KVB_OK) return s;
    decode_combine_kernel<<<dim3((unsigned)Hq, (unsigned)(D / 32)), 32 * COMB_GROUPS, 0, st>>>(
        pm, pl, po, pos, max_pos, (int)(split * DA_WARPS), Hq, D, out, status);
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
