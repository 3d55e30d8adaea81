// First token: logits = h W^T over the vocabulary for a few rows, and their argmax
// (ties to the lower token id).  Memory-bound: the vocab x hidden bf16 matrix is
// streamed once with 16-byte loads, one warp per vocabulary row at a time, every
// loaded chunk used for all n rows (held in shared memory as fp32).  The argmax
// is reduced per warp and merged with one 64-bit atomicMax per row on an
// order-preserving key (logit bits in the high word, inverted id in the low word).
#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

constexpr int THREADS = 256;
constexpr int BATCH = 8;

KVB_DEV uint32_t orderable(float f) {
    const uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__global__ void __launch_bounds__(THREADS)
lmhead_kernel(const uint16_t* __restrict__ W, int64_t vocab, int H, const float* __restrict__ x, int n,
              float* __restrict__ logits, unsigned long long* __restrict__ keys) {
    extern __shared__ float xs[];   // [n][H]
    for (int i = threadIdx.x; i < n * H; i += blockDim.x) xs[i] = x[i];
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
    unsigned long long best[KVB_LMHEAD_MAX_ROWS];
#pragma unroll
    for (int r = 0; r < KVB_LMHEAD_MAX_ROWS; ++r) best[r] = 0ull;
    const int vec = H / 8;
    for (int64_t v = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); v < vocab; v += warps) {
        const uint4* wr = reinterpret_cast<const uint4*>(W + v * H);
        float acc[KVB_LMHEAD_MAX_ROWS];
#pragma unroll
        for (int r = 0; r < KVB_LMHEAD_MAX_ROWS; ++r) acc[r] = 0.f;
        // BATCH independent 16-byte loads per lane in flight before any arithmetic
        for (int c0 = lane; c0 < vec; c0 += 32 * BATCH) {
            uint4 wv[BATCH];
#pragma unroll
            for (int u = 0; u < BATCH; ++u) {
                const int c = c0 + 32 * u;
                wv[u] = c < vec ? __ldcs(wr + c) : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < BATCH; ++u) {
                const int c = c0 + 32 * u;
                if (c >= vec) break;
                const uint4 w = wv[u];
                const float wf[8] = {bf16_lo(w.x), bf16_hi(w.x), bf16_lo(w.y), bf16_hi(w.y),
                                     bf16_lo(w.z), bf16_hi(w.z), bf16_lo(w.w), bf16_hi(w.w)};
#pragma unroll
                for (int r = 0; r < KVB_LMHEAD_MAX_ROWS; ++r) {
                    if (r < n) {
                        const float4* xr = reinterpret_cast<const float4*>(xs + r * H + c * 8);
                        const float4 a = xr[0], b = xr[1];
                        acc[r] = fmaf(wf[0], a.x, acc[r]); acc[r] = fmaf(wf[1], a.y, acc[r]);
                        acc[r] = fmaf(wf[2], a.z, acc[r]); acc[r] = fmaf(wf[3], a.w, acc[r]);
                        acc[r] = fmaf(wf[4], b.x, acc[r]); acc[r] = fmaf(wf[5], b.y, acc[r]);
                        acc[r] = fmaf(wf[6], b.z, acc[r]); acc[r] = fmaf(wf[7], b.w, acc[r]);
                    }
                }
            }
        }
#pragma unroll
        for (int r = 0; r < KVB_LMHEAD_MAX_ROWS; ++r) {
            if (r < n) {
                float s = acc[r];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
                if (lane == 0) {
                    if (logits) logits[(int64_t)r * vocab + v] = s;
                    const unsigned long long key =
                        ((unsigned long long)orderable(s) << 32) | (0xFFFFFFFFull - (unsigned long long)v);
                    best[r] = key > best[r] ? key : best[r];
                }
            }
        }
    }
    if (lane == 0) {
#pragma unroll
        for (int r = 0; r < KVB_LMHEAD_MAX_ROWS; ++r)
            if (r < n && best[r]) atomicMax(keys + r, best[r]);
    }
}

__global__ void argmax_finalize(const unsigned long long* keys, int n, int32_t* tokens) {
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r < n) tokens[r] = (int32_t)(0xFFFFFFFFull - (keys[r] & 0xFFFFFFFFull));
}

}  // namespace

kvb_status launch_lmhead(const uint16_t* W, int64_t vocab, int H, const float* x, int n, float* logits,
                         unsigned long long* keys, int32_t* tokens, cudaStream_t st) {
    if (n <= 0) return KVB_OK;
    kvb_status s = cuda_ok(cudaMemsetAsync(keys, 0, (size_t)n * sizeof(unsigned long long), st), "lm head: clear keys");
    if (s != KVB_OK) return s;
    const size_t smem = (size_t)n * H * sizeof(float);
    static std::atomic<uint64_t> smem_set{0};
    s = ensure_smem_limit((const void*)lmhead_kernel, KVB_LMHEAD_MAX_ROWS * 8192 * 4, smem_set, "lm head smem");
    if (s != KVB_OK) return s;
    // one wave of resident blocks, each warp striding over the vocabulary
    int per_sm = 0;
    s = cuda_ok(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, lmhead_kernel, THREADS, smem), "lm head occupancy");
    if (s != KVB_OK) return s;
    int64_t blocks = (vocab + THREADS / 32 - 1) / (THREADS / 32);
    const int64_t cap = (int64_t)num_sms() * (per_sm > 0 ? per_sm : 1);
    if (blocks > cap) blocks = cap;
    lmhead_kernel<<<(unsigned)blocks, THREADS, smem, st>>>(W, vocab, H, x, n, logits, keys);
    count_launch();
    s = cuda_ok(cudaGetLastError(), "lm head launch");
    if (s != KVB_OK) return s;
    argmax_finalize<<<(n + 31) / 32, 32, 0, st>>>(keys, n, tokens);
    count_launch();
    return cuda_ok(cudaGetLastError(), "argmax launch");
}

}  // namespace kvb
