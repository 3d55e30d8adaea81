// Fixed-position selections (EPIC / KVLink windows) and the per-token key-deviation
// histogram.  Both are tiny next to the prefill; they are written for clarity:
//   window select: clear a flag per context row, mark every row of every window,
//                  then one CTA compacts the flags in order (block scan per pass);
//   histogram:     deviation per row (the HKVD deviation kernel), then one thread per
//                  row counts the edges at or below its value and adds one to that bin
//                  (shared-memory counts, one global atomic per bin per block).
#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

constexpr int COMPACT_THREADS = 1024;

__global__ void mark_windows(const int32_t* __restrict__ win_start, int32_t n_win, int32_t window, int64_t n_ctx,
                             uint8_t* __restrict__ flags) {
    const int64_t total = (int64_t)n_win * window;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = (int64_t)win_start[t / window] + t % window;
        if (i >= 0 && i < n_ctx) flags[i] = 1;
    }
}

__device__ uint32_t scan_exclusive(uint32_t v, uint32_t* warp_sums, uint32_t* total) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[w] = x;
    __syncthreads();
    if (w == 0) {
        uint32_t s = lane < (int)(blockDim.x / 32) ? warp_sums[lane] : 0u;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        warp_sums[lane] = s;
    }
    __syncthreads();
    const uint32_t before = (w > 0 ? warp_sums[w - 1] : 0u) + x - v;
    *total = warp_sums[blockDim.x / 32 - 1];
    __syncthreads();
    return before;
}

// Ascending indices of the set flags; 16 flags per thread per pass.
__global__ void __launch_bounds__(COMPACT_THREADS)
compact_flags(const uint8_t* __restrict__ flags, int64_t n, int32_t* __restrict__ sel, int64_t* __restrict__ k_out) {
    __shared__ uint32_t warp_sums[32];
    constexpr int PER = 16;
    int64_t base_out = 0;
    for (int64_t base = 0; base < n; base += (int64_t)COMPACT_THREADS * PER) {
        const int64_t beg = base + (int64_t)threadIdx.x * PER;
        uint32_t bits = 0;
#pragma unroll
        for (int j = 0; j < PER; ++j)
            if (beg + j < n && flags[beg + j]) bits |= 1u << j;
        uint32_t total;
        const uint32_t before = scan_exclusive(__popc(bits), warp_sums, &total);
        int64_t o = base_out + before;
        while (bits) {
            const int j = __ffs(bits) - 1;
            bits &= bits - 1;
            sel[o++] = (int32_t)(beg + j);
        }
        base_out += total;
    }
    if (threadIdx.x == 0) *k_out = base_out;
}

__global__ void __launch_bounds__(256)
histogram_kernel(const float* __restrict__ dev, int64_t n, const float* __restrict__ edges, int n_edges,
                 unsigned long long* __restrict__ hist) {
    extern __shared__ uint32_t sm[];   // edges (as float bits) then counts [n_edges + 1]
    float* e = reinterpret_cast<float*>(sm);
    uint32_t* cnt = sm + n_edges;
    for (int j = threadIdx.x; j < n_edges; j += blockDim.x) e[j] = edges[j];
    for (int j = threadIdx.x; j <= n_edges; j += blockDim.x) cnt[j] = 0;
    __syncthreads();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const float d = dev[i];
        int b = 0;
        for (int j = 0; j < n_edges; ++j) b += (d >= e[j]);
        atomicAdd(&cnt[b], 1u);
    }
    __syncthreads();
    for (int j = threadIdx.x; j <= n_edges; j += blockDim.x)
        if (cnt[j]) atomicAdd(hist + j, (unsigned long long)cnt[j]);
}

}  // namespace

kvb_status launch_window_select(const int32_t* win_start, int32_t n_win, int32_t window, int64_t n_ctx,
                                uint8_t* flags, int32_t* sel, int64_t* k_out, cudaStream_t st) {
    kvb_status s = cuda_ok(cudaMemsetAsync(flags, 0, (size_t)n_ctx, st), "window select: clear flags");
    if (s != KVB_OK) return s;
    const int64_t total = (int64_t)n_win * window;
    if (total > 0) {
        int64_t blocks = (total + 255) / 256;
        if (blocks > (int64_t)num_sms() * 8) blocks = (int64_t)num_sms() * 8;
        mark_windows<<<(unsigned)blocks, 256, 0, st>>>(win_start, n_win, window, n_ctx, flags);
        count_launch();
        s = cuda_ok(cudaGetLastError(), "window mark launch");
        if (s != KVB_OK) return s;
    }
    compact_flags<<<1, COMPACT_THREADS, 0, st>>>(flags, n_ctx, sel, k_out);
    count_launch();
    return cuda_ok(cudaGetLastError(), "window compact launch");
}

kvb_status launch_deviation_histogram(const uint16_t* ka, int64_t lda, const uint16_t* kb, int64_t ldb, int64_t n,
                                      int kv_dim, const float* edges, int n_edges, float* dev,
                                      unsigned long long* hist, cudaStream_t st) {
    kvb_status s = cuda_ok(cudaMemsetAsync(hist, 0, (size_t)(n_edges + 1) * sizeof(unsigned long long), st),
                           "histogram: clear");
    if (s != KVB_OK || n == 0) return s;
    s = launch_deviation(ka, lda, kb, ldb, n, kv_dim, dev, st);
    if (s != KVB_OK) return s;
    int64_t blocks = (n + 255) / 256;
    if (blocks > (int64_t)num_sms() * 4) blocks = (int64_t)num_sms() * 4;
    histogram_kernel<<<(unsigned)blocks, 256, (size_t)(2 * n_edges + 1) * 4, st>>>(dev, n, edges, n_edges, hist);
    count_launch();
    return cuda_ok(cudaGetLastError(), "histogram launch");
}

}  // namespace kvb
