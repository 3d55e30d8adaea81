// HKVD selection: per-token squared key deviation and an exact top-k.
//
// dev[i] = sum_{h,d} (K_fresh[i,h,d] - K_cached[i,h,d])^2 in fp32, one warp per
// row with 16-byte loads.  Top-k is a radix select on the fp32 bit patterns
// (dev >= 0, so the unsigned order of the bits is the numeric order): four
// 8-bit passes narrow the k-th largest key with warp-aggregated shared-memory
// histograms, then an ordered compaction writes the selected indices in
// ascending order, taking keys equal to the threshold from the lowest index up.
// It runs on one thread-block cluster of 8 CTAs x 1024 threads: each CTA owns a
// contiguous eighth of the keys (up to 16 per thread, held in registers for the
// whole select), the CTAs' histograms are summed through distributed shared memory
// after every pass (each CTA reaches the same digit), and the compaction takes its
// output offset from the counts of the CTAs before it.
#include <cooperative_groups.h>

#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

constexpr int TOPK_THREADS = 1024;

__global__ void __launch_bounds__(256)
dev_kernel(const uint16_t* __restrict__ kf, int64_t ldf, const uint16_t* __restrict__ kc, int64_t ldc, int64_t n,
           int kv_dim, float* __restrict__ dev) {
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
    const int lane = threadIdx.x & 31;
    const int vec = kv_dim / 8;
    for (int64_t r = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); r < n; r += warps) {
        const uint4* a = reinterpret_cast<const uint4*>(kf + r * ldf);
        const uint4* b = reinterpret_cast<const uint4*>(kc + r * ldc);
        float acc = 0.f;
        for (int c = lane; c < vec; c += 32) {
            const uint4 x = a[c], y = b[c];
            const uint32_t xv[4] = {x.x, x.y, x.z, x.w}, yv[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float d0 = bf16_lo(xv[e]) - bf16_lo(yv[e]);
                const float d1 = bf16_hi(xv[e]) - bf16_hi(yv[e]);
                acc = fmaf(d0, d0, acc);
                acc = fmaf(d1, d1, acc);
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) dev[r] = acc;
    }
}

// exclusive prefix sum over the CTA; returns the total through *total
__device__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* warp_sums, uint32_t* total) {
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
        warp_sums[lane] = s;   // inclusive over warps
    }
    __syncthreads();
    const uint32_t before = (w > 0 ? warp_sums[w - 1] : 0u) + x - v;
    *total = warp_sums[blockDim.x / 32 - 1];
    __syncthreads();
    return before;
}

constexpr int TK_CTAS = 8, TK_KPT = 16;
constexpr int64_t TK_CLUSTER_MAX = (int64_t)TK_CTAS * TOPK_THREADS * TK_KPT;   // 131,072 keys

// warp-aggregated histogram increment for the keys whose bits above `shift + 8` match
KVB_DEV void hist_add(uint32_t* hist, uint32_t key, uint32_t mask, uint32_t prefix, int shift) {
    const bool in = (key & mask) == prefix;
    const uint32_t act = __activemask();
    const uint32_t want = __ballot_sync(act, in);
    if (in) {
        const uint32_t d = (key >> shift) & 255u;
        const uint32_t peers = __match_any_sync(want, d);
        if ((threadIdx.x & 31) == (__ffs(peers) - 1)) atomicAdd(&hist[d], __popc(peers));
    }
}

// Exact top-k of n <= TK_CLUSTER_MAX keys on one cluster of TK_CTAS CTAs.
__global__ void __cluster_dims__(TK_CTAS, 1, 1) __launch_bounds__(TOPK_THREADS, 1)
topk_cluster_kernel(const float* __restrict__ dev, int64_t n, int64_t k, int32_t* __restrict__ sel) {
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    __shared__ uint32_t hist[256];
    __shared__ uint32_t tot[256];
    __shared__ uint32_t warp_sums[32];
    __shared__ uint32_t s_digit, s_remaining;
    __shared__ uint32_t cnt[2];               // this CTA's keys above / equal to the threshold
    const int tid = threadIdx.x;
    // this thread's keys: indices [tbeg, tbeg + nk), contiguous, so the compaction keeps index order
    const int64_t tbeg = (int64_t)rank * TOPK_THREADS * TK_KPT + (int64_t)tid * TK_KPT;
    const int nk = (int)max((int64_t)0, min((int64_t)TK_KPT, n - tbeg));
    if (k <= 0) return;                       // k and n are the same for every CTA of the cluster
    if (k >= n) {
        for (int u = 0; u < nk; ++u) sel[tbeg + u] = (int32_t)(tbeg + u);
        return;
    }
    uint32_t key[TK_KPT];
#pragma unroll
    for (int u = 0; u < TK_KPT; ++u) key[u] = u < nk ? __float_as_uint(__ldg(dev + tbeg + u)) : 0u;
    uint32_t prefix = 0, mask = 0, remaining = (uint32_t)k;
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        if (tid < 256) hist[tid] = 0;
        __syncthreads();
#pragma unroll
        for (int u = 0; u < TK_KPT; ++u)
            if (u < nk) hist_add(hist, key[u], mask, prefix, shift);
        cluster.sync();                       // every CTA's histogram is complete
        if (tid < 256) {
            uint32_t sum = 0;
#pragma unroll
            for (int r = 0; r < TK_CTAS; ++r) sum += *cluster.map_shared_rank(&hist[tid], r);
            tot[tid] = sum;
        }
        __syncthreads();
        if (tid == 0) {
            uint32_t cum = 0;
            for (int d = 255; d >= 0; --d) {
                if (cum + tot[d] >= remaining) { s_digit = (uint32_t)d; s_remaining = remaining - cum; break; }
                cum += tot[d];
            }
        }
        __syncthreads();
        prefix |= s_digit << shift;
        mask |= 255u << shift;
        remaining = s_remaining;
        cluster.sync();                       // no CTA clears its histogram while another still reads it
    }
    // threshold key `prefix`: take every key above it and the first `remaining` equal ones
    uint32_t gt = 0, eq = 0;
#pragma unroll
    for (int u = 0; u < TK_KPT; ++u)
        if (u < nk) { gt += key[u] > prefix; eq += key[u] == prefix; }
    uint32_t gt_tot, eq_tot;
    const uint32_t gt_before = block_exclusive_scan(gt, warp_sums, &gt_tot);
    const uint32_t eq_before = block_exclusive_scan(eq, warp_sums, &eq_tot);
    if (tid == 0) { cnt[0] = gt_tot; cnt[1] = eq_tot; }
    cluster.sync();
    uint32_t gt_prev = 0, eq_prev = 0;        // counts of the CTAs holding lower indices
    for (int r = 0; r < rank; ++r) {
        gt_prev += *cluster.map_shared_rank(&cnt[0], r);
        eq_prev += *cluster.map_shared_rank(&cnt[1], r);
    }
    uint32_t eq_seen = eq_prev + eq_before;
    uint32_t out = gt_prev + gt_before + (eq_seen < remaining ? eq_seen : remaining);
#pragma unroll
    for (int u = 0; u < TK_KPT; ++u) {
        if (u < nk) {
            bool take = key[u] > prefix;
            if (key[u] == prefix) { take = eq_seen < remaining; ++eq_seen; }
            if (take) sel[out++] = (int32_t)(tbeg + u);
        }
    }
    cluster.sync();                           // keep this CTA's counts readable until every CTA has read them
}

// One CTA for any n (the cluster kernel above covers n <= TK_CLUSTER_MAX).
__global__ void __launch_bounds__(TOPK_THREADS)
topk_kernel(const float* __restrict__ dev, int64_t n, int64_t k, int32_t* __restrict__ sel) {
    __shared__ uint32_t hist[256];
    __shared__ uint32_t warp_sums[32];
    __shared__ uint32_t s_digit, s_remaining;
    const int tid = threadIdx.x;
    if (k <= 0) return;
    if (k >= n) {
        for (int64_t i = tid; i < n; i += TOPK_THREADS) sel[i] = (int32_t)i;
        return;
    }
    uint32_t prefix = 0, mask = 0, remaining = (uint32_t)k;
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        for (int i = tid; i < 256; i += TOPK_THREADS) hist[i] = 0;
        __syncthreads();
        for (int64_t i = tid; i < n; i += TOPK_THREADS) {
            const uint32_t key = __float_as_uint(__ldg(dev + i));
            const bool in = (key & mask) == prefix;
            const uint32_t act = __activemask();
            const uint32_t want = __ballot_sync(act, in);
            if (in) {
                const uint32_t d = (key >> shift) & 255u;
                const uint32_t peers = __match_any_sync(want, d);
                if ((threadIdx.x & 31) == (__ffs(peers) - 1)) atomicAdd(&hist[d], __popc(peers));
            }
        }
        __syncthreads();
        if (tid == 0) {
            uint32_t cum = 0;
            for (int d = 255; d >= 0; --d) {
                if (cum + hist[d] >= remaining) { s_digit = (uint32_t)d; s_remaining = remaining - cum; break; }
                cum += hist[d];
            }
        }
        __syncthreads();
        prefix |= s_digit << shift;
        mask |= 255u << shift;
        remaining = s_remaining;
        __syncthreads();
    }
    // threshold key `prefix`; take every key above it and the first `remaining` equal ones
    const int64_t seg = (n + TOPK_THREADS - 1) / TOPK_THREADS;
    const int64_t beg = (int64_t)tid * seg;
    const int64_t end = beg + seg < n ? beg + seg : n;
    uint32_t gt = 0, eq = 0;
    for (int64_t i = beg; i < end; ++i) {
        const uint32_t key = __float_as_uint(dev[i]);
        gt += key > prefix;
        eq += key == prefix;
    }
    uint32_t gt_tot, eq_tot;
    const uint32_t gt_before = block_exclusive_scan(gt, warp_sums, &gt_tot);
    const uint32_t eq_before = block_exclusive_scan(eq, warp_sums, &eq_tot);
    uint32_t out = gt_before + (eq_before < remaining ? eq_before : remaining);
    uint32_t eq_seen = eq_before;
    for (int64_t i = beg; i < end; ++i) {
        const uint32_t key = __float_as_uint(dev[i]);
        bool take = key > prefix;
        if (key == prefix) { take = eq_seen < remaining; ++eq_seen; }
        if (take) sel[out++] = (int32_t)i;
    }
}

// A wait that nothing completes: the bounded mbarrier wait gives up after limit_ns
// and records KVB_ERR_TIMEOUT (test hook for the kernels' timeout path).
__global__ void wait_timeout_kernel(int* status, uint64_t limit_ns) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    mbar_wait(&bar, 0, &abort_flag, status, limit_ns);
    __syncthreads();
}

}  // namespace

kvb_status launch_wait_timeout(int* status, uint64_t limit_ns, cudaStream_t st) {
    wait_timeout_kernel<<<1, 32, 0, st>>>(status, limit_ns);
    count_launch();
    return cuda_ok(cudaGetLastError(), "wait-timeout launch");
}

size_t hkvd_ws_bytes(int64_t) { return 0; }

kvb_status launch_deviation(const uint16_t* ka, int64_t lda, const uint16_t* kb, int64_t ldb, int64_t n, int kv_dim,
                            float* dev, cudaStream_t st) {
    int64_t blocks = (n + 7) / 8;
    const int64_t cap = (int64_t)num_sms() * 16;
    if (blocks > cap) blocks = cap;
    dev_kernel<<<(unsigned)blocks, 256, 0, st>>>(ka, lda, kb, ldb, n, kv_dim, dev);
    count_launch();
    return cuda_ok(cudaGetLastError(), "deviation launch");
}

kvb_status launch_hkvd(const uint16_t* k_fresh, int64_t ld_fresh, const uint16_t* k_cached, int64_t ld_cached,
                       int64_t n_ctx, int kv_dim, int64_t k, int32_t* sel_out, float* dev_out, void*,
                       cudaStream_t st) {
    if (n_ctx <= 0) return KVB_OK;
    int64_t blocks = (n_ctx + 7) / 8;
    const int64_t cap = (int64_t)num_sms() * 16;
    if (blocks > cap) blocks = cap;
    dev_kernel<<<(unsigned)blocks, 256, 0, st>>>(k_fresh, ld_fresh, k_cached, ld_cached, n_ctx, kv_dim, dev_out);
    count_launch();
    kvb_status s = cuda_ok(cudaGetLastError(), "deviation launch");
    if (s != KVB_OK || k <= 0) return s;
    if (n_ctx <= TK_CLUSTER_MAX)
        topk_cluster_kernel<<<TK_CTAS, TOPK_THREADS, 0, st>>>(dev_out, n_ctx, k, sel_out);
    else
        topk_kernel<<<1, TOPK_THREADS, 0, st>>>(dev_out, n_ctx, k, sel_out);
    count_launch();
    return cuda_ok(cudaGetLastError(), "top-k launch");
}

}  // namespace kvb
