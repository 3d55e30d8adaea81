// Sparse-query causal GQA flash attention on the 5th-generation tensor cores.
//
// Each CTA owns one (block of query rows, kv head) unit; units are numbered kv head
// major, heaviest row block first within a head, so that the CTAs resident at a time read
// the K/V of one or two kv heads (63 MB each at 124k keys), which L2 holds.  The G = Hq/Hkv query heads
// that share kv head g are packed with RPB = floor(128/G) query rows into the 128
// rows of one MMA tile (lane = row_in_block * G + head_in_group; the last 128 - RPB*G
// lanes idle when G does not divide 128), so every K/V tile loaded serves all G heads.
// Row r attends cache rows [lo_r, hi_r] where hi_r is the row's own cache index: this
// one predicate covers the sparse recompute rows of the selective layers, the dense
// causal prefill and the block-diagonal per-chunk prefill.
//
// Both A operands live in tensor memory, so each MMA reads only its K or V tile
// from shared memory: with A and B both in shared memory an M128 x N128 step
// needs the whole shared-memory bandwidth on its own, before the TMA writes.
// Key tiles are 144 rows: the widest that leaves room in the 512 TMEM columns for two S
// buffers, O and Q while three K/V stages (216 KB) fit in shared memory; every tile's
// barrier waits and commits then cover 1,152 cycles of MMAs instead of 1,024 with
// 128-key tiles.
// TMEM columns: S buffers [0, 144) and [160, 304) (P_j is written over the first 72
// columns of S_j's buffer), O [320, 448), Q [448, 512).
//
// The MMAs are issued by two threads.  The tensor pipe's instruction queue is shallow,
// so a thread that issues an MMA waits for roughly its execution, and every mbarrier
// wait and commit on an issuing thread leaves the pipe idle for its duration; with two
// issuers one thread's waits and commits overlap the other's MMAs.
//
// Pipeline per key tile j (144 keys):
//   TMA warp   : K_j and V_j together into a 3-deep ring (128-byte swizzle); slot
//                j % 3 is reused once P.V of the tile that held it has completed
//   S issuer   : waits for K_j, then (j >= 2) for P.V_{j-2}, which read P_{j-2} from the
//                TMEM buffer S_j overwrites (the two issuers' MMAs are not ordered with
//                each other); S_j = Q K_j^T into TMEM buffer j%2 (M=128, N=144, K=16
//                steps, A = Q from TMEM)
//   P.V issuer : waits for V_j, then for the softmax of tile j (a named barrier that the
//                softmax warps and this warp pass); O += P_j V_j (A = P from TMEM, V an
//                MN-major operand)
//   4 softmax warps (thread = row): load the row's Q into TMEM once; per tile
//                read S_j from TMEM, mask, online softmax with a lazily updated
//                running max (O is rescaled only when the max grows by more than
//                2^8, after P.V_{j-1} is done), write P_j over S_j.  The buffer's
//                previous P (tile j-2) was read by P.V_{j-2} before S_j was issued,
//                so the common path waits for nothing but S_j.
// Lazy rescaling keeps the result exact: every term uses the same reference max
// as the running sum it is divided by.
// Precision: Q.K^T runs on bf16 operands; P.V runs on fp16 operands - the
// softmax weights are rounded to fp16 (2^-11 relative instead of bf16's 2^-8),
// scaled by 2^7 so that they stay in fp16's normal range (p <= 2^15), and the
// V cache holds bf16-precision values in fp16 containers.
#include <float.h>

#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

constexpr int THREADS = 224;                 // producer, S issuer, 4 softmax warps, P.V issuer
constexpr int WARP_PV = 6;
constexpr int KT_ROWS = 144;                 // keys per tile
constexpr int STAGES = 3;                    // K and V ring depth
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t COL_S = 0, S_STRIDE = 160, COL_O = 320, COL_Q = 448;   // S buffers 32-column aligned
// P_j written -> P.V issuer: one named barrier that the 4 softmax warps and the P.V
// issuer's warp all pass with bar.sync once per key tile, in lockstep, on every path
// (also after a failed wait), so each phase completes and no warp can arrive twice in
// one phase.
constexpr uint32_t BAR_P = 1, BAR_P_COUNT = 5 * 32;
constexpr float RESCALE_LOG2 = 8.0f;
constexpr float P_SHIFT_LOG2 = 7.0f;         // P scaled by 2^7: max 2^(8+7) < 65504

template <int D>
struct Smem {
    static constexpr int CHUNK = KT_ROWS * 128;          // KT_ROWS rows x 128 bytes
    static constexpr int KV_BYTES = (D / 64) * CHUNK;    // one K or V tile
    static constexpr int OFF_K = 0;
    static constexpr int OFF_V = OFF_K + STAGES * KV_BYTES;
    static constexpr int OFF_BAR = OFF_V + STAGES * KV_BYTES;
    static constexpr int TOTAL = OFF_BAR + 256 + 1024;
};

template <int D>
__global__ void __launch_bounds__(THREADS, 1)
attn_kernel(const uint16_t* __restrict__ q, const __grid_constant__ CUtensorMap tmK,
            const __grid_constant__ CUtensorMap tmV, const AttnParams p, int num_blocks) {
    using S = Smem<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);
    // Barriers per key tile: kv_full (K_j and V_j landed; waited by both issuers), P_j
    // written (the named barrier BAR_P), s_full (S_j done) and pv_done (P.V_i done) as
    // commits.  P.V_i done frees slot i % STAGES for the producer (P_i was written after
    // S_i had been read), frees S buffer i % 2 for S_{i+2}, and tells a softmax that must
    // rescale O that the accumulation it rescales is complete.  Every waiter on pv_done
    // or kv_full either waits for each phase in turn or cannot be more than one phase
    // behind, so no parity wait meets a barrier two phases away.
    uint64_t* q_ready = bars + 0;                // Q rows stored into TMEM (4 warps)
    uint64_t* kv_full = bars + 1;                // [STAGES]: K_j and V_j in slot j % STAGES
    uint64_t* s_full = kv_full + STAGES;         // [2]: S_j done, phase j/2 of s_full[j % 2]
    uint64_t* pv_done = s_full + 2;              // [STAGES]: P.V_i done, phase i/3 of pv_done[i % 3]
    uint64_t* drain = pv_done + STAGES;          // P.V issuer's MMAs drained
    uint64_t* drain_s = drain + 1;               // S issuer's MMAs drained
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_s + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    int* red = reinterpret_cast<int*>(tmem_slot + 2);   // lo_min, hi_max, hi_min, lo_max

    const uint32_t warp = warp_id(), lane = lane_id();
    const int G = p.Hq / p.Hkv;
    const int RPB = 128 / G;
    // kv head major (the CTAs resident at a time read one or two heads' K/V, which L2 holds),
    // heaviest rows first within a head
    const int blk = num_blocks - 1 - (int)(blockIdx.x % num_blocks);
    const int g = (int)(blockIdx.x / num_blocks);
    const int64_t r0 = (int64_t)blk * RPB;

    if (threadIdx.x == 0) {
        mbar_init(q_ready, 4);
        for (int st = 0; st < STAGES; ++st) {
            mbar_init(&kv_full[st], 1);
            mbar_init(&pv_done[st], 1);
        }
        for (int b = 0; b < 2; ++b) mbar_init(&s_full[b], 1);
        mbar_init(drain, 1);
        mbar_init(drain_s, 1);
        *abort_flag = 0;
        red[0] = INT_MAX; red[1] = -1; red[2] = INT_MAX; red[3] = -1;
        fence_mbar_init();
    }
    if (warp == 1) { tmem_alloc(tmem_slot, TMEM_COLS); tmem_relinquish(); }
    __syncthreads();

    // this thread's row (softmax warps); key range of the whole block
    const uint32_t quarter = warp & 3;
    const int L = (int)(quarter * 32 + lane);
    const int64_t row = r0 + L / G;
    const int head = g * G + L % G;
    const bool valid = warp >= 2 && warp < WARP_PV && L < RPB * G && row < p.m;
    int hi = -1, lo = 0;
    if (valid) {
        hi = p.q_idx[row];
        lo = p.kv_lo ? p.kv_lo[row] : 0;
        atomicMin(&red[0], lo);
        atomicMax(&red[1], hi);
        atomicMin(&red[2], hi);
        atomicMax(&red[3], lo);
    }
    if (warp == 0 && lane == 0) { prefetch_tmap(&tmK); prefetch_tmap(&tmV); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int lo_min = red[0], hi_max = red[1], hi_min = red[2], lo_max = red[3];
    const int t_begin = lo_min / KT_ROWS;
    const int n_tiles = hi_max < 0 ? 0 : hi_max / KT_ROWS + 1 - t_begin;

    uint8_t* sK = smem + S::OFF_K;
    uint8_t* sV = smem + S::OFF_V;

    if (warp == 0) {
        if (lane == 0 && n_tiles > 0) {
            // ------------------------------------------------ TMA producer
            int issued = 0;
            for (int j = 0; j < n_tiles; ++j) {
                const int st = j % STAGES;
                const uint32_t ph = (uint32_t)(j / STAGES) & 1;
                const int y = (t_begin + j) * KT_ROWS;
                // slot st is free once P.V_{j-STAGES} is done (its S had been read before P was written)
                if (!mbar_wait(&pv_done[st], ph ^ 1, abort_flag, p.status)) break;
                mbar_expect_tx(&kv_full[st], 2 * S::KV_BYTES);
#pragma unroll
                for (int c = 0; c < D / 64; ++c) {
                    tma_load_2d(sK + st * S::KV_BYTES + c * S::CHUNK, &tmK, &kv_full[st], g * D + c * 64, y);
                    tma_load_2d(sV + st * S::KV_BYTES + c * S::CHUNK, &tmV, &kv_full[st], g * D + c * 64, y);
                }
                issued = j + 1;
            }
            // on the abort path, let the loads already issued land before exiting
            if (*abort_flag) {
                const uint64_t t0 = globaltimer();
                for (int j = (issued > STAGES ? issued - STAGES : 0); j < issued; ++j)
                    while (!mbar_try_wait(&kv_full[j % STAGES], (uint32_t)(j / STAGES) & 1) &&
                           globaltimer() - t0 < 1000000ull) {}
            }
        }
    } else if (warp == 1) {
        if (n_tiles > 0 && lane == 0) {
            // ------------------------------------------------ S issuer: S_j = Q K_j^T
            constexpr uint32_t IDESC_S = idesc_bf16(128, KT_ROWS, false);
            const uint32_t k0 = smem_u32(sK);
            bool ok = mbar_wait(q_ready, 0, abort_flag, p.status);
            tc_fence_after();
            for (int j = 0; j < n_tiles && ok; ++j) {
                const int b = j & 1, st = j % STAGES;
                // S buffer b last held P_{j-2}: wait until P.V_{j-2} (another thread's MMAs, so
                // not ordered with these) has read it.  Waits on pv_done are contiguous here
                // (tiles 0, 1, 2, ...), so each finds its barrier in the phase it asks for.
                // K_j first (it has almost always landed), so that nothing but the issue follows
                // the wait for P.V_{j-2}
                ok = mbar_wait(&kv_full[st], (uint32_t)(j / STAGES) & 1, abort_flag, p.status);
                if (ok && j >= 2)
                    ok = mbar_wait(&pv_done[(j - 2) % STAGES], (uint32_t)((j - 2) / STAGES) & 1, abort_flag, p.status);
                if (!ok) break;
                tc_fence_after();
                const uint64_t kd = sdesc_sw128(k0 + st * S::KV_BYTES, 16, 1024);
                const uint32_t sd = tmem_base + COL_S + b * S_STRIDE, qa = tmem_base + COL_Q;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    mma_f16_ts(sd, qa + kk * 8, sdesc_add(kd, (kk >> 2) * S::CHUNK + (kk & 3) * 32),
                               IDESC_S, kk > 0 ? 1u : 0u);
                mma_commit(&s_full[b]);
            }
            mma_commit(drain_s);
            const uint64_t t0 = globaltimer();
            while (!mbar_try_wait(drain_s, 0) && globaltimer() - t0 < kWaitLimitNs) {}
        }
        __syncwarp();
    } else if (warp == WARP_PV) {
        if (n_tiles > 0) {
            // ------------------------------------------------ P.V issuer: O += P_j V_j (lane 0; the
            // whole warp passes the named barrier for P)
            constexpr uint32_t IDESC_O = idesc_f16kind(128, D, true, false);   // fp16 P and V
            const uint32_t v0 = smem_u32(sV);
            bool ok = true;
            for (int j = 0; j < n_tiles; ++j) {
                const int st = j % STAGES;
                // V_j landed (waited before the barrier, while the softmax works; the phase
                // cannot move on before this thread commits P.V_j)
                if (lane == 0 && ok) ok = mbar_wait(&kv_full[st], (uint32_t)(j / STAGES) & 1, abort_flag, p.status);
                __syncwarp();
                named_bar_sync(BAR_P, BAR_P_COUNT);
                if (lane == 0 && ok) {
                    tc_fence_after();
                    const uint64_t vd = sdesc_sw128(v0 + st * S::KV_BYTES, S::CHUNK, 1024);
                    const uint32_t od = tmem_base + COL_O, pa = tmem_base + COL_S + (j & 1) * S_STRIDE;
                    mma_f16_ts(od, pa, vd, IDESC_O, j > 0 ? 1u : 0u);
#pragma unroll
                    for (int kk = 1; kk < KT_ROWS / 16; ++kk)
                        mma_f16_ts(od, pa + kk * 8, sdesc_add(vd, kk * 16 * 128), IDESC_O, 1u);
                    mma_commit(&pv_done[st]);
                }
            }
            if (lane == 0) {
                mma_commit(drain);
                const uint64_t t0 = globaltimer();
                while (!mbar_try_wait(drain, 0) && globaltimer() - t0 < kWaitLimitNs) {}
            }
            __syncwarp();
        }
    } else if (n_tiles > 0) {
        // ---------------------------------------------------- softmax warps (2..5)
        const float sl2 = p.scale_log2;
        const uint32_t lane_addr = (quarter * 32u) << 16;
        float m_run = -INFINITY, l_run = 0.f;
        bool ok = true;
        {
            // this row's query into TMEM columns [COL_Q, COL_Q + D/2): bf16 pairs, lane = row
            uint32_t qv[D / 2];
            if (valid) {
                const uint4* src = reinterpret_cast<const uint4*>(q + row * (int64_t)(p.Hq * D) + (int64_t)head * D);
#pragma unroll
                for (int c = 0; c < D / 8; ++c) {
                    const uint4 u = __ldg(src + c);
                    qv[4 * c] = u.x; qv[4 * c + 1] = u.y; qv[4 * c + 2] = u.z; qv[4 * c + 3] = u.w;
                }
            } else {
#pragma unroll
                for (int c = 0; c < D / 2; ++c) qv[c] = 0u;
            }
#pragma unroll
            for (int c = 0; c < D / 64; ++c) tmem_st32(tmem_base + lane_addr + COL_Q + c * 32, qv + c * 32);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(q_ready);
        }
        for (int j = 0; j < n_tiles; ++j) {
            const int b = j & 1;
            // after a failed wait the warp keeps looping without work, so that it still
            // passes every tile's P barrier with the P.V issuer
            if (ok) ok = mbar_wait_warp(&s_full[b], (j >> 1) & 1, abort_flag, p.status);
            if (!ok) {
                named_bar_sync(BAR_P, BAR_P_COUNT);
                continue;
            }
            tc_fence_after();
            uint32_t s[KT_ROWS];
#pragma unroll
            for (int c = 0; c < KT_ROWS / 32; ++c) tmem_ld32(tmem_base + lane_addr + b * S_STRIDE + c * 32, s + c * 32);
            if constexpr (KT_ROWS % 32)
                tmem_ld16(tmem_base + lane_addr + b * S_STRIDE + (KT_ROWS / 32) * 32,
                          *reinterpret_cast<uint32_t(*)[16]>(s + (KT_ROWS / 32) * 32));
            tmem_ld_wait();

            const int key0 = (t_begin + j) * KT_ROWS;
            const bool full_vis = key0 >= lo_max && key0 + KT_ROWS - 1 <= hi_min;
            if (!full_vis) {
#pragma unroll
                for (int c = 0; c < KT_ROWS; ++c) {
                    const int key = key0 + c;
                    if (key > hi || key < lo) s[c] = __float_as_uint(-INFINITY);
                }
            }
            // row max as a tree: 16 independent chains of three-input maxima, not one
            // 144-long dependent chain
            static_assert((KT_ROWS - 16) % 32 == 0, "max tree takes 32 keys per step");
            float mx[16];
#pragma unroll
            for (int c = 0; c < 16; ++c) mx[c] = __uint_as_float(s[c]);
#pragma unroll
            for (int c = 16; c < KT_ROWS; c += 32)
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    mx[e] = fmax3(mx[e], __uint_as_float(s[c + e]), __uint_as_float(s[c + 16 + e]));
#pragma unroll
            for (int w = 8; w > 0; w >>= 1)
#pragma unroll
                for (int c = 0; c < w; ++c) mx[c] = fmaxf(mx[c], mx[c + w]);
            const float mt = mx[0];
            const float m_new = fmaxf(m_run, mt);
            const bool resc = (m_new - m_run) * sl2 > RESCALE_LOG2;   // false when both are -inf
            float alpha = 1.f;
            if (resc) {
                alpha = fast_exp2((m_run - m_new) * sl2);           // 0 when m_run = -inf
                l_run *= alpha;
                m_run = m_new;
            }
            const float mref = ((m_run == -INFINITY) ? 0.f : m_run * sl2) - P_SHIFT_LOG2;
            // exponents and row sums on key pairs: one FFMA2 and one FADD2 per two keys
            uint32_t pk[KT_ROWS / 2];
            const uint64_t sl2x2 = f2_pack(sl2, sl2), nmref2 = f2_pack(-mref, -mref);
            uint64_t ls2[4] = {0ull, 0ull, 0ull, 0ull};   // (even keys, odd keys) partial sums
#pragma unroll
            for (int c = 0; c < KT_ROWS; c += 2) {
                float a0, a1;
                f2_unpack(f2_fma(f2_pack(__uint_as_float(s[c]), __uint_as_float(s[c + 1])), sl2x2, nmref2), a0, a1);
                const float e0 = fast_exp2(a0), e1 = fast_exp2(a1);
                ls2[(c >> 1) & 3] = f2_add(ls2[(c >> 1) & 3], f2_pack(e0, e1));
                pk[c / 2] = pack_f16(e0, e1);
            }
            {
                float l_even, l_odd;
                f2_unpack(f2_add(f2_add(ls2[0], ls2[1]), f2_add(ls2[2], ls2[3])), l_even, l_odd);
                l_run += l_even + l_odd;
            }

            // O is rescaled only once P.V_{j-1} has finished accumulating into it (the wait finds
            // pv_done[(j-1) % 3] in the right phase: S_j was issued after P.V_{j-2} completed, so
            // P.V_{j-4} is complete too); P_j itself goes into S buffer b, whose previous P (of
            // tile j-2) P.V_{j-2} had read before the S issuer wrote S_j
            if (j >= 1 && __any_sync(0xffffffffu, resc)) {
                if (!mbar_wait_warp(&pv_done[(j - 1) % STAGES], (uint32_t)((j - 1) / STAGES) & 1, abort_flag,
                                    p.status)) {
                    ok = false;
                    named_bar_sync(BAR_P, BAR_P_COUNT);
                    continue;
                }
                tc_fence_after();
                {
                    const uint32_t oaddr = tmem_base + lane_addr + COL_O;
#pragma unroll 1
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t o[32];
                        tmem_ld32(oaddr + c * 32, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                        tmem_st32(oaddr + c * 32, o);
                    }
                    tmem_st_wait();
                }
            }
            // P row L (fp16 pairs) over the S_j it was computed from
            tmem_st32(tmem_base + lane_addr + COL_S + b * S_STRIDE, pk);
            tmem_st32(tmem_base + lane_addr + COL_S + b * S_STRIDE + 32, pk + 32);
            static_assert(KT_ROWS == 144, "P store covers 72 columns");
            tmem_st8(tmem_base + lane_addr + COL_S + b * S_STRIDE + 64, pk + 64);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            named_bar_sync(BAR_P, BAR_P_COUNT);
        }
        if (ok && mbar_wait_warp(&pv_done[(n_tiles - 1) % STAGES], (uint32_t)((n_tiles - 1) / STAGES) & 1, abort_flag,
                                 p.status)) {
            tc_fence_after();
            const uint32_t oaddr = tmem_base + lane_addr + COL_O;
            const float inv = (l_run > 0.f) ? 1.f / l_run : 0.f;
            uint16_t* dst = p.out + row * (int64_t)(p.Hq * D) + (int64_t)head * D;
#pragma unroll 1
            for (int c = 0; c < D / 32; ++c) {
                uint32_t o[32];
                tmem_ld32(oaddr + c * 32, o);
                tmem_ld_wait();
                if (valid) {
                    uint4* d4 = reinterpret_cast<uint4*>(dst + c * 32);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        const int e = q4 * 8;
                        d4[q4] = make_uint4(pack_bf16(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv),
                                            pack_bf16(__uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv),
                                            pack_bf16(__uint_as_float(o[e + 4]) * inv, __uint_as_float(o[e + 5]) * inv),
                                            pack_bf16(__uint_as_float(o[e + 6]) * inv, __uint_as_float(o[e + 7]) * inv));
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, TMEM_COLS);
    }
}

template <int D>
kvb_status run(const uint16_t* q, const CUtensorMap& k, const CUtensorMap& v, const AttnParams& p, int nb,
               cudaStream_t st) {
    static std::atomic<uint64_t> smem_set{0};
    auto kern = attn_kernel<D>;
    kvb_status s = ensure_smem_limit((const void*)kern, Smem<D>::TOTAL, smem_set, "attn smem");
    if (s != KVB_OK) return s;
    const int64_t grid = (int64_t)nb * p.Hkv;
    kern<<<(unsigned)grid, THREADS, Smem<D>::TOTAL, st>>>(q, k, v, p, nb);
    count_launch();
    return cuda_ok(cudaGetLastError(), "attention launch");
}

}  // namespace

kvb_status launch_attn(const AttnParams& p, const uint16_t* q, const uint16_t* k_cache, const uint16_t* v_cache,
                       cudaStream_t st) {
    if (p.m <= 0) return KVB_OK;
    if (p.D != 64 && p.D != 128) return fail(KVB_ERR_UNSUPPORTED, "attention: head_dim %d not built", p.D);
    if (p.Hkv <= 0 || p.Hq % p.Hkv || p.Hq / p.Hkv > 128)
        return fail(KVB_ERR_UNSUPPORTED, "attention: Hq must be a multiple of Hkv with Hq/Hkv <= 128");
    const int G = p.Hq / p.Hkv, RPB = 128 / G;
    CUtensorMap tk, tv;
    const uint64_t kvd = (uint64_t)p.Hkv * p.D;
    kvb_status s = make_tmap_2d(&tk, k_cache, kvd, (uint64_t)p.n_kv, kvd, 64, KT_ROWS);
    if (s != KVB_OK) return s;
    s = make_tmap_2d(&tv, v_cache, kvd, (uint64_t)p.n_kv, kvd, 64, KT_ROWS, CU_TENSOR_MAP_DATA_TYPE_FLOAT16);
    if (s != KVB_OK) return s;
    const int64_t nb = (p.m + RPB - 1) / RPB;
    if (nb * p.Hkv > 0x7FFFFFFF) return fail(KVB_ERR_INVALID_ARG, "attention: too many rows");
    return p.D == 128 ? run<128>(q, tk, tv, p, (int)nb, st) : run<64>(q, tk, tv, p, (int)nb, st);
}

}  // namespace kvb
