// Row GEMM on the 5th-generation tensor cores: C = A B^T, bf16 operands, fp32
// accumulation in tensor memory, with the decoder-layer epilogues fused:
//   EPI_QKV    - optional bias, split into q / k / v, RoPE on q and k at each row's position,
//                q to a dense buffer, k / v to (optionally scattered) cache rows;
//   EPI_RESID  - x += C into the fp32 residual stream (O-proj and down-proj);
//   EPI_SWIGLU - the B tile holds 128 gate rows and 128 up rows; writes
//                silu(gate) * up as bf16 (the MLP's inner activation).
//
// Design: persistent CTAs (one per SM), 128 x 256 output tiles, K in steps of 64
// (one 128-byte swizzle atom), a 4-stage TMA ring, one elected thread issuing
// tcgen05.mma (M=128, N=256, K=16), and two 256-column accumulators in TMEM so
// the 4 epilogue warps drain tile i while the tensor core computes tile i+1.
// Warp roles: 0 = TMA producer, 1 = MMA issuer (+ TMEM owner), 2-5 = epilogue.
#include "common.cuh"
#include "internal.h"

namespace kvb {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;              // 16 KB
constexpr int B_BYTES = BN * BK * 2;              // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;    // 48 KB
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256;
constexpr int THREADS = 192;
constexpr int GROUP_M = 32;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t IDESC = idesc_bf16(BM, BN, false);

struct TileMap {
    int num_m, num_n;
    KVB_DEV void coords(int tile, int& tm, int& tn) const {
        const int per_group = GROUP_M * num_n;
        const int g = tile / per_group;
        const int first_m = g * GROUP_M;
        const int gsize = min(GROUP_M, num_m - first_m);
        const int local = tile - g * per_group;
        tm = first_m + local % gsize;
        tn = local / gsize;
    }
};

KVB_DEV void store16_bf16_as_f16(uint16_t* dst, const float* v) {
    uint4 a, b;
    a.x = pack_bf16_as_f16(v[0], v[1]);   a.y = pack_bf16_as_f16(v[2], v[3]);
    a.z = pack_bf16_as_f16(v[4], v[5]);   a.w = pack_bf16_as_f16(v[6], v[7]);
    b.x = pack_bf16_as_f16(v[8], v[9]);   b.y = pack_bf16_as_f16(v[10], v[11]);
    b.z = pack_bf16_as_f16(v[12], v[13]); b.w = pack_bf16_as_f16(v[14], v[15]);
    reinterpret_cast<uint4*>(dst)[0] = a;
    reinterpret_cast<uint4*>(dst)[1] = b;
}

KVB_DEV void store16_bf16(uint16_t* dst, const float* v) {
    uint4 a, b;
    a.x = pack_bf16(v[0], v[1]);   a.y = pack_bf16(v[2], v[3]);
    a.z = pack_bf16(v[4], v[5]);   a.w = pack_bf16(v[6], v[7]);
    b.x = pack_bf16(v[8], v[9]);   b.y = pack_bf16(v[10], v[11]);
    b.z = pack_bf16(v[12], v[13]); b.w = pack_bf16(v[14], v[15]);
    reinterpret_cast<uint4*>(dst)[0] = a;
    reinterpret_cast<uint4*>(dst)[1] = b;
}

// x[i] += b[i] for 16 fp32 accumulator words; b is 16-byte aligned
KVB_DEV void add_bias16(uint32_t* x, const float* b) {
    const float4* b4 = reinterpret_cast<const float4*>(b);
#pragma unroll
    for (int v = 0; v < 4; ++v) {
        const float4 t = __ldg(b4 + v);
        x[4 * v] = __float_as_uint(__uint_as_float(x[4 * v]) + t.x);
        x[4 * v + 1] = __float_as_uint(__uint_as_float(x[4 * v + 1]) + t.y);
        x[4 * v + 2] = __float_as_uint(__uint_as_float(x[4 * v + 2]) + t.z);
        x[4 * v + 3] = __float_as_uint(__uint_as_float(x[4 * v + 3]) + t.w);
    }
}

template <int EPI, int HD>
__global__ void __launch_bounds__(THREADS, 1)
gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
            const __grid_constant__ CUtensorMap tmB2, const GemmParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;   // [2] accumulator ready
    uint64_t* tempty = tfull + 2;       // [2] accumulator drained
    uint64_t* drain = tempty + 2;       // MMA completion at exit
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const uint32_t warp = warp_id(), lane = lane_id();
    const int out_cols = (EPI == EPI_SWIGLU) ? BN / 2 : BN;
    const TileMap tmap{(int)((p.M + BM - 1) / BM), (int)((p.N + out_cols - 1) / out_cols)};
    const int num_tiles = tmap.num_m * tmap.num_n;
    const int KB = (int)((p.K + BK - 1) / BK);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
        for (int a = 0; a < 2; ++a) { mbar_init(&tfull[a], 1); mbar_init(&tempty[a], 4); }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tmA); prefetch_tmap(&tmB); prefetch_tmap(&tmB2);
    }
    if (warp == 1) { tmem_alloc(tmem_slot, TMEM_COLS); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------ TMA producer
            int stage = 0; uint32_t phase = 0; bool ok = true;
            int issued_parity[STAGES];
#pragma unroll
            for (int s = 0; s < STAGES; ++s) issued_parity[s] = -1;
            for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x) {
                int tm, tn; tmap.coords(tile, tm, tn);
                const int m0 = tm * BM;
                for (int kb = 0; kb < KB; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.status)) { ok = false; break; }
                    uint8_t* sa = smem + stage * STAGE_BYTES;
                    uint8_t* sb = sa + A_BYTES;
                    mbar_expect_tx(&full[stage], STAGE_BYTES);
                    tma_load_2d(sa, &tmA, &full[stage], kb * BK, m0);
                    if (EPI == EPI_SWIGLU) {
                        tma_load_2d(sb, &tmB, &full[stage], kb * BK, tn * (BN / 2));
                        tma_load_2d(sb + B_BYTES / 2, &tmB2, &full[stage], kb * BK, tn * (BN / 2));
                    } else {
                        tma_load_2d(sb, &tmB, &full[stage], kb * BK, tn * BN);
                        tma_load_2d(sb + B_BYTES / 2, &tmB, &full[stage], kb * BK, tn * BN + BN / 2);
                    }
                    issued_parity[stage] = (int)phase;
                    if (++stage == STAGES) { stage = 0; phase ^= 1; }
                }
            }
            // on the abort path, let the loads already issued land before the CTA exits
            if (!ok) {
                const uint64_t t0 = globaltimer();
                for (int s = 0; s < STAGES; ++s)
                    if (issued_parity[s] >= 0)
                        while (!mbar_try_wait(&full[s], (uint32_t)issued_parity[s]) &&
                               globaltimer() - t0 < 1000000ull) {}
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------ MMA issuer
            int stage = 0; uint32_t phase = 0; int acc = 0; uint32_t acc_phase = 0; bool ok = true;
            for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x) {
                if (!mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag, p.status)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d = tmem_base + (uint32_t)(acc * BN);
                for (int kb = 0; kb < KB; ++kb) {
                    if (!mbar_wait(&full[stage], phase, abort_flag, p.status)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(smem + stage * STAGE_BYTES);
                    // descriptors built once per stage; each K step of 16 advances 32 bytes
                    const uint64_t ad = sdesc_sw128(a0, 16, 1024), bd = sdesc_sw128(a0 + A_BYTES, 16, 1024);
                    mma_bf16_ss(d, ad, bd, IDESC, kb != 0);
#pragma unroll
                    for (int k = 1; k < BK / 16; ++k)
                        mma_bf16_ss(d, sdesc_add(ad, k * 32), sdesc_add(bd, k * 32), IDESC, 1u);
                    mma_commit(&empty[stage]);
                    if (++stage == STAGES) { stage = 0; phase ^= 1; }
                }
                if (!ok) break;
                mma_commit(&tfull[acc]);
                if (++acc == 2) { acc = 0; acc_phase ^= 1; }
            }
            // wait for every MMA this thread issued before TMEM is released
            mma_commit(drain);
            const uint64_t t0 = globaltimer();
            while (!mbar_try_wait(drain, 0) && globaltimer() - t0 < kWaitLimitNs) {}
        }
    } else {
        // ---------------------------------------------------- epilogue (warps 2..5)
        const uint32_t quarter = warp & 3;
        const int row_in_tile = (int)(quarter * 32 + lane);
        int acc = 0; uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
            int tm, tn; tmap.coords(tile, tm, tn);
            if (!mbar_wait_warp(&tfull[acc], acc_phase, abort_flag, p.status)) break;
            tc_fence_after();
            const int64_t row = (int64_t)tm * BM + row_in_tile;
            const bool valid = row < p.M;
            const uint32_t taddr = tmem_base + ((quarter * 32u) << 16) + (uint32_t)(acc * BN);

            if constexpr (EPI == EPI_QKV) {
                constexpr int NH = BN / HD;
                // indices the caller supplies are checked where they are used: a position outside the
                // RoPE tables is rotated by position 0, a destination outside the k / v buffers writes
                // nothing; both are reported
                int64_t pos = valid ? (int64_t)p.rope_pos[row] : 0;
                if (pos < 0 || pos >= p.max_pos) {
                    set_status(p.status, KVB_ERR_INVALID_ARG);
                    pos = 0;
                }
                const float* crow = p.cos_t + pos * (HD / 2);
                const float* srow = p.sin_t + pos * (HD / 2);
                const int64_t dst = valid ? (p.kv_dst ? (int64_t)p.kv_dst[row] : row) : 0;
                const bool dst_ok = dst >= 0 && dst < p.n_kv_rows;
#pragma unroll 1
                for (int hh = 0; hh < NH; ++hh) {
                    const int c0 = tn * BN + hh * HD;          // column within this GEMM
                    if (c0 >= p.N) break;
                    const int colL = p.col_base + c0;          // column within [q | k | v]
                    uint16_t* outp;
                    uint16_t* outp2 = nullptr;   // bf16 copy of v (chunk-cache format)
                    bool rope = true, write = valid;
                    if (colL < p.q_dim) {
                        outp = p.q_out + row * p.q_dim + colL;
                    } else if (colL < p.q_dim + p.kv_dim) {
                        outp = p.k_out + dst * p.kv_dim + (colL - p.q_dim);
                        write = valid && dst_ok;
                    } else {
                        outp = p.v_out + dst * p.kv_dim + (colL - p.q_dim - p.kv_dim);
                        if (p.v_out_bf16) outp2 = p.v_out_bf16 + dst * p.kv_dim + (colL - p.q_dim - p.kv_dim);
                        rope = false;
                        write = valid && dst_ok;
                    }
                    if (valid && !dst_ok && colL >= p.q_dim) set_status(p.status, KVB_ERR_INVALID_ARG);
                    const uint32_t tcol = taddr + (uint32_t)(hh * HD);
                    if (rope) {
#pragma unroll 1
                        for (int c = 0; c < HD / 32; ++c) {
                            uint32_t x1[16], x2[16];
                            tmem_ld16(tcol + c * 16, x1);
                            tmem_ld16(tcol + HD / 2 + c * 16, x2);
                            tmem_ld_wait();
                            if (write) {
                                if (p.bias) {
                                    add_bias16(x1, p.bias + colL + c * 16);
                                    add_bias16(x2, p.bias + colL + HD / 2 + c * 16);
                                }
                                float y1[16], y2[16];
                                const float4* cp = reinterpret_cast<const float4*>(crow + c * 16);
                                const float4* sp = reinterpret_cast<const float4*>(srow + c * 16);
#pragma unroll
                                for (int v4 = 0; v4 < 4; ++v4) {
                                    const float4 cc = __ldg(cp + v4), ss = __ldg(sp + v4);
                                    const float cs[4] = {cc.x, cc.y, cc.z, cc.w};
                                    const float sn[4] = {ss.x, ss.y, ss.z, ss.w};
#pragma unroll
                                    for (int e = 0; e < 4; ++e) {
                                        const int i = v4 * 4 + e;
                                        const float a = __uint_as_float(x1[i]), b = __uint_as_float(x2[i]);
                                        y1[i] = a * cs[e] - b * sn[e];
                                        y2[i] = b * cs[e] + a * sn[e];
                                    }
                                }
                                store16_bf16(outp + c * 16, y1);
                                store16_bf16(outp + HD / 2 + c * 16, y2);
                            }
                        }
                    } else {
#pragma unroll 1
                        for (int c = 0; c < HD / 16; ++c) {
                            uint32_t x1[16];
                            tmem_ld16(tcol + c * 16, x1);
                            tmem_ld_wait();
                            if (write) {
                                if (p.bias) add_bias16(x1, p.bias + colL + c * 16);
                                float y[16];
#pragma unroll
                                for (int i = 0; i < 16; ++i) y[i] = __uint_as_float(x1[i]);
                                store16_bf16_as_f16(outp + c * 16, y);
                                if (outp2) store16_bf16(outp2 + c * 16, y);
                            }
                        }
                    }
                }
            } else if constexpr (EPI == EPI_RESID) {
#pragma unroll 1
                for (int c = 0; c < BN / 16; ++c) {
                    const int64_t col = (int64_t)tn * BN + c * 16;
                    if (col >= p.N) break;
                    uint32_t v[16];
                    tmem_ld16(taddr + c * 16, v);
                    tmem_ld_wait();
                    if (valid) {
                        float4* xp = reinterpret_cast<float4*>(p.x + row * p.ldx + col);
#pragma unroll
                        for (int v4 = 0; v4 < 4; ++v4) {
                            float4 o = xp[v4];
                            o.x += __uint_as_float(v[v4 * 4 + 0]);
                            o.y += __uint_as_float(v[v4 * 4 + 1]);
                            o.z += __uint_as_float(v[v4 * 4 + 2]);
                            o.w += __uint_as_float(v[v4 * 4 + 3]);
                            xp[v4] = o;
                        }
                    }
                }
            } else {  // EPI_SWIGLU
#pragma unroll 1
                for (int c = 0; c < (BN / 2) / 16; ++c) {
                    const int64_t col = (int64_t)tn * (BN / 2) + c * 16;
                    if (col >= p.N) break;
                    uint32_t g[16], u[16];
                    tmem_ld16(taddr + c * 16, g);
                    tmem_ld16(taddr + BN / 2 + c * 16, u);
                    tmem_ld_wait();
                    if (valid) {
                        float y[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const float gv = __uint_as_float(g[i]);
                            y[i] = gv / (1.0f + __expf(-gv)) * __uint_as_float(u[i]);
                        }
                        store16_bf16(p.out + row * p.ldo + col, y);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1; }
        }
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, TMEM_COLS);
    }
}

template <int EPI, int HD>
kvb_status run(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& b2, const GemmParams& p, int tiles,
               cudaStream_t st) {
    static std::atomic<uint64_t> smem_set{0};
    auto kern = gemm_kernel<EPI, HD>;
    kvb_status s = ensure_smem_limit((const void*)kern, SMEM_BYTES, smem_set, "gemm smem attribute");
    if (s != KVB_OK) return s;
    const int grid = tiles < num_sms() ? tiles : num_sms();
    kern<<<grid, THREADS, SMEM_BYTES, st>>>(a, b, b2, p);
    count_launch();
    return cuda_ok(cudaGetLastError(), "gemm launch");
}

}  // namespace

kvb_status launch_gemm(const GemmParams& p, const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                       const uint16_t* B2, cudaStream_t st) {
    if (p.M <= 0 || p.N <= 0) return KVB_OK;
    if (p.K <= 0 || p.K % 8 || lda % 8 || ldb % 8 || !aligned16(A) || !aligned16(B))
        return fail(KVB_ERR_INVALID_ARG, "gemm: K, lda, ldb must be multiples of 8 and A, B 16-byte aligned");
    CUtensorMap ta, tb, tb2;
    kvb_status s = make_tmap_2d(&ta, A, p.K, p.M, lda, BK, BM);
    if (s != KVB_OK) return s;
    s = make_tmap_2d(&tb, B, p.K, p.N, ldb, BK, BN / 2);
    if (s != KVB_OK) return s;
    if (p.epi == EPI_SWIGLU) {
        if (!B2 || !aligned16(B2)) return fail(KVB_ERR_INVALID_ARG, "gemm: SwiGLU needs an aligned up matrix");
        s = make_tmap_2d(&tb2, B2, p.K, p.N, ldb, BK, BN / 2);
        if (s != KVB_OK) return s;
    } else {
        tb2 = tb;
    }
    const int out_cols = p.epi == EPI_SWIGLU ? BN / 2 : BN;
    const int tiles = (int)(((p.M + BM - 1) / BM) * ((p.N + out_cols - 1) / out_cols));
    switch (p.epi) {
        case EPI_QKV:
            if (p.head_dim == 128) return run<EPI_QKV, 128>(ta, tb, tb2, p, tiles, st);
            if (p.head_dim == 64) return run<EPI_QKV, 64>(ta, tb, tb2, p, tiles, st);
            return fail(KVB_ERR_UNSUPPORTED, "gemm: head_dim %d not built (64 or 128)", p.head_dim);
        case EPI_RESID:
            if (p.N % 16) return fail(KVB_ERR_INVALID_ARG, "gemm: residual width must be a multiple of 16");
            return run<EPI_RESID, 0>(ta, tb, tb2, p, tiles, st);
        case EPI_SWIGLU:
            if (p.N % 16) return fail(KVB_ERR_INVALID_ARG, "gemm: MLP width must be a multiple of 16");
            return run<EPI_SWIGLU, 0>(ta, tb, tb2, p, tiles, st);
        default:
            return fail(KVB_ERR_INVALID_ARG, "gemm: unknown epilogue %d", p.epi);
    }
}

}  // namespace kvb
