// bf16 GEMMs of the CLEAR-MoE FFN on the 5th-generation tensor cores (tcgen05, sm_103a).
//
//   C[m, n] = epilogue( sum_k A[m, k] B[n, k] ),  A and B K-major bf16, fp32 accumulate in TMEM.
//
// One persistent, warp-specialised kernel per (N tile width, operand mode):
//   warps 0-7  epilogue: tcgen05.ld of the accumulator (warp w reads TMEM lane quarter w % 4 and
//              column half w / 4), bias+GELU / column scale / plain, round to bf16, stage through
//              shared memory, coalesced 16-byte stores; rows may be scattered (out[perm[slot]],
//              Algorithm 3 step 6);
//   warp 8     TMEM allocation and the single thread that issues tcgen05.mma (M=128, N=BN,
//              K=16 per instruction) and tcgen05.commit;
//   warp 9     TMA producer (dense / grouped modes): 128-byte-swizzled A and B tiles;
//   warps 10-13 gather producers (gather mode): the A rows of fc1 are tokens picked by the routing
//              permutation, so they are copied row by row with 16-byte cp.async straight into the
//              swizzled layout (chunk j of row r at r*128 + (j ^ (r & 7))*16), while B comes by TMA.
// Stages of a shared-memory ring are handed over by mbarriers (full: TMA bytes / cp.async
// arrivals; empty: tcgen05.commit). Two TMEM accumulators let the epilogue of one tile overlap the
// MMAs of the next. The grouped mode walks tiles (expert, m-tile, n-tile) from the device-resident
// expert offsets and chains two K segments into one accumulator: [t | z] x [U_r | W_e^res].
// Every wait is bounded; on time-out the CTA records CLEARMOE_ETIMEOUT, drains its in-flight
// copies and MMAs, frees TMEM and returns.
//
// The fp32 variant (TF32 = true, dense and grouped modes) runs fp32 operands on the TF32 tensor
// cores (kind::tf32, K = 8 per instruction, the same 128-byte rows and descriptors as bf16): a TMA
// box of 32 fp32 per row lands where 64 bf16 would, then warps 10-13 split every value v of the
// stage into h = v rounded to TF32 (written back in place) and its exact remainder l = v - h
// (written to a second half of the stage at the same offset), and each K step issues three MMAs,
// h_A h_B + h_A l_B + l_A h_B, into the fp32 accumulator. The dropped l_A l_B and the TF32 rounding of
// the remainders leave a relative error near 2^-21 per product, so fp32 layers keep their accuracy
// on the tensor cores (one TF32 product alone would be off by up to 2^-11).
#include <cstdint>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace cm {

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;
constexpr int TC_NUM_EPI = 8;  // two warps per TMEM lane quarter, each on half the columns
constexpr int TC_WARP_MMA = 8;
constexpr int TC_WARP_TMA = 9;
constexpr int TC_WARP_GATHER = 10;
constexpr int TC_GATHER_THREADS = 128;
constexpr int TC_THREADS_TMA = 32 * (TC_WARP_TMA + 1);
constexpr int TC_THREADS_GATHER = 32 * TC_WARP_GATHER + TC_GATHER_THREADS;

// K elements per stage: 64 bf16 or 32 fp32, a 128-byte row either way
template <bool TF32>
constexpr int tc_kelems() {
    return TF32 ? TC_BK / 2 : TC_BK;
}

template <int BN, bool TF32 = false>
struct TcCfg {
    static constexpr int A_BYTES = TC_BM * TC_BK * 2;
    static constexpr int B_BYTES = BN * TC_BK * 2;
    // fp32: the stage's second half holds the remainders of its first, at the same offsets
    static constexpr int HALF_BYTES = A_BYTES + B_BYTES;
    static constexpr int STAGE_BYTES = TF32 ? 2 * HALF_BYTES : HALF_BYTES;
    static constexpr int STAGES_RAW = (196 * 1024) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_RAW > 8 ? 8 : STAGES_RAW;
    static constexpr int HALF = BN / 2;               // columns per epilogue warp
    static constexpr int CW = HALF < 32 ? HALF : 32;  // epilogue columns per TMEM load
    static constexpr int STG_ROW = CW * 2 + 16;       // staging row pitch (bytes)
    static constexpr int STG_BYTES = TC_NUM_EPI * 32 * STG_ROW;
    static constexpr int TMEM_COLS = (2 * BN <= 32) ? 32 : (2 * BN <= 64) ? 64 : (2 * BN <= 128) ? 128
                                     : (2 * BN <= 256) ? 256 : 512;
    // + (fp32) the split stages' barriers and the two of the K-split handshake
    static constexpr int NBARS = 2 * STAGES + 5 + (TF32 ? STAGES + 2 : 0);
    // fp32 fc1 with the slots formed in its epilogue: the routing's prefix table [range][expert]
    // and the expert offsets
    static constexpr int TAB_BYTES = TF32 ? (TC2_TAB_CAP + CM_MAX_E) * 4 : 0;
    static constexpr int SMEM = 1024 + STAGES * STAGE_BYTES + STG_BYTES + TAB_BYTES + NBARS * 8 + 16 + 4 * 20;
};

struct TileInfo {
    int64_t m0;
    int rows;
    int n0;
    int e;
};

__device__ __forceinline__ TileInfo decode_tile(const TcGemmArgs& a, int tile, int n_tiles,
                                                const int* s_prefix, int BN) {
    TileInfo t;
    const int mt = tile / n_tiles;
    t.n0 = (tile % n_tiles) * BN;
    if (a.mode == TC_GROUPED) {
        int e = 0;
        while (e + 1 < a.E && s_prefix[e + 1] <= mt) ++e;
        const int64_t lo = tc_group_off(a, e), hi = tc_group_off(a, e + 1);
        t.m0 = lo + (int64_t)(mt - s_prefix[e]) * TC_BM;
        t.rows = (int)min((int64_t)TC_BM, hi - t.m0);
        t.e = e;
    } else {
        t.m0 = (int64_t)mt * TC_BM;
        t.rows = (int)min((int64_t)TC_BM, a.M - t.m0);
        t.e = 0;
    }
    return t;
}

__device__ __forceinline__ float tf32_rna(float x) {  // x rounded to TF32 (low 13 bits zero)
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}

__device__ __forceinline__ void umma_tf32(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Instruction descriptor: fp32 accumulator, A and B TF32 (format 2), both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_tf32_f32(int M, int N) {
    return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

template <int BN, int MODE, bool TF32>
__global__ void __launch_bounds__((MODE == TC_GATHER || TF32) ? TC_THREADS_GATHER : TC_THREADS_TMA, 1)
    tc_gemm_kernel(const __grid_constant__ TcGemmArgs a) {
    if (!a.pdl_trigger_late) pdl_launch_dependents();
    using C = TcCfg<BN, TF32>;
    constexpr int KE = tc_kelems<TF32>();
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    unsigned char* sm = smem_raw + ((1024 - (raw_addr & 1023)) & 1023);
    unsigned char* stg = sm + C::STAGES * C::STAGE_BYTES;
    int* s_tab = reinterpret_cast<int*>(stg + C::STG_BYTES);  // fp32 fused slots: [range][expert]
    int* s_off = s_tab + TC2_TAB_CAP;                            // [expert] offsets
    uint64_t* bars = reinterpret_cast<uint64_t*>(stg + C::STG_BYTES + C::TAB_BYTES);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NBARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    int* s_prefix = reinterpret_cast<int*>(tmem_slot + 4);  // [CM_MAX_E + 1]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (C::STAGES + s); };
    auto tfull_bar = [&](int i) { return bar0 + 8u * (2 * C::STAGES + i); };
    auto tempty_bar = [&](int i) { return bar0 + 8u * (2 * C::STAGES + 2 + i); };
    const uint32_t drain_bar = bar0 + 8u * (2 * C::STAGES + 4);
    auto split_bar = [&](int s) { return bar0 + 8u * (2 * C::STAGES + 5 + s); };  // fp32: stage split
    const uint32_t kjoin_bar = bar0 + 8u * (3 * C::STAGES + 5);  // fp32 K split: the epilogue warps' partials
    const uint32_t kdone_bar = bar0 + 8u * (3 * C::STAGES + 6);  // fp32 K split: the tile's last unit known
    // fp32 K split: units (tile, K range) instead of tiles
    const int ksp = TF32 ? (a.ksplit > 1 ? a.ksplit : 1) : 1;
    const uint64_t lim = (uint64_t)a.wait_limit_ns;

    const int n_tiles = a.N / BN;
    const int nk0 = (a.K0 + KE - 1) / KE;
    const int nk1 = MODE == TC_GROUPED ? (a.K1 + KE - 1) / KE : 0;
    const int nkb = nk0 + nk1;
    // K blocks [lo, hi) of a unit: the tile's blocks [kb0, nkb) (kb0 = nk0 for the class tokens' group)
    // cut into ksp equal ranges, range sp of them
    auto k_range = [&](const TileInfo& t, int sp, int& lo, int& hi) {
        const int kb0 = (MODE == TC_GROUPED && a.dense_last && t.e == a.E - 1) ? nk0 : 0;
        lo = kb0 + (nkb - kb0) * sp / ksp;
        hi = kb0 + (nkb - kb0) * (sp + 1) / ksp;
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(full_bar(s), MODE == TC_GATHER ? TC_GATHER_THREADS + 1 : 1);
            mbar_init(empty_bar(s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(tfull_bar(i), 1);
            mbar_init(tempty_bar(i), TC_NUM_EPI);
        }
        mbar_init(drain_bar, 1);
        if (TF32) {
            for (int s = 0; s < C::STAGES; ++s) mbar_init(split_bar(s), TC_GATHER_THREADS / 32);  // one per warp
            mbar_init(kjoin_bar, TC_NUM_EPI);
            mbar_init(kdone_bar, 1);
        }
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == TC_WARP_MMA) tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // everything above overlaps the predecessor kernel; from here on its results are read
    pdl_wait();
    if (a.pdl_trigger_late) pdl_launch_dependents();
    if (TF32 && MODE == TC_DENSE && a.rt_info && warp < TC_NUM_EPI) {
        // fp32 fc1 storing each token's row at its routing slot (as the 2-SM fc1 does): the
        // routing's prefix table, by the epilogue warps while the producer and MMA warps start.
        // Thread c holds range c's counts; per expert an exclusive scan over ranges (warp scans, warp
        // totals in s_off's tail, named barrier 1 among the epilogue warps).
        int* s_wt = s_tab + TC2_TAB_CAP - TC_NUM_EPI * CM_MAX_E;  // scratch below the table's end
        const int c = threadIdx.x;
        const int E = a.rt_E;
        int cnt[CM_MAX_E], incl[CM_MAX_E];
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) cnt[e] = (c < a.rt_ctas && e < E) ? __ldcg(a.rt_counts + (size_t)c * CM_MAX_E + e) : 0;
        int wt[CM_MAX_E];
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) {
            incl[e] = cnt[e];
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl[e], off);
                if (lane >= off) incl[e] += v;
            }
            wt[e] = __shfl_sync(0xffffffffu, incl[e], 31);
        }
        // the warp totals go to the table's last entries, read back before the table is written
        asm volatile("bar.sync 1, %0;" ::"n"(TC_NUM_EPI * 32) : "memory");
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e)
            if (lane == 0 && e < E) s_wt[warp * CM_MAX_E + e] = wt[e];
        asm volatile("bar.sync 1, %0;" ::"n"(TC_NUM_EPI * 32) : "memory");
        int before[CM_MAX_E], tot[CM_MAX_E];
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) {
            before[e] = incl[e] - cnt[e];
            tot[e] = 0;
            if (e < E)
                for (int w = 0; w < TC_NUM_EPI; ++w) {
                    const int v = s_wt[w * CM_MAX_E + e];
                    if (w < warp) before[e] += v;
                    tot[e] += v;
                }
        }
        asm volatile("bar.sync 1, %0;" ::"n"(TC_NUM_EPI * 32) : "memory");  // scratch read before the table is written
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e)
            if (e < E && c < a.rt_ctas) s_tab[c * E + e] = before[e];
        if (warp == 0) {  // lane e: expert offsets by a scan over experts
            int te = 0;
#pragma unroll
            for (int e = 0; e < CM_MAX_E; ++e)
                if (e == lane) te = tot[e];
            int sc = lane < E ? te : 0;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, sc, off);
                if (lane >= off) sc += v;
            }
            if (lane < E) {
                s_off[lane] = sc - te;
                if (blockIdx.x == 0) {
                    a.rt_out_counts[lane] = te;
                    a.rt_out_offsets[lane] = sc - te;
                    if (lane == E - 1) {
                        a.rt_out_offsets[E] = sc;
                        const int64_t n_cls = n_class_tokens(a.M, a.rt_cls_stride);
                        if (n_cls > 0) {  // the class tokens' group (the dense path)
                            a.rt_out_counts[E] = (int32_t)n_cls;
                            a.rt_out_offsets[E + 1] = sc + (int32_t)n_cls;
                        }
                    }
                }
            }
        }
        asm volatile("bar.sync 1, %0;" ::"n"(TC_NUM_EPI * 32) : "memory");
    }
    if (MODE == TC_GROUPED) {
        if (threadIdx.x == 0) {
            int acc = 0;
            for (int e = 0; e < a.E; ++e) {
                s_prefix[e] = acc;
                acc += (int)((tc_group_off(a, e + 1) - tc_group_off(a, e) + TC_BM - 1) / TC_BM);
            }
            s_prefix[a.E] = acc;
        }
        __syncthreads();
    }
    const uint32_t tmem_base = *tmem_slot;

    int m_tiles;
    if (MODE == TC_GROUPED)
        m_tiles = s_prefix[a.E];
    else
        m_tiles = (int)((a.M + TC_BM - 1) / TC_BM);
    const int num_tiles = m_tiles * n_tiles;

    if (MODE != TC_GATHER && warp == TC_WARP_TMA) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t ph = 0;
            uint32_t issued = 0;  // bit s: stage s has a load in flight or done
            uint32_t par = 0;     // bit s: parity of stage s's last load
            bool ok = true;
            for (int unit = blockIdx.x; unit < num_tiles * ksp && ok; unit += gridDim.x) {
                const TileInfo t = decode_tile(a, unit / ksp, n_tiles, s_prefix, BN);
                int klo, khi;  // the dense path's group (class tokens): the z x W2 segment alone
                k_range(t, unit % ksp, klo, khi);
                for (int kb = klo; kb < khi; ++kb) {
                    if (!mbar_wait(empty_bar(stage), ph ^ 1, abort_flag, a.status, lim)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sA = smem_u32(sm + stage * C::STAGE_BYTES);
                    const uint32_t sB = sA + C::A_BYTES;
                    mbar_arrive_expect_tx(full_bar(stage), C::HALF_BYTES);
                    if (kb < nk0) {
                        tma_load_2d(sA, &a.tmA0, kb * KE, (int)t.m0, full_bar(stage));
                        tma_load_2d(sB, &a.tmB0, kb * KE, t.n0, full_bar(stage));
                    } else {
                        const int kk = (kb - nk0) * KE;
                        tma_load_2d(sA, &a.tmA1, kk, (int)t.m0, full_bar(stage));
                        tma_load_2d(sB, &a.tmB1[t.e], kk, t.n0, full_bar(stage));
                    }
                    issued |= 1u << stage;
                    par = (par & ~(1u << stage)) | (ph << stage);
                    if (++stage == C::STAGES) {
                        stage = 0;
                        ph ^= 1;
                    }
                }
            }
            if (!ok) {  // let every copy in flight land before the CTA retires
                for (int s = 0; s < C::STAGES; ++s)
                    if (issued & (1u << s)) mbar_wait(full_bar(s), (par >> s) & 1, nullptr, a.status, 10000000ull);
            }
        }
    } else if (TF32 && warp >= TC_WARP_GATHER) {
        // ------------------------------------------------ fp32: split each landed stage
        // v -> h = TF32(v) in place, l = v - h (exact) in the stage's second half; the writes are
        // made visible to the tensor cores' (async) proxy before the warp's arrival.
        const int ct = threadIdx.x - TC_WARP_GATHER * 32;
        int stage = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int unit = blockIdx.x; unit < num_tiles * ksp && ok; unit += gridDim.x) {
            const TileInfo t = decode_tile(a, unit / ksp, n_tiles, s_prefix, BN);
            int klo, khi;
            k_range(t, unit % ksp, klo, khi);
            for (int kb = klo; kb < khi; ++kb) {
                if (!mbar_wait(full_bar(stage), ph, abort_flag, a.status, lim)) {
                    ok = false;
                    break;
                }
                float4* hi = reinterpret_cast<float4*>(sm + stage * C::STAGE_BYTES);
                float4* lo = reinterpret_cast<float4*>(sm + stage * C::STAGE_BYTES + C::HALF_BYTES);
#pragma unroll 4
                for (int i = ct; i < C::HALF_BYTES / 16; i += TC_GATHER_THREADS) {
                    const float4 v = hi[i];
                    const float4 h = make_float4(tf32_rna(v.x), tf32_rna(v.y), tf32_rna(v.z), tf32_rna(v.w));
                    hi[i] = h;
                    lo[i] = make_float4(v.x - h.x, v.y - h.y, v.z - h.z, v.w - h.w);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(split_bar(stage));
                if (++stage == C::STAGES) {
                    stage = 0;
                    ph ^= 1;
                }
            }
        }
    } else if (MODE == TC_GATHER && warp >= TC_WARP_GATHER) {
        // ------------------------------------------------ gather producers (fc1 in expert order)
        const int pt = threadIdx.x - TC_WARP_GATHER * 32;
        const int cch = pt & 7;   // 16-byte chunk of the 128-byte row segment
        const int rsub = pt >> 3; // rows rsub + 16 i
        const uint16_t* X = static_cast<const uint16_t*>(a.gather_src);
        int stage = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
            const TileInfo t = decode_tile(a, tile, n_tiles, s_prefix, BN);
            int64_t src[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int r = rsub + 16 * i;
                src[i] = (r < t.rows) ? (int64_t)a.rows[t.m0 + r] : -1;
                if ((uint64_t)src[i] >= (uint64_t)a.M) src[i] = -1;  // only a launch that gave up leaves such rows
            }
            for (int kb = 0; kb < nkb; ++kb) {
                if (!mbar_wait(empty_bar(stage), ph ^ 1, abort_flag, a.status, lim)) {
                    ok = false;
                    break;
                }
                const uint32_t sA = smem_u32(sm + stage * C::STAGE_BYTES);
                const uint32_t sB = sA + C::A_BYTES;
                if (pt == 0) {
                    mbar_arrive_expect_tx(full_bar(stage), C::B_BYTES);
                    tma_load_2d(sB, &a.tmB0, kb * TC_BK, t.n0, full_bar(stage));
                }
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int r = rsub + 16 * i;
                    if (src[i] >= 0)
                        cp_async_16(sA + r * 128 + ((cch ^ (r & 7)) << 4),
                                    X + src[i] * a.gather_ld + kb * TC_BK + cch * 8);
                }
                asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(full_bar(stage))
                             : "memory");
                if (++stage == C::STAGES) {
                    stage = 0;
                    ph ^= 1;
                }
            }
        }
        cp_async_wait<0>();
    } else if (warp == TC_WARP_MMA) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = TF32 ? idesc_tf32_f32(TC_BM, BN) : idesc_bf16_f32(TC_BM, BN);
            int stage = 0;
            uint32_t ph = 0;
            int acc = 0;
            uint32_t aph = 0;
            bool ok = true;
            for (int unit = blockIdx.x; unit < num_tiles * ksp && ok; unit += gridDim.x) {
                if (!mbar_wait(tempty_bar(acc), aph ^ 1, abort_flag, a.status, lim)) break;
                tc_fence_after();
                const uint32_t dtm = tmem_base + acc * BN;
                int kb0, khi;
                k_range(decode_tile(a, unit / ksp, n_tiles, s_prefix, BN), unit % ksp, kb0, khi);
                for (int kb = kb0; kb < khi; ++kb) {
                    // fp32: the stage once split (its bytes landed before the split warps read them)
                    if (!mbar_wait(TF32 ? split_bar(stage) : full_bar(stage), ph, abort_flag, a.status, lim)) {
                        ok = false;
                        break;
                    }
                    if (MODE == TC_GATHER || TF32) fence_proxy_async_smem();
                    tc_fence_after();
                    const uint32_t sA = smem_u32(sm + stage * C::STAGE_BYTES);
                    const uint32_t sB = sA + C::A_BYTES;
                    const int kvalid = kb < nk0 ? min(KE, a.K0 - kb * KE) : min(KE, a.K1 - (kb - nk0) * KE);
                    if constexpr (TF32) {
                        // K = 8 per MMA; columns past K were filled with zeros by the TMA
                        const int steps = (kvalid + 7) >> 3;
                        for (int k = 0; k < steps; ++k) {
                            const uint64_t ah = sdesc_kmajor_sw128(sA + k * 32), bh = sdesc_kmajor_sw128(sB + k * 32);
                            const uint64_t al = sdesc_kmajor_sw128(sA + C::HALF_BYTES + k * 32);
                            const uint64_t bl = sdesc_kmajor_sw128(sB + C::HALF_BYTES + k * 32);
                            umma_tf32(dtm, ah, bh, idesc, (kb > kb0 || k > 0) ? 1u : 0u);
                            umma_tf32(dtm, ah, bl, idesc, 1u);
                            umma_tf32(dtm, al, bh, idesc, 1u);
                        }
                    } else {
                        const int steps = kvalid >> 4;
                        for (int k = 0; k < steps; ++k)
                            umma_bf16(dtm, sdesc_kmajor_sw128(sA + k * 32), sdesc_kmajor_sw128(sB + k * 32),
                                      idesc, (kb > kb0 || k > 0) ? 1u : 0u);
                    }
                    umma_commit(empty_bar(stage));
                    if (++stage == C::STAGES) {
                        stage = 0;
                        ph ^= 1;
                    }
                }
                if (!ok) break;
                umma_commit(tfull_bar(acc));
                acc ^= 1;
                if (acc == 0) aph ^= 1;
            }
            umma_commit(drain_bar);  // every MMA issued above has completed once this fires
            mbar_wait(drain_bar, 0, nullptr, a.status, 10000000ull);
        }
        __syncwarp();
    } else if (warp < TC_NUM_EPI) {
        // ------------------------------------------------ epilogue
        const int q = warp & 3;
        const int c_lo = (warp >> 2) * C::HALF;
        unsigned char* wstg = stg + warp * 32 * C::STG_ROW;
        constexpr int LPR = C::CW / 8;  // lanes per staged row (16 bytes each)
        constexpr int RPP = 32 / LPR;   // rows per store pass
        int acc = 0;
        uint32_t aph = 0;
        uint32_t kph = 0;  // fp32 K split: parity of the handshake barriers
        volatile int* s_last = reinterpret_cast<volatile int*>(tmem_slot + 2);
        for (int unit = blockIdx.x; unit < num_tiles * ksp; unit += gridDim.x) {
            const int tile = unit / ksp;
            const TileInfo t = decode_tile(a, tile, n_tiles, s_prefix, BN);
            int klo = 0, khi = 1;
            if (TF32) k_range(t, unit % ksp, klo, khi);
            if (!mbar_wait(tfull_bar(acc), aph, abort_flag, a.status, lim)) break;
            tc_fence_after();
            const int r = q * 32 + lane;
            int64_t orow = -1;
            // rows scattered by the grouped epilogue, or by a dense GEMM given a row map (t at its slot)
            if (r < t.rows)
                orow = (a.epi == TC_EPI_SCATTER || (a.mode == TC_DENSE && a.rows)) ? (int64_t)a.rows[t.m0 + r] : t.m0 + r;
            if (TF32 && MODE == TC_DENSE && a.rt_info && r < t.rows) {
                // fp32 fc1: token m's slot from its routing word (expert | rank in its range << 8)
                const int64_t m = t.m0 + r;
                const uint32_t w = (uint32_t)a.rt_info[m];
                const int e = (int)(w & 0xffu);
                orow = -1;
                if (a.rt_cls_stride > 0 && m % a.rt_cls_stride == 0)  // class token: the dense path's slots
                    orow = a.M - n_class_tokens(a.M, a.rt_cls_stride) + m / a.rt_cls_stride;
                else if (e < a.rt_E)
                    orow = (int64_t)s_off[e] + s_tab[(int)(m / a.rt_chunk) * a.rt_E + e] + (int)(w >> 8);
                if ((uint64_t)orow >= (uint64_t)a.M) orow = -1;  // only a routing that gave up
                if (orow >= 0 && t.n0 == 0 && c_lo == 0 && unit % ksp == 0) a.rt_perm[orow] = (int32_t)m;
            }
            const float rsc = (a.group_scale && r < t.rows) ? tc_row_scale(a, t.m0 + r) : 1.f;
            if ((uint64_t)orow >= (uint64_t)a.M) orow = -1;
            // the LayerNorm folded into A: (mean, rstd) of the token whose row this lane holds
            float2 ln = make_float2(0.f, 1.f);
            if (a.ln_stats && r < t.rows) {
                const int64_t tok = a.mode == TC_GATHER ? (int64_t)a.rows[t.m0 + r] : t.m0 + r;
                if ((uint64_t)tok < (uint64_t)a.M) ln = a.ln_stats[tok];
            }
            for (int c = c_lo; c < c_lo + C::HALF; c += C::CW) {
                uint32_t v[32];
                const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN + c;
                if constexpr (C::CW == 8) {
                    CM_TMEM_LD_X8(taddr, v);
                } else {
                    CM_TMEM_LD_X16(taddr, v);
                    if constexpr (C::CW == 32) CM_TMEM_LD_X16(taddr + 16, (v + 16));
                }
                tmem_wait_ld();
                float f[C::CW];
#pragma unroll
                for (int j = 0; j < C::CW; ++j) f[j] = klo < khi ? __uint_as_float(v[j]) : 0.f;
                if (TF32 && ksp > 1) {  // a K range's partial tile, finished by the tile's last unit below
                    if (r < t.rows) {
                        float4* w4 = reinterpret_cast<float4*>(a.ws + ((int64_t)unit * TC_BM + r) * BN + c);
#pragma unroll
                        for (int j4 = 0; j4 < C::CW / 4; ++j4)
                            w4[j4] = make_float4(f[4 * j4], f[4 * j4 + 1], f[4 * j4 + 2], f[4 * j4 + 3]);
                    }
                    continue;
                }
                const int nb = t.n0 + c;
                if (a.ln_stats) {  // W LN(y) = rstd (W y - mean c), c_n = sum_k W[n, k]
#pragma unroll
                    for (int j = 0; j < C::CW; ++j) f[j] = ln.y * fmaf(-ln.x, __ldg(a.ln_colsum + nb + j), f[j]);
                }
                if (TF32 && (a.epi == TC_EPI_BIAS_GELU || a.epi == TC_EPI_BIAS_RELU || a.out_bias)) {
                    // fp32 bias (b1, or fc2's b2), then GELU (CUDA's erff) or ReLU for fc1
                    const bool fc1 = a.epi == TC_EPI_BIAS_GELU || a.epi == TC_EPI_BIAS_RELU;
                    const float4* bp = reinterpret_cast<const float4*>(static_cast<const float*>(fc1 ? a.bias : a.out_bias) + nb);
#pragma unroll
                    for (int j4 = 0; j4 < C::CW / 4; ++j4) {
                        const float4 b = __ldg(bp + j4);
                        const float bb[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                        for (int h = 0; h < 4; ++h) {
                            const float v = f[4 * j4 + h] + bb[h];
                            f[4 * j4 + h] = a.epi == TC_EPI_BIAS_GELU ? gelu_erf(v) : a.epi == TC_EPI_BIAS_RELU ? fmaxf(v, 0.f) : v;
                        }
                    }
                } else if (a.epi == TC_EPI_BIAS_GELU) {
                    const uint4* bp = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(a.bias) + nb);
#pragma unroll
                    for (int j8 = 0; j8 < C::CW / 8; ++j8) {
                        const uint4 b = __ldg(bp + j8);
                        const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                        for (int h = 0; h < 4; ++h) {
                            const float2 g = gelu_pair_as(
                                __fadd2_rn(make_float2(f[j8 * 8 + 2 * h], f[j8 * 8 + 2 * h + 1]),
                                           make_float2(bf16_lo(bw[h]), bf16_hi(bw[h]))));
                            f[j8 * 8 + 2 * h] = g.x;
                            f[j8 * 8 + 2 * h + 1] = g.y;
                        }
                    }
                } else if (a.epi == TC_EPI_BIAS_RELU) {
                    const uint4* bp = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(a.bias) + nb);
#pragma unroll
                    for (int j8 = 0; j8 < C::CW / 8; ++j8) {
                        const uint4 b = __ldg(bp + j8);
                        const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                        for (int h = 0; h < 4; ++h) {
                            f[j8 * 8 + 2 * h] = fmaxf(f[j8 * 8 + 2 * h] + bf16_lo(bw[h]), 0.f);
                            f[j8 * 8 + 2 * h + 1] = fmaxf(f[j8 * 8 + 2 * h + 1] + bf16_hi(bw[h]), 0.f);
                        }
                    }
                } else if (a.out_bias) {
                    const uint4* bp = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(a.out_bias) + nb);
#pragma unroll
                    for (int j8 = 0; j8 < C::CW / 8; ++j8) {
                        const uint4 b = __ldg(bp + j8);
                        const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                        for (int h = 0; h < 4; ++h) {
                            f[j8 * 8 + 2 * h] += bf16_lo(bw[h]);
                            f[j8 * 8 + 2 * h + 1] += bf16_hi(bw[h]);
                        }
                    }
                } else if (a.epi == TC_EPI_SCALE) {
#pragma unroll
                    for (int j4 = 0; j4 < C::CW / 4; ++j4) {
                        const float4 s4 = __ldg(reinterpret_cast<const float4*>(a.scale + nb) + j4);
                        f[4 * j4] *= s4.x;
                        f[4 * j4 + 1] *= s4.y;
                        f[4 * j4 + 2] *= s4.z;
                        f[4 * j4 + 3] *= s4.w;
                    }
                }
                if (a.group_scale) {
#pragma unroll
                    for (int j = 0; j < C::CW; ++j) f[j] *= rsc;
                }
                if (a.c_f32) {  // fp32 output: each lane stores its row's values as computed
                    if (orow >= 0) {
                        float4* dstf = reinterpret_cast<float4*>(static_cast<float*>(a.C) + orow * a.ldc + nb);
#pragma unroll
                        for (int j4 = 0; j4 < C::CW / 4; ++j4)
                            dstf[j4] = make_float4(f[4 * j4], f[4 * j4 + 1], f[4 * j4 + 2], f[4 * j4 + 3]);
                    }
                    continue;
                }
                uint4* dst = reinterpret_cast<uint4*>(wstg + lane * C::STG_ROW);
#pragma unroll
                for (int j8 = 0; j8 < C::CW / 8; ++j8)
                    dst[j8] = make_uint4(pack_bf16(f[8 * j8], f[8 * j8 + 1]), pack_bf16(f[8 * j8 + 2], f[8 * j8 + 3]),
                                         pack_bf16(f[8 * j8 + 4], f[8 * j8 + 5]), pack_bf16(f[8 * j8 + 6], f[8 * j8 + 7]));
                __syncwarp();
#pragma unroll
                for (int p = 0; p < LPR; ++p) {
                    const int rr = p * RPP + lane / LPR;
                    const int64_t o = __shfl_sync(0xffffffffu, orow, rr);
                    const uint4 val = *reinterpret_cast<const uint4*>(wstg + rr * C::STG_ROW + (lane % LPR) * 16);
                    if (o >= 0)
                        *reinterpret_cast<uint4*>(static_cast<uint16_t*>(a.C) + o * a.ldc + nb + (lane % LPR) * 8) = val;
                }
                __syncwarp();
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty_bar(acc));
            acc ^= 1;
            if (acc == 0) aph ^= 1;
            if (TF32 && ksp > 1) {
                // The epilogue warps' partial stores, then one arrival on the tile's counter: the unit
                // that completes it (and resets it) adds the ksp partials in split order and finishes
                // the tile. The handshake uses bounded mbarrier waits.
                __threadfence();
                __syncwarp();
                if (lane == 0) mbar_arrive(kjoin_bar);
                if (warp == 0 && lane == 0) {
                    int last = 0;
                    if (mbar_wait(kjoin_bar, kph, abort_flag, a.status, lim)) {
                        last = atomicAdd(a.cnt + tile, 1) == ksp - 1;
                        if (last) a.cnt[tile] = 0;
                    }
                    *s_last = last;
                    mbar_arrive(kdone_bar);
                }
                const bool done = mbar_wait(kdone_bar, kph, abort_flag, a.status, lim);
                kph ^= 1;
                if (done && *s_last && orow >= 0) {
                    __threadfence();
                    for (int c = c_lo; c < c_lo + C::HALF; c += C::CW) {
                        float f[C::CW];
#pragma unroll
                        for (int j = 0; j < C::CW; ++j) f[j] = 0.f;
                        for (int sp = 0; sp < ksp; ++sp) {
                            const float4* w4 =
                                reinterpret_cast<const float4*>(a.ws + (((int64_t)tile * ksp + sp) * TC_BM + r) * BN + c);
#pragma unroll
                            for (int j4 = 0; j4 < C::CW / 4; ++j4) {
                                const float4 pv = __ldcg(w4 + j4);
                                f[4 * j4] += pv.x;
                                f[4 * j4 + 1] += pv.y;
                                f[4 * j4 + 2] += pv.z;
                                f[4 * j4 + 3] += pv.w;
                            }
                        }
                        const int nb = t.n0 + c;
                        if (a.epi == TC_EPI_BIAS_GELU || a.epi == TC_EPI_BIAS_RELU || a.out_bias) {
                            const bool fc1 = a.epi == TC_EPI_BIAS_GELU || a.epi == TC_EPI_BIAS_RELU;
                            const float* bp = static_cast<const float*>(fc1 ? a.bias : a.out_bias) + nb;
#pragma unroll
                            for (int j = 0; j < C::CW; ++j) {
                                const float v = f[j] + __ldg(bp + j);
                                f[j] = a.epi == TC_EPI_BIAS_GELU ? gelu_erf(v) : a.epi == TC_EPI_BIAS_RELU ? fmaxf(v, 0.f) : v;
                            }
                        } else if (a.epi == TC_EPI_SCALE) {
#pragma unroll
                            for (int j = 0; j < C::CW; ++j) f[j] *= __ldg(a.scale + nb + j);
                        }
                        if (a.group_scale) {
#pragma unroll
                            for (int j = 0; j < C::CW; ++j) f[j] *= rsc;
                        }
                        float4* dstf = reinterpret_cast<float4*>(static_cast<float*>(a.C) + orow * a.ldc + nb);
#pragma unroll
                        for (int j4 = 0; j4 < C::CW / 4; ++j4)
                            dstf[j4] = make_float4(f[4 * j4], f[4 * j4 + 1], f[4 * j4 + 2], f[4 * j4 + 3]);
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == TC_WARP_MMA) tmem_dealloc(tmem_base, C::TMEM_COLS);
}

// ------------------------------------------------------------------ host side
int tc_pick_bn(int mode, int N) {
    (void)mode;
    const int cands[5] = {256, 128, 64, 32, 16};
    for (int c : cands)
        if (N % c == 0) return c;
    return 0;
}

TcTf32Plan tc_plan_tf32(int N, int K, int64_t m_tiles, int num_sms, int64_t ws_floats, int cnt_len) {
    // Cost: bytes the busiest SM moves, i.e. rounds of units x (the unit's TMA stages + the partial
    // tiles its tile's last unit reads back).
    const int64_t kb = (K + 31) / 32;
    const int cands[4] = {128, 64, 32, 16};
    TcTf32Plan best = {0, 1};
    int64_t best_cost = INT64_MAX;
    if (num_sms < 1) num_sms = 1;
    for (int bn : cands) {
        if (N % bn) continue;
        const int64_t tiles = m_tiles * (N / bn);
        int64_t ks = 1;
        if (tiles < num_sms && tiles <= cnt_len) {
            ks = num_sms / tiles;
            if (ks > 8) ks = 8;
            if (ks > kb / 4) ks = kb / 4;
            while (ks > 1 && tiles * ks * TC_BM * bn > ws_floats) --ks;
            if (ks < 1) ks = 1;
        }
        const int64_t rounds = (tiles * ks + num_sms - 1) / num_sms;
        const int64_t unit = (kb + ks - 1) / ks * (TC_BM * 128 + bn * 128);
        const int64_t fix = ks > 1 ? (ks + 1) * (int64_t)TC_BM * bn * 4 : 0;
        const int64_t cost = rounds * (unit + fix);
        if (cost < best_cost) {
            best_cost = cost;
            best = TcTf32Plan{bn, (int)ks};
        }
    }
    return best;
}

template <int BN, int MODE, bool TF32>
static cudaError_t launch_one(const TcGemmArgs& a, int num_sms, cudaStream_t s) {
    using C = TcCfg<BN, TF32>;
    const cudaError_t e = smem_attr_once((const void*)tc_gemm_kernel<BN, MODE, TF32>, C::SMEM);
    if (e != cudaSuccess) return e;
    const int n_tiles = a.N / BN;
    int64_t m_tiles = (a.M + TC_BM - 1) / TC_BM;
    if (MODE == TC_GROUPED) m_tiles += a.E;
    // units: tiles, or (fp32 with a K split) tiles x ksplit
    const int64_t tiles = m_tiles * n_tiles * ((TF32 && a.ksplit > 1) ? a.ksplit : 1);
    const int grid = (int)(tiles < num_sms ? tiles : num_sms);
    if (grid <= 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3((MODE == TC_GATHER || TF32) ? TC_THREADS_GATHER : TC_THREADS_TMA);
    cfg.dynamicSmemBytes = C::SMEM;
    cfg.stream = s;
    cudaLaunchAttribute attr_pdl[1];
    attr_pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr_pdl[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr_pdl;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, tc_gemm_kernel<BN, MODE, TF32>, a);
}

template <int MODE>
static cudaError_t launch_mode(const TcGemmArgs& a, int bn, int num_sms, cudaStream_t s) {
    switch (bn) {
        case 256: return launch_one<256, MODE, false>(a, num_sms, s);
        case 128: return launch_one<128, MODE, false>(a, num_sms, s);
        case 64: return launch_one<64, MODE, false>(a, num_sms, s);
        case 32: return launch_one<32, MODE, false>(a, num_sms, s);
        case 16: return launch_one<16, MODE, false>(a, num_sms, s);
        default: return cudaErrorInvalidValue;
    }
}

template <int MODE>
static cudaError_t launch_mode_tf32(const TcGemmArgs& a, int bn, int num_sms, cudaStream_t s) {
    switch (bn) {
        case 128: return launch_one<128, MODE, true>(a, num_sms, s);
        case 64: return launch_one<64, MODE, true>(a, num_sms, s);
        case 32: return launch_one<32, MODE, true>(a, num_sms, s);
        case 16: return launch_one<16, MODE, true>(a, num_sms, s);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_tc_gemm(const TcGemmArgs& a, int num_sms, cudaStream_t s) {
    if (a.tf32) {  // fp32 operands: dense and grouped modes, fp32 output
        if (a.mode == TC_GATHER || !a.c_f32 || a.ln_stats || a.ln_aug) return cudaErrorInvalidValue;
        const int bn = a.bn_tf32;
        if (bn <= 0 || a.N % bn) return cudaErrorInvalidValue;
        if (a.ksplit > 1) {  // the workspace and counters must hold every tile's partials
            int64_t m_tiles = (a.M + TC_BM - 1) / TC_BM;
            if (a.mode == TC_GROUPED) m_tiles += a.E;
            const int64_t tiles = m_tiles * (a.N / bn);
            if (!a.ws || !a.cnt || tiles > a.cnt_len || tiles * a.ksplit * TC_BM * bn > a.ws_floats)
                return cudaErrorInvalidValue;
        }
        if (a.mode == TC_GROUPED) return launch_mode_tf32<TC_GROUPED>(a, bn, num_sms, s);
        return launch_mode_tf32<TC_DENSE>(a, bn, num_sms, s);
    }
    const int bn = tc_pick_bn(a.mode, a.N);
    if (bn == 0) return cudaErrorInvalidValue;
    if (a.mode == TC_GATHER) return launch_mode<TC_GATHER>(a, bn, num_sms, s);
    if (a.mode == TC_GROUPED) return launch_mode<TC_GROUPED>(a, bn, num_sms, s);
    return launch_mode<TC_DENSE>(a, bn, num_sms, s);
}

namespace {
constexpr int kMaxDevices = 64;
struct AttrEntry {
    int dev;
    const void* fn;
    int bytes;
};
std::mutex g_attr_mu;
AttrEntry g_attr[256];
int g_nattr = 0;
int g_sms[kMaxDevices] = {};
}  // namespace

cudaError_t smem_attr_once(const void* fn, int bytes) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_attr_mu);
    for (int i = 0; i < g_nattr; ++i)
        if (g_attr[i].dev == dev && g_attr[i].fn == fn && g_attr[i].bytes >= bytes) return cudaSuccess;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    for (int i = 0; i < g_nattr; ++i)
        if (g_attr[i].dev == dev && g_attr[i].fn == fn) {
            g_attr[i].bytes = bytes;
            return cudaSuccess;
        }
    if (g_nattr < 256) g_attr[g_nattr++] = AttrEntry{dev, fn, bytes};  // else set again on every call
    return cudaSuccess;
}

int current_device_sms() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    std::lock_guard<std::mutex> lock(g_attr_mu);
    if (dev >= 0 && dev < kMaxDevices && g_sms[dev]) return g_sms[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    if (dev >= 0 && dev < kMaxDevices) g_sms[dev] = n;
    return n;
}

typedef CUresult (*PFN_encodeTiled_t)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                      const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                      const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                      CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// Encoded maps are cached by (base, rows, cols, box rows, box chunks), which determine them
// entirely: a forward encodes up to ~20 maps, and the driver call costs microseconds each on the host.
namespace {
struct TmapEntry {
    const void* base;
    int64_t rows, cols;
    int box_rows, box_chunks, elem;
    bool valid;
    CUtensorMap map;
};
constexpr int TMAP_CACHE = 64;
TmapEntry g_tmaps[TMAP_CACHE];
int g_tmap_next = 0;
std::mutex g_tmap_mu;
}  // namespace

static int encode_tmap_uncached(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows,
                                int box_chunks, int elem);

static int encode_tmap_cached(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows,
                              int box_chunks, int elem) {
    std::lock_guard<std::mutex> lock(g_tmap_mu);
    for (int i = 0; i < TMAP_CACHE; ++i) {
        const TmapEntry& c = g_tmaps[i];
        if (c.valid && c.base == base && c.rows == rows && c.cols == cols && c.box_rows == box_rows &&
            c.box_chunks == box_chunks && c.elem == elem) {
            *map = c.map;
            return 0;
        }
    }
    const int rc = encode_tmap_uncached(map, base, rows, cols, box_rows, box_chunks, elem);
    if (rc == 0) {
        TmapEntry& c = g_tmaps[g_tmap_next];
        c = TmapEntry{base, rows, cols, box_rows, box_chunks, elem, true, *map};
        g_tmap_next = (g_tmap_next + 1) % TMAP_CACHE;
    }
    return rc;
}

int encode_tmap_bf16(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows) {
    return encode_tmap_cached(map, base, rows, cols, box_rows, 0, 2);
}

int encode_tmap_bf16_chunks(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows,
                            int box_chunks) {
    if (box_chunks < 1 || cols % TC_BK != 0 || box_chunks > cols / TC_BK) return -2;
    return encode_tmap_cached(map, base, rows, cols, box_rows, box_chunks, 2);
}

int encode_tmap_f32(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows) {
    if (cols % 4 != 0) return -2;  // the row pitch must be a multiple of 16 bytes
    return encode_tmap_cached(map, base, rows, cols, box_rows, 0, 4);
}

static int encode_tmap_uncached(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows,
                                int box_chunks, int elem) {
    static PFN_encodeTiled_t fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !p)
            return -1;
        fn = reinterpret_cast<PFN_encodeTiled_t>(p);
    }
    CUresult r;
    if (elem == 4) {  // fp32 [rows x cols]: boxes of 32 columns (128 bytes) x box_rows rows
        const cuuint64_t gdim[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
        const cuuint64_t gstride[1] = {(cuuint64_t)cols * 4};
        const cuuint32_t box[2] = {(cuuint32_t)(TC_BK / 2), (cuuint32_t)box_rows};
        const cuuint32_t es[2] = {1, 1};
        r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), gdim, gstride, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    } else if (box_chunks == 0) {  // [rows x cols]: boxes of 64 columns x box_rows rows
        const cuuint64_t gdim[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
        const cuuint64_t gstride[1] = {(cuuint64_t)cols * 2};
        const cuuint32_t box[2] = {(cuuint32_t)TC_BK, (cuuint32_t)box_rows};
        const cuuint32_t es[2] = {1, 1};
        r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    } else {  // the same matrix as {64 columns, rows, cols / 64 chunks}: boxes of 64 x box_rows x box_chunks
        const cuuint64_t gdim[3] = {(cuuint64_t)TC_BK, (cuuint64_t)rows, (cuuint64_t)(cols / TC_BK)};
        const cuuint64_t gstride[2] = {(cuuint64_t)cols * 2, (cuuint64_t)TC_BK * 2};
        const cuuint32_t box[3] = {(cuuint32_t)TC_BK, (cuuint32_t)box_rows, (cuuint32_t)box_chunks};
        const cuuint32_t es[3] = {1, 1, 1};
        r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), gdim, gstride, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    }
    return r == CUDA_SUCCESS ? 0 : -2;
}

}  // namespace cm
