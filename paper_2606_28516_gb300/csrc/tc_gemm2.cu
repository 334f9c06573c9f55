// 2-SM bf16 GEMMs of the CLEAR-MoE FFN (tcgen05 cta_group::2, sm_103a).
//
// A cluster of two CTAs (one per SM of a pair) computes a 256 x 256 tile: CTA r loads A rows
// [m0 + 128 r, +128) and B rows [n0 + 128 r, +128) into its own shared memory, and one thread of
// the even CTA issues tcgen05.mma.cta_group::2 (M = 256, N = 256, K = 16), which reads A split by M
// and B split by N across the two CTAs and leaves rows [128 r, +128) of the accumulator in CTA r's
// tensor memory. Each SM thus holds half of the B tile: a k-block costs it 32 KB of operands for
// 128 x 256 x 64 MACs instead of 48 KB, so a 6-stage ring covers the load latency.
//
// Hand-offs: both CTAs' TMA loads complete on the even CTA's full barrier (the odd CTA's loads
// name it through the cluster); the even CTA's MMA commits arrive on both CTAs' empty / tfull
// barriers (multicast); the epilogue warps of both CTAs arrive on the even CTA's tempty barrier.
// Modes: dense (one K segment, epilogue bias+GELU / plain store; with a LayerNorm folded into A, one
// more K block of 16 useful columns carries -mean W 1 and the bias add scales by rstd) and grouped (the residual
// experts: tile pairs never straddle an expert, K chain [z | t] x [W_e | U_r]; with dense_last
// the last group is the class tokens' dense path, K chain z x W2 alone). Store epilogues may add
// an output bias (fc2's b2). With a.rows set,
// output row m goes to C[a.rows[m]] (fc1: inv[token] = slot; grouped: perm[slot] = token).
// Every wait is bounded; both CTAs always reach the closing cluster barrier.
#include "common.cuh"
#include "internal.h"

namespace cm {
// Tile configuration by pair-tile width BN (256, 192 or 128 columns) and epilogue warps NEPI (8,
// or 12 for short K, where the epilogue rather than the MMA bounds a tile).
template <int BN_, int NEPI_ = 8>
struct T2 {
    static constexpr int BM = 128;                        // rows per CTA; the pair covers 256
    static constexpr int BN = BN_;                        // columns per pair tile
    static constexpr int BH = BN / 2;                     // B rows per CTA
    static constexpr int BK = 64;
    static constexpr int A_BYTES = BM * BK * 2;           // 16 KB
    static constexpr int B_BYTES = BH * BK * 2;           // 16 KB (BN 256), 12 KB (192), 8 KB (128)
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    // at most 192 KB of operands (6 / 6 / 8 stages); 160 KB with 12 epilogue warps (their staging)
    static constexpr int STAGES = (NEPI_ == 8 ? 192 : 160) * 1024 / STAGE_BYTES;
    static constexpr int NUM_EPI = NEPI_;                 // two or three per TMEM lane quarter
    static constexpr int WARP_MMA = NUM_EPI, WARP_TMA = NUM_EPI + 1;
    static constexpr int THREADS = 32 * (WARP_TMA + 1);
    static constexpr int CW = 32;                         // columns per tensor-memory read
    static constexpr int NCH = BN / CW;                   // 32-column chunks per tile
    // chunks of the tile of epilogue warp group g (the warps g * 4 .. g * 4 + 3): [g NCH / G, (g + 1) NCH / G)
    static constexpr int GROUPS = NUM_EPI / 4;
    // Staging: 1 KB per epilogue warp (32 x STG_ROW bytes), which each half warp in turn fills
    // with its 16 rows of one 32-column chunk as 64-byte rows (layout at the epilogue).
    static constexpr int STG_ROW = 32;
    static constexpr int STG_BYTES = NUM_EPI * 32 * STG_ROW;
    static constexpr int BIAS_CAP = TC2_BIAS_CAP;         // fp32 bias / scale staged in shared memory
    static constexpr int TAB_CAP = TC2_TAB_CAP;           // routing prefix table (fused fc1)
    static constexpr int NBARS = 2 * STAGES + 7;  // + 2 for the router inside fc1
    static constexpr int FR_B_BYTES = 16 * BK * 2;        // the router unit's B box per CTA: 16 rows of W_g
    static constexpr int SMEM =
        1024 + STAGES * STAGE_BYTES + STG_BYTES + BIAS_CAP * 4 + (TAB_CAP + CM_MAX_E) * 4 + NBARS * 8 + 128;
    static constexpr int TMEM_COLS = 2 * BN <= 256 ? 256 : 512;  // two accumulators (a power of 2)
};

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t map_to_rank(uint32_t smem_addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr), "r"(rank));
    return r;
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int32_t c0, int32_t c1,
                                                 uint32_t bar_cluster) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.cta_group::2"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar_cluster)
        : "memory");
}
__device__ __forceinline__ void tma_load_2d_pair_hint(uint32_t dst, const CUtensorMap* map, int32_t c0, int32_t c1,
                                                      uint32_t bar_cluster, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.cta_group::2.L2::cache_hint"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar_cluster), "l"(policy)
        : "memory");
}
// Four rows (r0..r3, one row high boxes of 64 bf16 each) of a 2-D tensor into 512 contiguous bytes
// of shared memory, in the layout a four-row box would have there; completion on the even CTA's barrier.
__device__ __forceinline__ void tma_gather4_pair(uint32_t dst, const CUtensorMap* map, int32_t c0, int32_t r0,
                                                 int32_t r1, int32_t r2, int32_t r3, uint32_t bar_cluster) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes.cta_group::2"
        " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(bar_cluster)
        : "memory");
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ void umma2_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma2_commit_both(uint32_t bar) {  // arrive on bar in both CTAs
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            bar),
        "h"((unsigned short)3)
        : "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_cluster) {
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}

struct PairTile {
    int64_t m0;  // first row of the pair tile (CTA r starts at m0 + 128 r)
    int64_t hi;  // rows >= hi belong to another expert or lie past T
    int n0;
    int e;
    bool router;  // the router unit of the pair tile (the router inside fc1)
};

// Kernel variants: the plain dense and grouped GEMMs, the dense GEMM with the router unit (the
// router inside fc1), and the grouped GEMM whose z rows are gathered by slot. Each variant is its own
// instantiation, so the plain kernels carry none of the others' code.
enum Tc2Var { TC2_PLAIN = 0, TC2_ROUTER = 1, TC2_GATHER = 2, TC2_EPI12 = 3 };
// TC2_EPI12: the plain dense GEMM with 12 epilogue warps (three per TMEM lane quarter) and a 160 KB
// operand ring, for short K (fc1 at d <= 512), where the epilogue's GELU bounds a tile.
template <int BN, int VAR>
using T2v = T2<BN, VAR == TC2_EPI12 ? 12 : 8>;

// Units per 256-row pair tile: the column tiles, plus the router unit when the router runs inside fc1.
template <int VAR>
__device__ __forceinline__ int units_per_pair(int n_tiles) {
    return n_tiles + (VAR == TC2_ROUTER ? 1 : 0);
}

template <int BN, int VAR>
__device__ __forceinline__ PairTile decode_pair(const TcGemmArgs& a, int unit, int n_tiles, const int* s_prefix) {
    constexpr int BM = T2<BN>::BM;
    PairTile t;
    const int nup = units_per_pair<VAR>(n_tiles);
    const int mp = unit / nup;
    t.n0 = (unit % nup) * BN;
    t.router = VAR == TC2_ROUTER && (unit % nup) == n_tiles;
    if (a.mode == TC_GROUPED) {
        int e = 0;
        while (e + 1 < a.E && s_prefix[e + 1] <= mp) ++e;
        t.m0 = tc_group_off(a, e) + (int64_t)(mp - s_prefix[e]) * 2 * BM;
        t.hi = tc_group_off(a, e + 1);
        t.e = e;
    } else {
        t.m0 = (int64_t)mp * 2 * BM;
        t.hi = a.M;
        t.e = 0;
    }
    return t;
}

template <int BN_, int MODE, int VAR>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(T2v<BN_, VAR>::THREADS, 1)
    tc_gemm2_kernel(const __grid_constant__ TcGemmArgs a) {
    using C = T2v<BN_, VAR>;
    constexpr int BM = C::BM, BN = C::BN, BH = C::BH, BK = C::BK, A_BYTES = C::A_BYTES;
    constexpr int STAGE_BYTES = C::STAGE_BYTES, STAGES = C::STAGES, NUM_EPI = C::NUM_EPI;
    constexpr int WARP_MMA = C::WARP_MMA, WARP_TMA = C::WARP_TMA, CW = C::CW;
    constexpr int STG_ROW = C::STG_ROW, STG_BYTES = C::STG_BYTES, BIAS_CAP = C::BIAS_CAP, NBARS = C::NBARS;
    constexpr int TMEM_COLS = C::TMEM_COLS;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    unsigned char* sm = smem_raw + ((1024 - (raw_addr & 1023)) & 1023);
    unsigned char* stg = sm + STAGES * STAGE_BYTES;
    float* s_bias = reinterpret_cast<float*>(stg + STG_BYTES);
    int* s_tab = reinterpret_cast<int*>(s_bias + BIAS_CAP);  // [range][expert] tokens before
    int* s_off = s_tab + C::TAB_CAP;                           // [expert] offsets
    uint64_t* bars = reinterpret_cast<uint64_t*>(s_off + CM_MAX_E);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NBARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    int* s_prefix = reinterpret_cast<int*>(tmem_slot + 4);  // [CM_MAX_E + 1]

    if (!a.pdl_trigger_late) pdl_launch_dependents();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const bool leader = rank == 0;
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto tfull_bar = [&](int i) { return bar0 + 8u * (2 * STAGES + i); };
    auto tempty_bar = [&](int i) { return bar0 + 8u * (2 * STAGES + 2 + i); };
    const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);
    // the router inside fc1: the four lane-quarter warps' expert counts of a router unit are
    // exchanged through shared memory, double-buffered, each buffer guarded by its own barrier
    auto fr_bar = [&](int i) { return bar0 + 8u * (2 * STAGES + 5 + i); };
    int* s_frc = s_tab;                                            // [2][4][CM_MAX_E] counts
    float* s_frb = reinterpret_cast<float*>(s_tab + 8 * CM_MAX_E);  // [CM_MAX_E] b_g
    const uint64_t lim = (uint64_t)a.wait_limit_ns;

    const int n_tiles = a.N / BN;
    const int nk0 = (a.K0 + BK - 1) / BK;
    // grouped: the z x W_e^res segment; dense: the LayerNorm augmentation block, if any
    const int nk1 = MODE == TC_GROUPED ? (a.K1 + BK - 1) / BK : (a.ln_aug ? 1 : 0);
    const int nkb = nk0 + nk1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full_bar(s), 1);   // the even CTA's producer arrives; both CTAs' bytes land here
            mbar_init(empty_bar(s), 1);  // one multicast commit per stage
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(tfull_bar(i), 1);
            mbar_init(tempty_bar(i), 2 * NUM_EPI);  // epilogue warps of both CTAs
        }
        mbar_init(drain_bar, 1);
        mbar_init(fr_bar(0), 4);  // the quarter warps of the first column group
        mbar_init(fr_bar(1), 4);
        *abort_flag = 0;
        mbar_fence_init();
    }
    // The bias or the column scale (weights, not produced by the previous kernel) as fp32, once per CTA.
    if (MODE == TC_DENSE && (a.epi == TC_EPI_BIAS_GELU || a.epi == TC_EPI_BIAS_RELU) && warp < NUM_EPI) {
        const uint16_t* b = static_cast<const uint16_t*>(a.bias);
        for (int n = threadIdx.x; n < a.N; n += NUM_EPI * 32) s_bias[n] = __uint_as_float((uint32_t)b[n] << 16);
    } else if (MODE == TC_DENSE && a.epi == TC_EPI_SCALE && warp < NUM_EPI) {
        for (int n = threadIdx.x; n < a.N; n += NUM_EPI * 32) s_bias[n] = a.scale[n];
    } else if (a.out_bias && warp < NUM_EPI) {
        const uint16_t* b = static_cast<const uint16_t*>(a.out_bias);
        for (int n = threadIdx.x; n < a.N; n += NUM_EPI * 32) s_bias[n] = __uint_as_float((uint32_t)b[n] << 16);
    }
    if (VAR == TC2_ROUTER && threadIdx.x < a.fr_E)  // the router's bias (a weight)
        s_frb[threadIdx.x] = __uint_as_float((uint32_t) static_cast<const uint16_t*>(a.fr_bias)[threadIdx.x] << 16);
    // Tensor memory for the pair: allocated collectively by one warp of each CTA. The two CTAs
    // must see the same base (the even CTA's MMAs name it for both); a mismatch aborts cleanly.
    if (warp == WARP_MMA) {
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // barriers initialised and TMEM bases written in both CTAs
    tc_fence_after();
    // everything above overlaps the predecessor kernel; from here on its results are read (by
    // every thread, or by the roles that read them: see pdl_wait_role)
    if (a.pdl_wait_role == 0 || (a.pdl_wait_role == 1 && warp < NUM_EPI)) pdl_wait();
    if (a.pdl_trigger_late) pdl_launch_dependents();
    if (MODE == TC_DENSE && a.rt_info && warp < NUM_EPI) {
        // Routing prefix table, by the epilogue warps while the producer and MMA warps start:
        // thread c holds routing range c's counts; per expert, an exclusive scan over ranges (warp
        // scans, warp totals in the staging area, named barrier 1 among the epilogue warps).
        int* s_wt = reinterpret_cast<int*>(stg);  // [NUM_EPI][CM_MAX_E], before the staging is used
        const int c = threadIdx.x;
        const int E = a.rt_E;
        int cnt[CM_MAX_E], incl[CM_MAX_E];
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) cnt[e] = 0;
        if (c < a.rt_ctas) {
            const int4* row = reinterpret_cast<const int4*>(a.rt_counts + (size_t)c * CM_MAX_E);
#pragma unroll
            for (int q = 0; q < CM_MAX_E / 4; ++q) {
                if (4 * q < E) {
                    const int4 v = __ldcg(row + q);
                    cnt[4 * q] = v.x;
                    cnt[4 * q + 1] = v.y;
                    cnt[4 * q + 2] = v.z;
                    cnt[4 * q + 3] = v.w;
                }
            }
        }
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) {
            incl[e] = cnt[e];
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl[e], off);
                if (lane >= off) incl[e] += v;
            }
            if (lane == 31 && e < E) s_wt[warp * CM_MAX_E + e] = incl[e];
        }
        asm volatile("bar.sync 1, %0;" ::"n"(NUM_EPI * 32) : "memory");
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) {
            if (e < E) {
                int before = incl[e] - cnt[e];
                for (int w = 0; w < warp; ++w) before += s_wt[w * CM_MAX_E + e];
                if (c < a.rt_ctas) s_tab[c * E + e] = before;
            }
        }
        if (warp == 0) {  // lane e: expert totals, offsets by a scan over experts
            int tot = 0;
            if (lane < E)
                for (int w = 0; w < NUM_EPI; ++w) tot += s_wt[w * CM_MAX_E + lane];
            int sc = tot;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, sc, off);
                if (lane >= off) sc += v;
            }
            if (lane < E) {
                s_off[lane] = sc - tot;
                if (blockIdx.x == 0) {
                    a.rt_out_counts[lane] = tot;
                    a.rt_out_offsets[lane] = sc - tot;
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
        asm volatile("bar.sync 1, %0;" ::"n"(NUM_EPI * 32) : "memory");
    }
    if (MODE == TC_GROUPED) {
        if (threadIdx.x == 0) {
            int acc = 0;
            for (int e = 0; e < a.E; ++e) {
                s_prefix[e] = acc;
                acc += (int)((tc_group_off(a, e + 1) - tc_group_off(a, e) + 2 * BM - 1) / (2 * BM));
            }
            s_prefix[a.E] = acc;
        }
        __syncthreads();
    }
    const uint32_t tmem_base = *tmem_slot;
    uint32_t peer_base;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(peer_base) : "r"(map_to_rank(smem_u32(tmem_slot), rank ^ 1)));
    const bool tmem_ok = peer_base == tmem_base;
    if (!tmem_ok && threadIdx.x == 0) set_status(a.status, CLEARMOE_ECUDA);
    constexpr int nacc = 2;  // accumulator buffers

    int m_pairs;
    if (MODE == TC_GROUPED)
        m_pairs = s_prefix[a.E];
    else
        m_pairs = (int)((a.M + 2 * BM - 1) / (2 * BM));
    const int num_units = tmem_ok ? m_pairs * units_per_pair<VAR>(n_tiles) : 0;
    const int cid = blockIdx.x >> 1, ncl = gridDim.x >> 1;

    if (warp == WARP_TMA) {
        // ------------------------------------------------ producers (both CTAs)
        // Lane 0 waits for free stages and issues the tile loads; with the z rows gathered by slot
        // (a1_rows) every lane issues one four-row gather per stage (32 x 4 = the CTA's 128 rows),
        // otherwise lane 0 runs alone.
        const uint32_t full_leader0 = map_to_rank(full_bar(0), 0);
        const uint64_t pol_a = l2_policy_evict_first();
        constexpr bool gather = VAR == TC2_GATHER;
        bool waited = a.pdl_wait_role != 2;  // role 2: wait before the first t-segment load
        int stage = 0;
        uint32_t ph = 0;
        bool ok = gather || lane == 0;
        for (int u = cid; u < num_units && ok; u += ncl) {
            const PairTile t = decode_pair<BN, VAR>(a, u, n_tiles, s_prefix);
            const int am = (int)(t.m0 + (int64_t)rank * BM);
            // the router unit: CTA r supplies W_g rows [16 r, +16) of the 256 x 32 MMA
            const int bn = t.router ? (int)rank * 16 : t.n0 + (int)rank * BH;
            const uint32_t stage_tx = t.router ? 2u * (A_BYTES + C::FR_B_BYTES) : 2u * STAGE_BYTES;
            const int nkb_t = (MODE == TC_GROUPED && a.dense_last && t.e == a.E - 1) ? nk1 : nkb;
            int32_t gr[4] = {0, 0, 0, 0};
            if (gather) {  // this lane's four slots; slots past M take the last one (their rows are dropped)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    int64_t sl = (int64_t)am + 4 * lane + j;
                    if (sl > a.M - 1) sl = a.M - 1;
                    const int32_t tok = a.a1_rows[sl];
                    gr[j] = (uint32_t)tok < (uint64_t)a.M ? tok : 0;  // only a routing that gave up
                }
            }
            for (int kb = 0; kb < nkb_t; ++kb) {
                int w_ok = 1;
                if (lane == 0) w_ok = mbar_wait(empty_bar(stage), ph ^ 1, abort_flag, a.status, lim);
                if constexpr (gather) w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
                if (!w_ok) {
                    ok = false;
                    break;
                }
                const uint32_t sA = smem_u32(sm + stage * STAGE_BYTES);
                const uint32_t sB = sA + A_BYTES;
                const uint32_t fb = full_leader0 + 8u * stage;  // the even CTA's full barrier
                if (leader && lane == 0) mbar_arrive_expect_tx(full_bar(stage), stage_tx);
                const CUtensorMap* mA;
                const CUtensorMap* mB;
                int kk;
                bool gathered = false;
                if (MODE != TC_GROUPED) {  // x x W (or x x W_g), then the augmentation block
                    mA = kb < nk0 ? &a.tmA0 : &a.tmA1;
                    mB = t.router ? &a.tmR : kb < nk0 ? &a.tmB0 : &a.tmB1[0];
                    kk = kb < nk0 ? kb * BK : 0;
                } else if (kb < nk1) {  // z x W_e^res
                    mA = &a.tmA1;
                    mB = &a.tmB1[t.e];
                    kk = kb * BK;
                    gathered = gather;
                } else {  // t x U_r
                    if (!waited) {
                        pdl_wait();
                        waited = true;
                    }
                    mA = &a.tmA0;
                    mB = &a.tmB0;
                    kk = (kb - nk1) * BK;
                }
                if (gathered) {
                    tma_gather4_pair(sA + 512u * lane, mA, kk, gr[0], gr[1], gr[2], gr[3], fb);
                } else if (lane == 0) {
                    if (a.a_evict_first)
                        tma_load_2d_pair_hint(sA, mA, kk, am, fb, pol_a);
                    else
                        tma_load_2d_pair(sA, mA, kk, am, fb);
                }
                if (lane == 0) tma_load_2d_pair(sB, mB, kk, bn, fb);
                if (++stage == STAGES) {
                    stage = 0;
                    ph ^= 1;
                }
            }
        }
    } else if (warp == WARP_MMA) {
        // ------------------------------------------------ MMA issuer (even CTA)
        if (leader && lane == 0) {
            const uint32_t idesc_t = idesc_bf16_f32(2 * BM, BN);
            const uint32_t idesc_r = idesc_bf16_f32(2 * BM, 32);  // the router unit: 256 x 32
            const int nup = units_per_pair<VAR>(n_tiles);
            // Stage s's descriptors are the stage-0 ones plus the byte offset / 16 in the start
            // address field (every shared address here is below 256 KB, so the field never carries).
            const uint64_t dA0 = sdesc_kmajor_sw128(smem_u32(sm));
            int stage = 0;
            uint32_t ph = 0;
            int acc = 0;
            uint32_t aph = 0;
            bool ok = true;
            for (int u = cid; u < num_units && ok; u += ncl) {
                if (!mbar_wait(tempty_bar(acc), aph ^ 1, abort_flag, a.status, lim)) break;
                tc_fence_after();
                const uint32_t dtm = tmem_base + acc * BN;
                const uint32_t idesc = (VAR == TC2_ROUTER && u % nup == n_tiles) ? idesc_r : idesc_t;
                int nkb_t = nkb;  // the dense path's group: the z x W2 segment alone
                if (MODE == TC_GROUPED && a.dense_last && decode_pair<BN, VAR>(a, u, n_tiles, s_prefix).e == a.E - 1)
                    nkb_t = nk1;
                for (int kb = 0; kb < nkb_t; ++kb) {
                    if (!mbar_wait(full_bar(stage), ph, abort_flag, a.status, lim)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t da = dA0 + (uint64_t)((stage * STAGE_BYTES) >> 4);
                    const uint64_t db = da + (uint64_t)(A_BYTES >> 4);
                    int krem;
                    if (MODE != TC_GROUPED)  // the augmentation block's products sit in its first 16 columns
                        krem = kb < nk0 ? a.K0 - kb * BK : 16;
                    else
                        krem = kb < nk1 ? a.K1 - kb * BK : a.K0 - (kb - nk1) * BK;
                    if (krem >= BK) {
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)  // 16 K-elements = 32 bytes = 2 descriptor units
                            umma2_bf16(dtm, da + 2 * k, db + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                    } else {
                        for (int k = 0; k < (krem >> 4); ++k)
                            umma2_bf16(dtm, da + 2 * k, db + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                    }
                    umma2_commit_both(empty_bar(stage));
                    if (++stage == STAGES) {
                        stage = 0;
                        ph ^= 1;
                    }
                }
                if (!ok) break;
                umma2_commit_both(tfull_bar(acc));
                if (++acc == nacc) {
                    acc = 0;
                    aph ^= 1;
                }
            }
            asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(drain_bar)
                         : "memory");
            mbar_wait(drain_bar, 0, nullptr, a.status, 10000000ull);
        }
        __syncwarp();
    } else if (warp < NUM_EPI) {
        // ------------------------------------------------ epilogue (both CTAs, own 128 rows)
        const int q = warp & 3;  // a warp reads the TMEM lanes of its index mod 4
        // this warp's columns of every tile: chunks [grp NCH / GROUPS, (grp + 1) NCH / GROUPS)
        const int grp = warp >> 2;
        const int c_lo = CW * (grp * C::NCH / C::GROUPS), c_hi = CW * ((grp + 1) * C::NCH / C::GROUPS);
        unsigned char* wstg = stg + warp * 32 * STG_ROW;
        // Staging by half warps: the 16 rows of lanes 16 h .. 16 h + 15 as 64-byte rows (a 32-column
        // chunk), 16-byte piece j of row r at piece j ^ ((r >> 1) & 3) (conflict-free for the
        // row-wise writes and the 4-lanes-per-row reads); each store instruction then writes
        // 8 rows x 64 contiguous bytes.
        static_assert(CW == 32 && 16 * 64 == 32 * STG_ROW, "a half warp's 64-byte rows fill the warp's staging");
        const uint32_t tempty_leader0 = map_to_rank(tempty_bar(0), 0);
        int acc = 0;
        uint32_t aph = 0;
        int fr_it = 0;  // router units handled so far (the router inside fc1)
        for (int u = cid; u < num_units; u += ncl) {
            const PairTile t = decode_pair<BN, VAR>(a, u, n_tiles, s_prefix);
            const int64_t mrow = t.m0 + (int64_t)rank * BM + q * 32 + lane;
            // the token's routing word, loaded before the accumulator wait so that the wait hides it
            const uint32_t rtw = (MODE == TC_DENSE && a.rt_info && mrow < t.hi) ? (uint32_t)a.rt_info[mrow] : 0u;
            // the LayerNorm folded into A: (mean, rstd) of this lane's row, loaded early for the same reason
            const float2 ln = (a.ln_stats && mrow < t.hi) ? a.ln_stats[mrow] : make_float2(0.f, 1.f);
            if (!mbar_wait(tfull_bar(acc), aph, abort_flag, a.status, lim)) break;
            tc_fence_after();
            if (VAR == TC2_ROUTER && t.router) {
                // The router unit: accumulator columns [0, E) of this lane's row hold W_g x. The four
                // warps of the first column group (one per lane quarter) add b_g, take the argmax
                // (lowest index on ties), count each expert's rows of the quarter by ballots, and
                // exchange the counts through shared memory (a barrier per buffer, bounded waits):
                // rank = earlier quarters' rows of the expert + earlier lanes' of this quarter.
                if (c_lo == 0) {
                    const int E = a.fr_E;
                    const int rb = fr_it & 1;
                    int* rc = s_frc + rb * 4 * CM_MAX_E;
                    uint32_t v[16];
                    CM_TMEM_LD_X16(tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN, v);
                    tmem_wait_ld();
                    int esel = -1;
                    if (mrow < t.hi) {
                        float bv = -INFINITY;
                        int be = 0x7fffffff;
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            if (e < E) {
                                const float l = __uint_as_float(v[e]) + s_frb[e];
                                if (l > bv || (l == bv && e < be)) {
                                    bv = l;
                                    be = e;
                                }
                            }
                        }
                        esel = be < E ? be : 0;  // only reachable with non-finite logits
                    }
                    int rk = 0;
                    for (int e = 0; e < E; ++e) {
                        const unsigned mk = __ballot_sync(0xffffffffu, esel == e);
                        if (lane == 0) rc[q * CM_MAX_E + e] = __popc(mk);
                        if (esel == e) rk = __popc(mk & ((1u << lane) - 1u));
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(fr_bar(rb));
                    if (mbar_wait(fr_bar(rb), (uint32_t)(fr_it >> 1) & 1u, abort_flag, a.status, lim)) {
                        if (esel >= 0) {
                            int base = 0;
                            for (int qq = 0; qq < q; ++qq) base += rc[qq * CM_MAX_E + esel];
                            a.fr_idx[mrow] = esel;
                            a.fr_info[mrow] = esel | ((base + rk) << 8);
                        }
                        const int64_t rng = t.m0 / FR_RANGE + rank;  // this CTA's 128-row range
                        if (q == 0 && lane < E && rng * FR_RANGE < a.M) {
                            int c = 0;
                            for (int qq = 0; qq < 4; ++qq) c += rc[qq * CM_MAX_E + lane];
                            a.fr_counts[rng * CM_MAX_E + lane] = c;
                        }
                    }
                }
                ++fr_it;
            } else {
                int64_t orow = -1;
                if (mrow < t.hi) {
                    if (MODE == TC_DENSE && a.rt_info) {  // the token's routing slot
                        const uint32_t w = rtw;
                        const int e = (int)(w & 0xffu);
                        const int rc = (int)((uint32_t)mrow / (uint32_t)a.rt_chunk);  // T < 2^31
                        if (a.rt_cls_stride > 0 && (uint32_t)mrow % (uint32_t)a.rt_cls_stride == 0)  // class token
                            orow = a.M - n_class_tokens(a.M, a.rt_cls_stride) + (uint32_t)mrow / (uint32_t)a.rt_cls_stride;
                        else if (e < a.rt_E)
                            orow = (int64_t)s_off[e] + s_tab[rc * a.rt_E + e] + (int)(w >> 8);
                        if ((uint64_t)orow >= (uint64_t)a.M) orow = -1;  // only a routing that gave up
                        if (orow >= 0 && t.n0 == 0 && c_lo == 0) a.rt_perm[orow] = (int32_t)mrow;  // once per token
                    } else {
                        orow = a.rows ? (int64_t)a.rows[mrow] : mrow;
                        if ((uint64_t)orow >= (uint64_t)a.M) orow = -1;  // only a routing that gave up
                    }
                }
                const float rsc = (a.group_scale && mrow < t.hi) ? tc_row_scale(a, mrow) : 1.f;
                // with the mean term in the accumulator (augmentation block) the bias add also scales by
                // rstd: fma(acc, 1, b) = acc + b exactly, so without the LayerNorm nothing changes
                const float lns = (a.ln_stats && !a.ln_colsum) ? ln.y : 1.f;
                const float2 lns2 = make_float2(lns, lns);
                // this lane stores warp rows 16 h + 8 p + lane / 4 (h, p < 2), 16-byte piece lane % 4 of
                // each 32-column chunk: their destinations, once per tile
                uint16_t* dst_row[4];
    #pragma unroll
                for (int hp = 0; hp < 4; ++hp) {
                    const int64_t o = __shfl_sync(0xffffffffu, orow, 8 * hp + lane / 4);
                    dst_row[hp] = o >= 0 ? static_cast<uint16_t*>(a.C) + o * a.ldc + t.n0 + (lane % 4) * 8 : nullptr;
                }
                for (int c = c_lo; c < c_hi; c += CW) {
                    uint32_t v[CW];
                    const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN + c;
                    CM_TMEM_LD_X16(taddr, v);
                    CM_TMEM_LD_X16(taddr + 16, (v + 16));
                    tmem_wait_ld();
                    float f[CW];
    #pragma unroll
                    for (int j = 0; j < CW; ++j) f[j] = __uint_as_float(v[j]);
                    const int nb = t.n0 + c;
                    if (a.ln_stats && a.ln_colsum) {  // W LN(y) = rstd (W y - mean c), c_n = sum_k W[n, k]
                        const float4* cp = reinterpret_cast<const float4*>(a.ln_colsum + nb);  // same for all lanes
    #pragma unroll
                        for (int j4 = 0; j4 < CW / 4; ++j4) {
                            const float4 c4 = __ldg(cp + j4);
                            f[4 * j4] = ln.y * fmaf(-ln.x, c4.x, f[4 * j4]);
                            f[4 * j4 + 1] = ln.y * fmaf(-ln.x, c4.y, f[4 * j4 + 1]);
                            f[4 * j4 + 2] = ln.y * fmaf(-ln.x, c4.z, f[4 * j4 + 2]);
                            f[4 * j4 + 3] = ln.y * fmaf(-ln.x, c4.w, f[4 * j4 + 3]);
                        }
                    }
                    if (a.epi == TC_EPI_BIAS_GELU) {
                        const float4* bp = reinterpret_cast<const float4*>(s_bias + nb);  // same for all lanes
    #pragma unroll
                        for (int j4 = 0; j4 < CW / 4; ++j4) {
                            const float4 b = bp[j4];
                            const float2 g0 = gelu_pair_as(
                                __ffma2_rn(make_float2(f[4 * j4], f[4 * j4 + 1]), lns2, make_float2(b.x, b.y)));
                            const float2 g1 = gelu_pair_as(
                                __ffma2_rn(make_float2(f[4 * j4 + 2], f[4 * j4 + 3]), lns2, make_float2(b.z, b.w)));
                            f[4 * j4] = g0.x;
                            f[4 * j4 + 1] = g0.y;
                            f[4 * j4 + 2] = g1.x;
                            f[4 * j4 + 3] = g1.y;
                        }
                    } else if (a.epi == TC_EPI_BIAS_RELU) {
                        const float4* bp = reinterpret_cast<const float4*>(s_bias + nb);  // same for all lanes
    #pragma unroll
                        for (int j4 = 0; j4 < CW / 4; ++j4) {
                            const float4 b = bp[j4];
                            f[4 * j4] = fmaxf(fmaf(f[4 * j4], lns, b.x), 0.f);
                            f[4 * j4 + 1] = fmaxf(fmaf(f[4 * j4 + 1], lns, b.y), 0.f);
                            f[4 * j4 + 2] = fmaxf(fmaf(f[4 * j4 + 2], lns, b.z), 0.f);
                            f[4 * j4 + 3] = fmaxf(fmaf(f[4 * j4 + 3], lns, b.w), 0.f);
                        }
                    } else if (a.out_bias) {
                        const float4* bp = reinterpret_cast<const float4*>(s_bias + nb);  // same for all lanes
    #pragma unroll
                        for (int j4 = 0; j4 < CW / 4; ++j4) {
                            const float4 b = bp[j4];
                            const float2 p0 = __fadd2_rn(make_float2(f[4 * j4], f[4 * j4 + 1]), make_float2(b.x, b.y));
                            const float2 p1 = __fadd2_rn(make_float2(f[4 * j4 + 2], f[4 * j4 + 3]), make_float2(b.z, b.w));
                            f[4 * j4] = p0.x;
                            f[4 * j4 + 1] = p0.y;
                            f[4 * j4 + 2] = p1.x;
                            f[4 * j4 + 3] = p1.y;
                        }
                    } else if (a.epi == TC_EPI_SCALE) {
                        const float4* sp = reinterpret_cast<const float4*>(s_bias + nb);  // same for all lanes
    #pragma unroll
                        for (int j4 = 0; j4 < CW / 4; ++j4) {
                            const float4 sc = sp[j4];
                            const float2 p0 = __fmul2_rn(make_float2(f[4 * j4], f[4 * j4 + 1]), make_float2(sc.x, sc.y));
                            const float2 p1 = __fmul2_rn(make_float2(f[4 * j4 + 2], f[4 * j4 + 3]), make_float2(sc.z, sc.w));
                            f[4 * j4] = p0.x;
                            f[4 * j4 + 1] = p0.y;
                            f[4 * j4 + 2] = p1.x;
                            f[4 * j4 + 3] = p1.y;
                        }
                    }
                    if (a.group_scale) {
    #pragma unroll
                        for (int j2 = 0; j2 < CW / 2; ++j2) {
                            const float2 p2 = __fmul2_rn(make_float2(f[2 * j2], f[2 * j2 + 1]), make_float2(rsc, rsc));
                            f[2 * j2] = p2.x;
                            f[2 * j2 + 1] = p2.y;
                        }
                    }
                    if (a.c_f32) {  // fp32 output: each lane stores its row's 32 values as computed
                        if (orow >= 0) {
                            float4* dstf = reinterpret_cast<float4*>(static_cast<float*>(a.C) + orow * a.ldc + nb);
    #pragma unroll
                            for (int j4 = 0; j4 < CW / 4; ++j4)
                                dstf[j4] = make_float4(f[4 * j4], f[4 * j4 + 1], f[4 * j4 + 2], f[4 * j4 + 3]);
                        }
                        continue;
                    }
    #pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        if ((lane >> 4) == h) {
                            const int rw = lane & 15;
                            unsigned char* dst = wstg + rw * 64;
    #pragma unroll
                            for (int j8 = 0; j8 < 4; ++j8) {
                                const float* g = f + 8 * j8;
                                *reinterpret_cast<uint4*>(dst + ((j8 ^ ((rw >> 1) & 3)) << 4)) =
                                    make_uint4(pack_bf16(g[0], g[1]), pack_bf16(g[2], g[3]), pack_bf16(g[4], g[5]),
                                               pack_bf16(g[6], g[7]));
                            }
                        }
                        __syncwarp();
    #pragma unroll
                        for (int p = 0; p < 2; ++p) {
                            const int rr = 8 * p + lane / 4;  // row of the half
                            const int ch = (lane % 4) ^ ((rr >> 1) & 3);
                            const uint4 val = *reinterpret_cast<const uint4*>(wstg + rr * 64 + ch * 16);
                            if (dst_row[2 * h + p]) *reinterpret_cast<uint4*>(dst_row[2 * h + p] + c) = val;
                        }
                        __syncwarp();
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(tempty_leader0 + 8u * acc);  // the even CTA's tempty
            if (++acc == nacc) {
                acc = 0;
                aph ^= 1;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync();  // no copy, commit or remote arrival is left in flight towards either CTA
    tc_fence_after();
    if (warp == WARP_MMA)
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS)
                     : "memory");
}

int tc2_pick_bn(int mode, int N) {
    if (mode != TC_DENSE && mode != TC_GROUPED) return 0;
    if (N % 256 == 0) return 256;
    if (N % 192 == 0) return 192;  // e.g. d = 384: two 192-wide tiles instead of three 128-wide ones
    if (N % 128 == 0) return 128;
    return 0;
}

template <int BN, int MODE, int VAR>
static cudaError_t launch2(const TcGemmArgs& a, int num_sms, cudaStream_t s) {
    using C = T2v<BN, VAR>;
    const void* fn = (const void*)tc_gemm2_kernel<BN, MODE, VAR>;
    const cudaError_t e = smem_attr_once(fn, C::SMEM);
    if (e != cudaSuccess) return e;
    const int n_tiles = a.N / BN;
    int64_t m_pairs = (a.M + 2 * C::BM - 1) / (2 * C::BM);
    if (a.mode == TC_GROUPED) m_pairs += a.E;
    const int64_t units = m_pairs * (n_tiles + (VAR == TC2_ROUTER ? 1 : 0));
    int64_t clusters = units < num_sms / 2 ? units : num_sms / 2;
    if (clusters <= 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * clusters));
    cfg.blockDim = dim3(C::THREADS);
    cfg.dynamicSmemBytes = C::SMEM;
    cfg.stream = s;
    cudaLaunchAttribute attr_pdl[1];
    attr_pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr_pdl[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr_pdl;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, tc_gemm2_kernel<BN, MODE, VAR>, a);
}

template <int BN>
static cudaError_t launch2_var(const TcGemmArgs& a, int num_sms, cudaStream_t s) {
    if (a.mode == TC_GROUPED)
        return a.a1_rows ? launch2<BN, TC_GROUPED, TC2_GATHER>(a, num_sms, s) : launch2<BN, TC_GROUPED, TC2_PLAIN>(a, num_sms, s);
    if constexpr (BN == 256) {
        if (a.epi12) return launch2<BN, TC_DENSE, TC2_EPI12>(a, num_sms, s);
    }
    return a.fr_E > 0 ? launch2<BN, TC_DENSE, TC2_ROUTER>(a, num_sms, s) : launch2<BN, TC_DENSE, TC2_PLAIN>(a, num_sms, s);
}

cudaError_t launch_tc_gemm2(const TcGemmArgs& a, int num_sms, cudaStream_t s) {
    const int bn = tc2_pick_bn(a.mode, a.N);
    const bool staged = a.epi == TC_EPI_BIAS_GELU || a.epi == TC_EPI_BIAS_RELU ||
                        a.epi == TC_EPI_SCALE;  // fp32 vector in shared memory
    if (!bn || (staged && (a.mode != TC_DENSE || a.N > TC2_BIAS_CAP))) return cudaErrorInvalidValue;
    if (a.out_bias && (staged || a.N > TC2_BIAS_CAP)) return cudaErrorInvalidValue;
    // the LayerNorm fold: the augmentation block only ahead of a bias epilogue, and with the
    // statistics but no column sums only together with it
    const bool bias_epi = a.epi == TC_EPI_BIAS_GELU || a.epi == TC_EPI_BIAS_RELU;
    if (a.ln_aug && (a.mode != TC_DENSE || !bias_epi || !a.ln_stats || a.ln_colsum)) return cudaErrorInvalidValue;
    if (a.ln_stats && !a.ln_colsum && !a.ln_aug) return cudaErrorInvalidValue;
    // the router inside fc1: dense mode, fc1's own epilogue, token order, none of the other row maps
    if (a.fr_E > 0 && (a.mode != TC_DENSE || a.fr_E > CM_MAX_E || a.epi != TC_EPI_BIAS_GELU || a.ln_aug ||
                       a.ln_stats || a.rt_info || a.rows || a.c_f32 || a.group_scale || !a.fr_bias || !a.fr_idx ||
                       !a.fr_info || !a.fr_counts))
        return cudaErrorInvalidValue;
    if (a.a1_rows && a.mode != TC_GROUPED) return cudaErrorInvalidValue;
    // twelve epilogue warps: the plain dense GEMM at 256-wide tiles (short-K fc1)
    if (a.epi12 && (a.mode != TC_DENSE || bn != 256 || a.fr_E > 0)) return cudaErrorInvalidValue;
    if (bn == 256) return launch2_var<256>(a, num_sms, s);
    if (bn == 192) return launch2_var<192>(a, num_sms, s);
    return launch2_var<128>(a, num_sms, s);
}

}  // namespace cm
