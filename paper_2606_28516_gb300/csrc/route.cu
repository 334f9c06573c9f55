// Routing of the CLEAR-MoE FFN (Algorithm 3, steps 3-4):
//   logits = W_g x + b_g (linear router), a = argmax (lowest index on ties),
//   per-expert histogram, exclusive prefix sum, and the stable permutation perm[slot] = token.
//
// route_kernel: CTA b owns a contiguous range of `chunk` tokens and never waits for another CTA.
//   phase 1: stream x once from HBM, router logits and argmax per token, the range's histogram.
//            bf16: one CTA per SM; a producer thread copies the CTA's rows, 16 at a time, into a
//            ring of shared-memory stages with 1-D bulk copies (mbarrier-tracked, so the bytes in
//            flight cost no registers) and eight consumer warps take one 16-row stage each;
//   then:    the histogram row goes to cta_counts, and each token's rank among the range's
//            earlier tokens of its expert (warp match masks) to tinfo, packed with the expert.
// The slot of token t in range c is offsets[e] + (tokens of e in ranges before c) + its rank, in
// token order within each expert, which makes the sort stable. It is formed by the consumer of
// the routing: the fc1 epilogue of the 2-SM GEMM (which then stores z rows at their slots and
// writes perm), or route_finalize_kernel (perm and inv ahead of the other paths).
// bf16 tokens: the d x E contraction runs on the legacy warp MMA (m16n8k16, fp32 accumulate):
// x fragments from the shared-memory stage, W_g fragments staged once in shared memory (reading
// them through L1 in the inner loop was measured slower), and the K order of each fragment is
// permuted identically for x and W_g, which leaves every dot product unchanged.
// fp32 tokens: fp32 FMA on the CUDA cores (an fp32 router decision needs fp32 products).
// Class tokens (cls_stride > 0, t % cls_stride == 0) skip the router: idx = E, no histogram entry
// and no rank; their slots T - n_cls + t / cls_stride follow the experts' (the dense path).
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace cm {

constexpr int RT_THREADS = 256;                 // fp32 router: 8 warps
constexpr int RT_BF16_THREADS = 288;            // bf16 router: 8 consumer warps + 1 producer warp
constexpr int RT_MAX_WARPS = RT_BF16_THREADS / 32;
constexpr int RT_STAGE_ROWS = 16;               // rows per ring stage (one MMA row group)

__device__ __forceinline__ uint4 ldg_nc_v4(const uint4* p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// better (value, index) with the lower index winning exact ties
__device__ __forceinline__ void arg_better(float& bv, int& be, float v, int e) {
    if (v > bv || (v == bv && e < be)) {
        bv = v;
        be = e;
    }
}

// bf16: W_g rows in shared memory with a 64-byte pad, so that the 16-byte B-fragment reads of a
// quarter warp (two rows, four 16-byte column groups each) hit all 32 banks once. Token stages
// stay contiguous (one bulk copy per 16 rows, 2-way conflicts on the A-fragment reads): neither
// per-row copies into padded rows nor a 128-byte-swizzled tensor copy was measured faster.
__host__ __device__ inline int wrow_bytes(int d) { return d * 2 + 64; }
__host__ __device__ inline size_t frag_bytes(int dtype, int d, int E) {
    if (dtype == CLEARMOE_BF16) return (size_t)E * wrow_bytes(d);
    return (size_t)E * d * 4;
}

// Dynamic shared memory: [router weights] [bf16: ring of S stages] [bf16: 2 S + 1 mbarriers]
// [per-row word: expert | local rank << 8, when chunk words fit; else that word lives in idx in
// global memory (the CTA's own rows, visible block-wide after __syncthreads) until phase 2
// rewrites idx with the expert alone], so the footprint does not grow with T.
// The ring has one slot per consumer warp (S = 8, or 4 when eight stages do not fit): consumer
// warp w alone reads slot w, for stages w, w + S, ..., so each of its mbarrier waits is for the
// phase right after the one it last consumed (a parity wait cannot tell phases two apart).
constexpr size_t RT_SMEM_MAX = 220 * 1024;
struct RouteLayout {
    size_t ring, bars, sidx, scnt, total;
    int S, stage_bytes;
    bool sidx_in_smem;
};
__host__ __device__ inline RouteLayout route_layout(int dtype, int d, int E, int chunk) {
    RouteLayout L;
    const size_t frag = (frag_bytes(dtype, d, E) + 127) & ~(size_t)127;
    L.stage_bytes = RT_STAGE_ROWS * d * 2;
    L.S = 0;
    L.ring = frag;
    if (dtype == CLEARMOE_BF16)  // eight slots when they fit beside W_g and the barriers, else four
        L.S = (L.ring + 8 * (size_t)L.stage_bytes + 17 * 8 <= RT_SMEM_MAX) ? 8 : 4;
    L.bars = (L.ring + (size_t)L.S * L.stage_bytes + 15) & ~(size_t)15;
    L.sidx = L.bars + (size_t)(2 * L.S + 1) * 8;  // bf16: ring barriers + the W_g barrier
    // expert ids of the CTA's rows: in shared memory when they fit, else read back from idx
    // per row a 4-byte word; bf16 also keeps each 16-row stage's per-expert counts (2 bytes each)
    const size_t rows_bytes =
        (size_t)chunk * 4 + (dtype == CLEARMOE_BF16 ? (size_t)((chunk + 15) / 16) * CM_MAX_E * 2 : 0);
    L.scnt = L.sidx + (size_t)chunk * 4;
    L.sidx_in_smem = L.sidx + rows_bytes <= RT_SMEM_MAX;
    L.total = L.sidx + (L.sidx_in_smem ? rows_bytes : 0);
    return L;
}
static size_t route_smem(int dtype, int d, int E, int chunk) { return route_layout(dtype, d, E, chunk).total; }

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

// W_g's B fragments held in registers (bf16, E <= 8, d <= RT_WREG_D): 4 registers per 32 columns
constexpr int RT_WREG_D = 768;
inline bool route_wreg(int dtype, int d, int E) { return dtype == CLEARMOE_BF16 && E <= 8 && d <= RT_WREG_D; }

template <bool BF16, bool WREG>
__global__ void __launch_bounds__(BF16 ? RT_BF16_THREADS : RT_THREADS) route_kernel(const RouteArgs a, const int chunk) {
    constexpr int NTHREADS = BF16 ? RT_BF16_THREADS : RT_THREADS;
    constexpr int NWARPS = NTHREADS / 32;
    constexpr int NCONS_MAX = 8;  // warps computing logits (bf16: the first S warps)
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ int s_count[CM_MAX_E];
    __shared__ int s_run[CM_MAX_E];
    __shared__ int s_wc[RT_MAX_WARPS][CM_MAX_E];
    __shared__ int s_abort;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int E = a.E, d = a.d;
    const int64_t row0 = (int64_t)blockIdx.x * chunk;
    const int nrows = (int)max((int64_t)0, min((int64_t)chunk, a.T - row0));
    const int nchunk = d / 32;
    const int NT = (E + 7) / 8;
    const RouteLayout lay = route_layout(BF16 ? CLEARMOE_BF16 : CLEARMOE_F32, d, E, chunk);
    // per-row expert after phase 1: in shared memory when it fits, else read back from idx
    uint32_t* sinfo = lay.sidx_in_smem ? reinterpret_cast<uint32_t*>(smem + lay.sidx) : nullptr;
    auto info_of = [&](int i) -> uint32_t { return sinfo ? sinfo[i] : (uint32_t)__ldcg(a.idx + row0 + i); };
    // bf16 with the words in shared memory: ranks within 16-row stages during phase 1 (scnt holds
    // each stage's per-expert counts), so that only a scan over stages remains afterwards
    uint16_t* scnt = (BF16 && sinfo) ? reinterpret_cast<uint16_t*>(smem + lay.scnt) : nullptr;
    auto record = [&](int i, int e, int rank) {  // phase 1 result of row i: idx, its word, histogram
        a.idx[row0 + i] = e;
        if (sinfo) sinfo[i] = (uint32_t)e | ((uint32_t)rank << 8);
        if (e < E) atomicAdd(&s_count[e], 1);  // e == E: a class token
    };

    if (tid < CM_MAX_E) s_count[tid] = 0;
    if (tid == 0) s_abort = 0;

    // ---------------- phase 1: router logits + argmax for this CTA's rows
    if constexpr (BF16) {
        const int S = lay.S, SB = lay.stage_bytes;
        const uint32_t ring = smem_u32(smem + lay.ring);
        const uint32_t bar0 = smem_u32(smem + lay.bars);
        auto full_bar = [&](int s) { return bar0 + 8u * s; };
        auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
        const int nstages = (nrows + RT_STAGE_ROWS - 1) / RT_STAGE_ROWS;
        volatile int* abort_flag = &s_abort;
        // ---- producer: stage k = rows [16 k, 16 k + 16) of this CTA, ring slot k % S. Its thread
        // initialises the barriers, copies W_g's rows into shared memory (first in its queue, on
        // their own barrier) and then streams the stages.
        const bool producer = tid == NCONS_MAX * 32;
        const uint32_t wbar = bar0 + 8u * (2 * S);
        const int WRB = wrow_bytes(d);
        if (producer) {
            for (int s = 0; s < S; ++s) {
                mbar_init(full_bar(s), 1);
                mbar_init(empty_bar(s), 1);
            }
            mbar_init(wbar, 1);
            mbar_fence_init();
        }
        __syncthreads();  // barriers initialised
        if (producer) {
            mbar_arrive_expect_tx(wbar, (uint32_t)E * d * 2);
            const unsigned char* Wb = static_cast<const unsigned char*>(a.Wg);
            for (int e = 0; e < E; ++e) bulk_g2s(smem_u32(smem) + e * WRB, Wb + (size_t)e * d * 2, d * 2, wbar);
        }
        pdl_wait();  // from here on the previous kernel's results (x) are read and outputs written
        // the next kernel may start now (its CTAs set up, and may read x, while this one streams):
        // released only after the wait, so every kernel before this one has completed by then
        pdl_launch_dependents();
        if (warp == NCONS_MAX) {
            if (producer) {
                const unsigned char* xb = static_cast<const unsigned char*>(a.x) + row0 * d * 2;
                int k = 0;
                for (; k < nstages; ++k) {
                    const int s = k % S;
                    if (!mbar_wait(empty_bar(s), ((k / S) & 1) ^ 1, abort_flag, a.status, (uint64_t)a.wait_limit_ns))
                        break;
                    if (k == a.debug_skip && blockIdx.x == 0) continue;  // fault injection: withhold a stage
                    const int rows = min(RT_STAGE_ROWS, nrows - k * RT_STAGE_ROWS);
                    const uint32_t bytes = (uint32_t)rows * d * 2;
                    mbar_arrive_expect_tx(full_bar(s), bytes);
                    bulk_g2s(ring + s * SB, xb + (size_t)k * SB, bytes, full_bar(s));
                }
                if (k < nstages) {  // gave up: let the copies in flight land before moving on
                    for (int j = max(0, k - S); j < k; ++j)
                        mbar_wait(full_bar(j % S), (j / S) & 1, nullptr, a.status, 10000000ull);
                }
                mbar_wait(wbar, 0, nullptr, a.status, 10000000ull);  // W_g's rows have landed too
            }
        } else if (warp < S) {
            // ---- consumers: warp w owns slot w and takes stages w, w + S, w + 2 S, ...
            const uint16_t* bgp = static_cast<const uint16_t*>(a.bg);
            const int g = lane >> 2, tig = lane & 3;
            const uint4 zero = make_uint4(0, 0, 0, 0);
            // B fragment of n-tile nt, 32-column chunk c: 8 consecutive bf16 of W_g row nt*8 + g,
            // columns c*32 + tig*8 (rows past E are zero)
            const uint4* wfr[2];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
                wfr[nt] = (nt < NT && nt * 8 + g < E)
                              ? reinterpret_cast<const uint4*>(smem + (size_t)(nt * 8 + g) * WRB + tig * 16)
                              : nullptr;
            const bool w_ok = nstages == 0 || mbar_wait(wbar, 0, abort_flag, a.status, (uint64_t)a.wait_limit_ns);
            constexpr int NWC = WREG ? RT_WREG_D / 32 : 1;  // register copy of the fragments (WREG)
            uint4 wreg[NWC];
            if constexpr (WREG) {
#pragma unroll
                for (int c = 0; c < NWC; ++c) wreg[c] = (c < nchunk && wfr[0] && w_ok) ? wfr[0][4 * c] : zero;
            }
            for (int k = warp; w_ok && k < nstages; k += S) {
                const int s = warp;
                if (!mbar_wait(full_bar(s), (k / S) & 1, abort_flag, a.status, (uint64_t)a.wait_limit_ns)) break;
                const int rows = min(RT_STAGE_ROWS, nrows - k * RT_STAGE_ROWS);
                const bool vA = g < rows, vB = g + 8 < rows;
                const unsigned char* st = smem + lay.ring + (size_t)s * SB;
                const uint4* pA = reinterpret_cast<const uint4*>(st + (size_t)g * d * 2) + tig;
                const uint4* pB = reinterpret_cast<const uint4*>(st + (size_t)(g + 8) * d * 2) + tig;
                // four independent accumulator chains (K steps 4j + q go to chain q), summed at the end
                float part[2][4][4];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int q = 0; q < 4; ++q)
#pragma unroll
                        for (int i = 0; i < 4; ++i) part[nt][q][i] = 0.f;
                if constexpr (WREG) {
#pragma unroll
                    for (int c = 0; c < NWC; c += 2) {  // one n-tile, fragments in registers
                        if (c < nchunk) {
                            const uint4 xa0 = vA ? pA[4 * c] : zero, xa1 = vA ? pA[4 * c + 4] : zero;
                            const uint4 xb0 = vB ? pB[4 * c] : zero, xb1 = vB ? pB[4 * c + 4] : zero;
                            const uint4 w0 = wreg[c], w1 = wreg[c + 1];
                            mma_bf16_16816(part[0][0], xa0.x, xb0.x, xa0.y, xb0.y, w0.x, w0.y);
                            mma_bf16_16816(part[0][1], xa0.z, xb0.z, xa0.w, xb0.w, w0.z, w0.w);
                            mma_bf16_16816(part[0][2], xa1.x, xb1.x, xa1.y, xb1.y, w1.x, w1.y);
                            mma_bf16_16816(part[0][3], xa1.z, xb1.z, xa1.w, xb1.w, w1.z, w1.w);
                        }
                    }
                } else {
                    for (int c = 0; c < nchunk; c += 2) {  // d % 64 == 0: nchunk is even
                        const uint4 xa0 = vA ? pA[4 * c] : zero, xa1 = vA ? pA[4 * c + 4] : zero;
                        const uint4 xb0 = vB ? pB[4 * c] : zero, xb1 = vB ? pB[4 * c + 4] : zero;
#pragma unroll
                        for (int nt = 0; nt < 2; ++nt) {
                            if (nt < NT) {
                                const uint4 w0 = wfr[nt] ? wfr[nt][4 * c] : zero;
                                const uint4 w1 = wfr[nt] ? wfr[nt][4 * c + 4] : zero;
                                mma_bf16_16816(part[nt][0], xa0.x, xb0.x, xa0.y, xb0.y, w0.x, w0.y);
                                mma_bf16_16816(part[nt][1], xa0.z, xb0.z, xa0.w, xb0.w, w0.z, w0.w);
                                mma_bf16_16816(part[nt][2], xa1.x, xb1.x, xa1.y, xb1.y, w1.x, w1.y);
                                mma_bf16_16816(part[nt][3], xa1.z, xb1.z, xa1.w, xb1.w, w1.z, w1.w);
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(empty_bar(s));  // the stage is no longer read
                float acc[2][4];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        acc[nt][i] = (part[nt][0][i] + part[nt][1][i]) + (part[nt][2][i] + part[nt][3][i]);
                // D fragment: acc[nt][0..1] = row g, experts nt*8 + 2*tig + {0,1}; [2..3] = row g+8
                float2 lnA = make_float2(0.f, 1.f), lnB = make_float2(0.f, 1.f);  // (mean, rstd)
                if (a.ln_stats) {
                    const int64_t tA = row0 + (int64_t)k * RT_STAGE_ROWS + g;
                    if (vA) lnA = a.ln_stats[tA];
                    if (vB) lnB = a.ln_stats[tA + 8];
                }
                float bA = -INFINITY, bB = -INFINITY;
                int eA = 0x7fffffff, eB = 0x7fffffff;
#pragma unroll
                for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        const int e = nt * 8 + 2 * tig + j;
                        if (nt < NT && e < E) {
                            const uint16_t bb = bgp[e];
                            const float bias = __uint_as_float((uint32_t)bb << 16);
                            float lA = acc[nt][j], lB = acc[nt][2 + j];
                            if (a.ln_stats) {  // W_g LN(y) = rstd (W_g y - mean g)
                                const float ge = a.ln_wsum[e];
                                lA = lnA.y * fmaf(-lnA.x, ge, lA);
                                lB = lnB.y * fmaf(-lnB.x, ge, lB);
                            }
                            arg_better(bA, eA, lA + bias, e);
                            arg_better(bB, eB, lB + bias, e);
                        }
                    }
                }
#pragma unroll
                for (int off = 1; off <= 2; off <<= 1) {
                    const float ovA = __shfl_xor_sync(0xffffffffu, bA, off);
                    const int oeA = __shfl_xor_sync(0xffffffffu, eA, off);
                    const float ovB = __shfl_xor_sync(0xffffffffu, bB, off);
                    const int oeB = __shfl_xor_sync(0xffffffffu, eB, off);
                    arg_better(bA, eA, ovA, oeA);
                    arg_better(bB, eB, ovB, oeB);
                }
                if (eA > E - 1) eA = 0;  // only reachable with non-finite logits
                if (eB > E - 1) eB = 0;
                if (a.cls_stride > 0) {  // class tokens: group E, outside every expert's ballot
                    const int64_t tA = row0 + (int64_t)k * RT_STAGE_ROWS + g;
                    if (tA % a.cls_stride == 0) eA = E;
                    if ((tA + 8) % a.cls_stride == 0) eB = E;
                }
                int rankA = 0, rankB = 0;
                if (scnt) {
                    // rank of each row among the stage's earlier rows of its expert, from one ballot
                    // per expert over the lanes holding rows 0-7 (eA) and rows 8-15 (eB)
                    unsigned selAA = 0, selBA = 0, selBB = 0;
                    for (int e = 0; e < E; ++e) {
                        const unsigned mA = __ballot_sync(0xffffffffu, tig == 0 && vA && eA == e);
                        const unsigned mB = __ballot_sync(0xffffffffu, tig == 0 && vB && eB == e);
                        if (eA == e) selAA = mA;
                        if (eB == e) {
                            selBA = mA;
                            selBB = mB;
                        }
                        if (lane == 0) scnt[k * CM_MAX_E + e] = (uint16_t)(__popc(mA) + __popc(mB));
                    }
                    const unsigned below = (1u << (4 * g)) - 1u;  // lanes of rows before row g
                    rankA = __popc(selAA & below);
                    rankB = __popc(selBA) + __popc(selBB & below);
                }
                if (tig == 0) {
                    const int iA = k * RT_STAGE_ROWS + g, iB = iA + 8;
                    if (vA) record(iA, eA, rankA);
                    if (vB) record(iB, eB, rankB);
                }
            }
        }
    } else {
        float* Wf = reinterpret_cast<float*>(smem);
        if (a.w_bf16) {  // bf16 router weights on fp32 tokens: widened exactly
            const uint16_t* W = static_cast<const uint16_t*>(a.Wg);
            for (int i = tid; i < E * d; i += NTHREADS) Wf[i] = bf16_to_f32(W[i]);
        } else {
            const float* W = static_cast<const float*>(a.Wg);
            for (int i = tid; i < E * d; i += NTHREADS) Wf[i] = W[i];
        }
        pdl_wait();
        pdl_launch_dependents();
        __syncthreads();
        auto bias_of = [&](int e) -> float {
            return a.w_bf16 ? bf16_to_f32(static_cast<const uint16_t*>(a.bg)[e]) : static_cast<const float*>(a.bg)[e];
        };
        // one row per lane: each lane streams its row in 16-float chunks (float4 loads; the L1
        // merges the 32 rows' sectors) against W_g broadcast from shared memory, fp32 FMA in k
        // order, so a warp routes 32 rows with no cross-lane reduction (d % 4 == 0)
        const float* X = static_cast<const float*>(a.x);
        for (int b0 = warp * 32; b0 < nrows; b0 += NWARPS * 32) {
            const int i = b0 + lane;
            const bool valid = i < nrows;
            const float4* xr = reinterpret_cast<const float4*>(X + (row0 + (valid ? i : 0)) * d);
            float acc[CM_MAX_E];
#pragma unroll
            for (int e = 0; e < CM_MAX_E; ++e) acc[e] = 0.f;
            for (int k4 = 0; k4 < d / 4; k4 += 4) {
                float4 xv[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) xv[j] = (k4 + j < d / 4) ? xr[k4 + j] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    if (k4 + j < d / 4) {
#pragma unroll
                        for (int e = 0; e < CM_MAX_E; ++e) {
                            if (e < E) {
                                const float4 w = reinterpret_cast<const float4*>(Wf + (size_t)e * d)[k4 + j];
                                acc[e] = fmaf(xv[j].x, w.x, acc[e]);
                                acc[e] = fmaf(xv[j].y, w.y, acc[e]);
                                acc[e] = fmaf(xv[j].z, w.z, acc[e]);
                                acc[e] = fmaf(xv[j].w, w.w, acc[e]);
                            }
                        }
                    }
                }
            }
            if (a.ln_stats) {  // W_g LN(y) = rstd (W_g y - mean g)
                const float2 st = valid ? a.ln_stats[row0 + i] : make_float2(0.f, 1.f);
#pragma unroll
                for (int e = 0; e < CM_MAX_E; ++e)
                    if (e < E) acc[e] = st.y * fmaf(-st.x, a.ln_wsum[e], acc[e]);
            }
            float bv = -INFINITY;
            int be = 0x7fffffff;
#pragma unroll
            for (int e = 0; e < CM_MAX_E; ++e)
                if (e < E) arg_better(bv, be, acc[e] + bias_of(e), e);
            if (be > E - 1) be = 0;  // only reachable with non-finite logits
            if (a.cls_stride > 0 && (row0 + i) % a.cls_stride == 0) be = E;  // a class token
            if (valid) record(i, be, 0);
        }
    }
    __syncthreads();

    // ---------------- this CTA's histogram, and each row's rank among the CTA's earlier rows of
    // its expert (warp match masks, then a per-expert prefix over warps and over passes), which
    // makes the final order stable. The slots themselves are assigned by the consumer of the
    // routing (the fc1 epilogue, or route_finalize_kernel): no CTA ever waits for another.
    if (tid < E) a.cta_counts[(size_t)blockIdx.x * CM_MAX_E + tid] = s_count[tid];
    if (scnt) {
        // per expert, an exclusive scan of the stage counts (one warp per expert, 32 stages a
        // step), then rank = the stage's prefix + the rank within the stage
        const int nst = (nrows + RT_STAGE_ROWS - 1) / RT_STAGE_ROWS;
        for (int e = warp; e < E; e += NWARPS) {
            int carry = 0;
            for (int k0 = 0; k0 < nst; k0 += 32) {
                const int k = k0 + lane;
                const int v = k < nst ? scnt[k * CM_MAX_E + e] : 0;
                int incl = v;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const int o = __shfl_up_sync(0xffffffffu, incl, off);
                    if (lane >= off) incl += o;
                }
                if (k < nst) scnt[k * CM_MAX_E + e] = (uint16_t)(carry + incl - v);
                carry += __shfl_sync(0xffffffffu, incl, 31);
            }
        }
        __syncthreads();
        for (int i = tid; i < nrows; i += NTHREADS) {
            const uint32_t w = sinfo[i];
            const int e = (int)(w & 0xffu);
            // class tokens (e == E) and rows a launch that gave up never routed take no slot here
            a.tinfo[row0 + i] =
                e < E ? e | ((scnt[(i / RT_STAGE_ROWS) * CM_MAX_E + e] + (int)((w >> 8) & 0xffu)) << 8) : E;
        }
        return;
    }
    const unsigned lt = (1u << lane) - 1u;
    if (tid < CM_MAX_E) s_run[tid] = 0;
    for (int i0 = 0; i0 < nrows; i0 += NTHREADS) {
        if (tid < NWARPS * CM_MAX_E) (&s_wc[0][0])[tid] = 0;
        __syncthreads();
        const int i = i0 + tid;
        const bool valid = i < nrows;
        int e = valid ? (int)(info_of(i) & 0xffu) : CM_MAX_E + 1;
        // class tokens (e == E) and rows a launch that gave up never routed take no rank
        const bool ranked = valid && e < E;
        if (!ranked) e = CM_MAX_E + 1;
        const unsigned same = __match_any_sync(0xffffffffu, e);
        const int rank = __popc(same & lt);
        if (ranked && rank == 0) s_wc[warp][e] = __popc(same);
        __syncthreads();
        int pre = 0, own = 0;  // lane l < E: expert l's rows in this CTA before this warp's rows
        if (lane < E) {
            pre = s_run[lane];
            for (int w = 0; w < warp; ++w) pre += s_wc[w][lane];
            own = s_wc[warp][lane];
        }
        const int base_e = __shfl_sync(0xffffffffu, pre, ranked ? e : 0);
        if (ranked)
            a.tinfo[row0 + i] = e | ((base_e + rank) << 8);
        else if (valid)
            a.tinfo[row0 + i] = E;
        __syncthreads();  // every warp has read s_run and s_wc
        if (warp == NWARPS - 1 && lane < E) s_run[lane] = pre + own;
    }
}

// Slots of one routing range (the same ranges as route_kernel: CTA b owns rows [b chunk, +chunk)):
// the per-expert sums of the G ranges' histograms before this one and over all (thread b reads row
// b), offsets by a scan over experts, then slot = offsets[e] + before + local rank for every row.
// Writes perm, inv (if set), counts and offsets (range 0), and unpacks idx when it carried the
// packed words. Class tokens take slot T - n_cls + t / cls_stride; counts[E] = n_cls and
// offsets[E + 1] = T then describe their group.
__global__ void __launch_bounds__(256) route_finalize_kernel(const RouteArgs a, const int chunk, const int G) {
    __shared__ int s_wb[8][CM_MAX_E], s_wt[8][CM_MAX_E], s_base[CM_MAX_E];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, E = a.E;
    const int64_t row0 = (int64_t)blockIdx.x * chunk;
    const int nrows = (int)max((int64_t)0, min((int64_t)chunk, a.T - row0));
    const int64_t n_cls = n_class_tokens(a.T, a.cls_stride);
    pdl_wait();  // everything below reads the routing kernel's output
    pdl_launch_dependents();
    int bef[CM_MAX_E], tot[CM_MAX_E];
#pragma unroll
    for (int e = 0; e < CM_MAX_E; ++e) bef[e] = tot[e] = 0;
    for (int b = tid; b < G; b += 256) {
        const int4* row = reinterpret_cast<const int4*>(a.cta_counts + (size_t)b * CM_MAX_E);
#pragma unroll
        for (int q = 0; q < CM_MAX_E / 4; ++q) {
            if (4 * q < E) {
                const int4 v = __ldcg(row + q);
                const int c4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    tot[4 * q + j] += c4[j];
                    if (b < (int)blockIdx.x) bef[4 * q + j] += c4[j];
                }
            }
        }
    }
#pragma unroll
    for (int e = 0; e < CM_MAX_E; ++e) {
        if (e < E) {
            const int vb = __reduce_add_sync(0xffffffffu, bef[e]);
            const int vt = __reduce_add_sync(0xffffffffu, tot[e]);
            if (lane == 0) {
                s_wb[warp][e] = vb;
                s_wt[warp][e] = vt;
            }
        }
    }
    __syncthreads();
    if (warp == 0) {
        int b = 0, t = 0;
        if (lane < E)
            for (int w = 0; w < 8; ++w) {
                b += s_wb[w][lane];
                t += s_wt[w][lane];
            }
        int incl = t;  // inclusive scan of the totals over experts (lanes)
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += v;
        }
        if (lane < E) {
            s_base[lane] = incl - t + b;
            if (blockIdx.x == 0) {
                a.counts[lane] = t;
                a.offsets[lane] = incl - t;
                if (lane == E - 1) {
                    a.offsets[E] = incl;
                    if (n_cls > 0) {  // the dense path's group
                        a.counts[E] = (int32_t)n_cls;
                        a.offsets[E + 1] = incl + (int32_t)n_cls;
                    }
                }
            }
        }
    }
    __syncthreads();
    const bool unpack = a.tinfo == a.idx;
    for (int i = tid; i < nrows; i += 256) {
        const int64_t tok = row0 + i;
        if (a.cls_stride > 0 && tok % a.cls_stride == 0) {  // a class token: the dense path's slots
            const int64_t slot = a.T - n_cls + tok / a.cls_stride;
            a.perm[slot] = (int32_t)tok;
            if (a.inv) a.inv[tok] = (int32_t)slot;
            if (unpack) a.idx[tok] = E;
            continue;
        }
        const uint32_t w = (uint32_t)a.tinfo[row0 + i];
        const int e = (int)(w & 0xffu);
        if (e >= E) continue;  // only a routing launch that gave up leaves such words
        const int64_t slot = (int64_t)s_base[e] + (int)(w >> 8);
        if (slot >= a.T) continue;
        a.perm[slot] = (int32_t)(row0 + i);
        if (a.inv) a.inv[row0 + i] = (int32_t)slot;
        if (unpack) a.idx[row0 + i] = e;
    }
}

// At most 32 rows of the histogram exchange per thread (a 32-bit mask of rows read).
int route_max_ctas(int num_sms, int, int, int) { return min(num_sms * 8, 32 * RT_THREADS); }

int route_grid(int64_t T, int d, int E, int dtype, int num_sms, int* grid, int* chunk) {
    const bool bf16 = dtype == CLEARMOE_BF16;
    int occ = 0;
    int64_t want = (int64_t)num_sms * (bf16 ? 1 : 2);  // bf16: one CTA per SM owns the ring
    // equal ranges over all CTAs (a range's last 16-row stage may be partial)
    int64_t ch = (T + want - 1) / want;
    // the shared-memory attribute belongs to a device: set once per device
    if (smem_attr_once((const void*)route_kernel<true, false>, (int)RT_SMEM_MAX) != cudaSuccess ||
        smem_attr_once((const void*)route_kernel<true, true>, (int)RT_SMEM_MAX) != cudaSuccess ||
        smem_attr_once((const void*)route_kernel<false, false>, (int)RT_SMEM_MAX) != cudaSuccess) {
        (void)cudaGetLastError();
        return -1;
    }
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return -1;
    }
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    // occupancy queries are cached: (device, dtype, d, E, shared-memory bytes) -> CTAs per SM
    static struct { int dev, dtype, d, E; size_t smem; int occ; } cache[64];
    static int ncache = 0;
    for (int iter = 0; iter < 4; ++iter) {
        const size_t smem = route_smem(dtype, d, E, (int)ch);
        occ = -1;
        for (int i = 0; i < ncache; ++i)
            if (cache[i].dev == dev && cache[i].dtype == dtype && cache[i].d == d && cache[i].E == E &&
                cache[i].smem == smem)
                occ = cache[i].occ;
        if (occ < 0) {
            const void* fn = !bf16 ? (const void*)route_kernel<false, false>
                             : route_wreg(dtype, d, E) ? (const void*)route_kernel<true, true>
                                                       : (const void*)route_kernel<true, false>;
            cudaError_t err = cudaOccupancyMaxActiveBlocksPerMultiprocessorWithFlags(
                &occ, fn, bf16 ? RT_BF16_THREADS : RT_THREADS, smem, cudaOccupancyDefault);
            if (err != cudaSuccess) return -1;
            if (ncache < 64) cache[ncache++] = {dev, dtype, d, E, smem, occ};
        }
        if (occ <= 0) return -2;
        const int64_t maxg = (int64_t)occ * num_sms;
        if (want <= maxg) break;
        want = maxg;
        ch = (T + want - 1) / want;
    }
    if (ch < 16) ch = 16;
    if (ch >= ((int64_t)1 << 24)) return -2;  // a row's local rank must fit in 24 bits
    *chunk = (int)ch;
    *grid = (int)((T + ch - 1) / ch);
    return 0;
}

cudaError_t launch_route(const RouteArgs& a, int grid, int chunk, cudaStream_t s) {
    const bool bf16 = a.dtype == CLEARMOE_BF16;
    const size_t smem = route_smem(a.dtype, a.d, a.E, chunk);  // the attribute is set by route_grid
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(bf16 ? RT_BF16_THREADS : RT_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (!bf16) return cudaLaunchKernelEx(&cfg, route_kernel<false, false>, a, chunk);
    if (route_wreg(a.dtype, a.d, a.E)) return cudaLaunchKernelEx(&cfg, route_kernel<true, true>, a, chunk);
    return cudaLaunchKernelEx(&cfg, route_kernel<true, false>, a, chunk);
}

cudaError_t launch_route_finalize(const RouteArgs& a, int grid, int chunk, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, route_finalize_kernel, a, chunk, grid);
}

}  // namespace cm
