// Routing of the CLEAR-MoE FFN (Algorithm 3, steps 3-4):
//   logits = W_g x + b_g (linear router), a = argmax (lowest index on ties),
//   per-expert histogram, exclusive prefix sum, and the stable permutation perm[slot] = token.
//
// Every routing kernel gives CTA b a contiguous range of `chunk` tokens, and no CTA ever waits for
// another: each writes its range's histogram to cta_counts and, per token, (expert | rank among the
// range's earlier tokens of that expert << 8) to tinfo. The slot of token t in range c is
// offsets[e] + (tokens of e in ranges before c) + its rank, in token order within each expert,
// which makes the sort stable. It is formed by the consumer of the routing: the fc1 epilogue of
// the 2-SM GEMM (which then stores z rows at their slots and writes perm), or route_finalize_kernel
// (perm and inv ahead of the other paths).
//
// bf16 tokens (route_tc_kernel): the d x E contraction runs on the tensor cores. One CTA per SM
//   streams its range as 128-row blocks into a ring of shared-memory stages, each stage nkc K blocks
//   (64 columns) of a block, loaded as 16 TMA boxes of 8 rows x nkc K blocks (128-byte swizzle), so
//   that every box reads nkc x 128 contiguous bytes of each of its rows (a box of 128 rows x 64
//   columns, 128 bytes per row, kept DRAM 45 % busy); W_g sits in shared memory as the B operand (16
//   rows, rows past E read as zero). One thread issues tcgen05.mma (M = 128, N = 16, K = 16, fp32
//   accumulator in tensor memory, two accumulators); four epilogue warps, one per TMEM lane quarter,
//   read their 32 rows' logits with tcgen05.ld, take the argmax per row (one row per lane, no
//   shuffles) and the ranks by one ballot per expert, exchanging the four warps' counts through
//   shared memory, and write idx and the final per-token word. A range's last, partial block loads
//   only the boxes that hold its rows, so that at most 7 rows past the range are read.
// fp32 tokens (route_f32_kernel): fp32 FMA on the CUDA cores (an fp32 router decision needs fp32
//   products), one row per lane, or a row split over up to 32 lanes when a CTA's range is short,
//   then the ranks from warp match masks.
// Class tokens (cls_stride > 0, t % cls_stride == 0) skip the router: idx = E, no histogram entry
// and no rank; their slots T - n_cls + t / cls_stride follow the experts' (the dense path).
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace cm {

// better (value, index) with the lower index winning exact ties
__device__ __forceinline__ void arg_better(float& bv, int& be, float v, int e) {
    if (v > bv || (v == bv && e < be)) {
        bv = v;
        be = e;
    }
}

// ------------------------------------------------------------------ bf16: tcgen05 router
constexpr int RTC_THREADS = 192;  // warps 0-3: epilogue (TMEM lane quarters), 4: producer, 5: MMA
constexpr int RTC_BM = 128;       // rows per block (the MMA's M)
constexpr int RTC_BK = 64;        // columns per K block (128 bytes)
constexpr int RTC_BOX_ROWS = 8;   // rows per TMA box: one 128-byte swizzle atom per K block
constexpr int RTC_WBOX_BYTES = 16 * RTC_BK * 2;  // W_g's box per K block: 16 rows, 2 KB
constexpr int RTC_MAX_STAGES = 16;
constexpr int RTC_TMEM_COLS = 32;  // two 16-column accumulators
#ifndef RTC_NKC_MAX
#define RTC_NKC_MAX 6  // K blocks per stage at most (6 x 128 contiguous bytes of each row per box)
#endif
// dynamic shared memory: the 227 KB a CTA may hold, less the kernel's static arrays and a margin
constexpr size_t RTC_SMEM_CAP = 227 * 1024 - 1024 - 256;

struct RouteTcArgs {
    RouteArgs r;
    CUtensorMap tmX;  // x [T x d] as {64, T, d / 64}: boxes of 64 x 8 rows x nkc K blocks
    CUtensorMap tmW;  // W_g [E x d]: boxes of 64 columns x 16 rows (rows past E read as zero)
    int chunk;
};

// A stage holds nkc K blocks of a 128-row block: 16 boxes of 8 rows, box b at b * nkc KB, its K
// block c at + c KB (an 8 x 128-byte swizzle atom), so the MMA reads K block c of the 128 rows
// with 8-row atoms nkc KB apart. Each box reads nkc x 128 contiguous bytes of each of its rows.
// Dynamic shared memory: [W_g: d / 64 boxes of 2 KB] [ring: S stages] [2 S + 6 mbarriers] [TMEM
// base]; the base is aligned to 1024 bytes in the kernel (the swizzle atom). nkc is the largest
// divisor of d / 64 up to RTC_NKC_MAX that leaves room for two stages.
struct RouteTcLayout {
    int nkc, S;
    size_t stage_bytes, w_bytes, ring, bars, total;
};
__host__ __device__ inline RouteTcLayout route_tc_layout(int d) {
    RouteTcLayout L;
    const int nk = d / RTC_BK;
    L.w_bytes = (size_t)nk * RTC_WBOX_BYTES;
    L.ring = L.w_bytes;
    const size_t avail = RTC_SMEM_CAP - 1024 - L.w_bytes - (2 * RTC_MAX_STAGES + 6) * 8 - 16;
    L.nkc = 1;
    L.S = 1;
    for (int c = 1; c <= RTC_NKC_MAX && c <= nk; ++c) {
        if (nk % c) continue;
        int S = (int)(avail / ((size_t)RTC_BM * c * RTC_BK * 2));
        if (S > RTC_MAX_STAGES) S = RTC_MAX_STAGES;
        if (S < 2) continue;
        L.nkc = c;
        L.S = S;
    }
    L.stage_bytes = (size_t)RTC_BM * L.nkc * RTC_BK * 2;
    L.bars = L.ring + (size_t)L.S * L.stage_bytes;
    L.total = 1024 + L.bars + (size_t)(2 * L.S + 6) * 8 + 16;
    return L;
}

__global__ void __launch_bounds__(RTC_THREADS, 1) route_tc_kernel(const __grid_constant__ RouteTcArgs A) {
    const RouteArgs& a = A.r;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ int s_cnt[2][4][CM_MAX_E];  // per block (double-buffered): each quarter warp's expert counts
    __shared__ float s_b[CM_MAX_E], s_g[CM_MAX_E];
    __shared__ int s_abort;
    const uint32_t raw = smem_u32(smem_raw);
    unsigned char* sm = smem_raw + ((1024 - (raw & 1023)) & 1023);
    const RouteTcLayout lay = route_tc_layout(a.d);
    const int S = lay.S;
    const uint32_t w_u32 = smem_u32(sm);
    const uint32_t ring_u32 = w_u32 + (uint32_t)lay.ring;
    const uint32_t bar0 = w_u32 + (uint32_t)lay.bars;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + lay.bars + (size_t)(2 * S + 6) * 8);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
    const uint32_t wbar = bar0 + 8u * (2 * S);
    auto tfull_bar = [&](int i) { return bar0 + 8u * (2 * S + 1 + i); };
    auto tempty_bar = [&](int i) { return bar0 + 8u * (2 * S + 3 + i); };
    const uint32_t drain_bar = bar0 + 8u * (2 * S + 5);
    volatile int* abort_flag = &s_abort;
    const uint64_t lim = (uint64_t)a.wait_limit_ns;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int E = a.E, nk = a.d / RTC_BK, nkc = lay.nkc, nh = nk / nkc;
    const uint32_t stage_bytes = (uint32_t)lay.stage_bytes, box_bytes = (uint32_t)nkc * RTC_BOX_ROWS * RTC_BK * 2;
    const int64_t row0 = (int64_t)blockIdx.x * A.chunk;
    const int nrows = (int)max((int64_t)0, min((int64_t)A.chunk, a.T - row0));
    const int nblk = (nrows + RTC_BM - 1) / RTC_BM;
    const bool producer = warp == 4 && lane == 0, issuer = warp == 5 && lane == 0;

    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_bar(s), 1);   // the producer's arrive + the stage's bytes
            mbar_init(empty_bar(s), 1);  // one commit once the stage's MMAs have read it
        }
        mbar_init(wbar, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(tfull_bar(i), 1);   // one commit per block
            mbar_init(tempty_bar(i), 4);  // the four epilogue warps
        }
        mbar_init(drain_bar, 1);
        s_abort = 0;
        mbar_fence_init();
    }
    if (warp == 5) tmem_alloc(smem_u32(tmem_slot), RTC_TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // W_g (a weight, not written by the previous kernel) is requested before the launch-overlap wait
    if (producer && nblk > 0) {
        mbar_arrive_expect_tx(wbar, (uint32_t)(nk * RTC_WBOX_BYTES));
        for (int kc = 0; kc < nk; ++kc) tma_load_2d(w_u32 + kc * RTC_WBOX_BYTES, &A.tmW, kc * RTC_BK, 0, wbar);
    }
    pdl_wait();  // from here on the previous kernel's results (x) are read and outputs written
    // the next kernel may start now (its CTAs set up, and may read x, while this one streams):
    // released only after the wait, so every kernel before this one has completed by then
    pdl_launch_dependents();
    if (tid < CM_MAX_E) {
        s_b[tid] = tid < E ? bf16_to_f32(static_cast<const uint16_t*>(a.bg)[tid]) : 0.f;
        s_g[tid] = (a.ln_stats && tid < E) ? a.ln_wsum[tid] : 0.f;
    }
    __syncthreads();
    const uint32_t tmem = *tmem_slot;

    if (producer) {
        // stage k = K blocks [h nkc, +nkc) of block j, with j = k / nh and h = k % nh; ring slot k % S
        int k = 0;
        bool ok = true;
        for (int j = 0; j < nblk && ok; ++j) {
            const int rows = min(RTC_BM, nrows - j * RTC_BM);
            const int r = (int)(row0 + (int64_t)j * RTC_BM);  // T <= 2^30
            const int nbox = (rows + RTC_BOX_ROWS - 1) / RTC_BOX_ROWS;  // the last block may be partial
            const uint32_t bytes = (uint32_t)nbox * box_bytes;
            for (int h = 0; h < nh; ++h, ++k) {
                const int s = k % S;
                if (!mbar_wait(empty_bar(s), ((k / S) & 1) ^ 1, abort_flag, a.status, lim)) {
                    ok = false;
                    break;
                }
                if (k == a.debug_skip && blockIdx.x == 0) continue;  // fault injection: withhold a stage
                const uint32_t dst = ring_u32 + (uint32_t)s * stage_bytes;
                mbar_arrive_expect_tx(full_bar(s), bytes);
                for (int b = 0; b < nbox; ++b)
                    tma_load_3d(dst + (uint32_t)b * box_bytes, &A.tmX, 0, r + b * RTC_BOX_ROWS, h * nkc, full_bar(s));
            }
        }
        if (!ok)  // gave up: let the copies in flight land before the CTA moves on
            for (int j = max(0, k - S); j < k; ++j)
                mbar_wait(full_bar(j % S), (j / S) & 1, nullptr, a.status, 10000000ull);
        if (nblk > 0) mbar_wait(wbar, 0, nullptr, a.status, 10000000ull);  // W_g's boxes have landed too
    } else if (issuer) {
        const uint32_t idesc = idesc_bf16_f32(RTC_BM, 16);
        // a K block's descriptor is the ring base's plus the byte offset / 16 (addresses stay below
        // 256 KB): 8-row atoms nkc KB apart in x's stages, 1 KB apart in W_g's boxes
        const uint64_t dA0 = sdesc_kmajor_sw128_sbo(ring_u32, (uint32_t)nkc * 1024u);
        const uint64_t dW0 = sdesc_kmajor_sw128(w_u32);
        bool ok = nblk == 0 || mbar_wait(wbar, 0, abort_flag, a.status, lim);
        int k = 0;
        for (int j = 0; j < nblk && ok; ++j) {
            const int acc = j & 1;
            if (!mbar_wait(tempty_bar(acc), ((j >> 1) & 1) ^ 1, abort_flag, a.status, lim)) break;
            tc_fence_after();
            const uint32_t dtm = tmem + (uint32_t)acc * 16;
            for (int h = 0; h < nh; ++h, ++k) {
                const int s = k % S;
                if (!mbar_wait(full_bar(s), (k / S) & 1, abort_flag, a.status, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int c = 0; c < nkc; ++c) {
                    const uint64_t da = dA0 + (uint64_t)((s * stage_bytes + c * 1024u) >> 4);
                    const uint64_t dw = dW0 + (uint64_t)(((h * nkc + c) * RTC_WBOX_BYTES) >> 4);
#pragma unroll
                    for (int kk = 0; kk < RTC_BK / 16; ++kk)  // 16 columns = 32 bytes = 2 descriptor units
                        umma_bf16(dtm, da + 2 * kk, dw + 2 * kk, idesc, (h > 0 || c > 0 || kk > 0) ? 1u : 0u);
                }
                umma_commit(empty_bar(s));
            }
            if (!ok) break;
            umma_commit(tfull_bar(acc));
        }
        umma_commit(drain_bar);  // every MMA issued has completed before tensor memory is released
        mbar_wait(drain_bar, 0, nullptr, a.status, 10000000ull);
    } else if (warp < 4) {
        // epilogue: warp q reads TMEM lanes [32 q, +32) = rows 32 q .. 32 q + 31 of each block. Every
        // warp runs all nblk iterations (a wait that gave up only skips the work), so the named
        // barrier below is reached the same number of times by all four.
        const int q = warp;
        const unsigned below = (1u << lane) - 1u;
        const bool lnf = a.ln_stats != nullptr;
        float bias[CM_MAX_E], gsum[CM_MAX_E];  // b_g and, with the LayerNorm folded, W_g's row sums
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) {
            bias[e] = s_b[e];
            gsum[e] = s_g[e];
        }
        int run = 0;  // lane e < E: expert e's rows of the range in the blocks so far
        for (int j = 0; j < nblk; ++j) {
            const int acc = j & 1;
            const int i = j * RTC_BM + q * 32 + lane;  // row within the range
            const bool valid = i < nrows;
            const int64_t row = row0 + i;
            const float2 ln = (lnf && valid) ? a.ln_stats[row] : make_float2(0.f, 1.f);
            // the warp agrees on the outcome, so that its tcgen05.ld runs on all lanes or none
            const bool ok = __all_sync(0xffffffffu, mbar_wait(tfull_bar(acc), (j >> 1) & 1, abort_flag, a.status, lim));
            int esel = -1;  // this lane's expert (E: a class token; -1: no row)
            if (ok) {
                tc_fence_after();
                uint32_t v[16];
                CM_TMEM_LD_X16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)acc * 16, v);
                tmem_wait_ld();
                if (valid) {
                    float bv = -INFINITY;
                    int be = 0x7fffffff;
#pragma unroll
                    for (int e = 0; e < CM_MAX_E; ++e) {
                        if (e < E) {
                            float l = __uint_as_float(v[e]);
                            if (lnf) l = ln.y * fmaf(-ln.x, gsum[e], l);  // W_g LN(y) = rstd (W_g y - mean g)
                            arg_better(bv, be, l + bias[e], e);
                        }
                    }
                    esel = be < E ? be : 0;  // only reachable with non-finite logits
                    if (a.cls_stride > 0 && row % a.cls_stride == 0) esel = E;  // a class token
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty_bar(acc));  // the accumulator may be overwritten
            // ranks: earlier blocks' rows of the expert + earlier quarters' + earlier lanes'. The lanes
            // that picked the same expert form one match group; its first lane records the group's size.
            const unsigned same = __match_any_sync(0xffffffffu, esel);
            const int rk = __popc(same & below);
            int* cw = &s_cnt[j & 1][q][0];
            if (lane < CM_MAX_E) cw[lane] = 0;
            __syncwarp();
            if (esel >= 0 && esel < E && rk == 0) cw[esel] = __popc(same);
            const int* cb = &s_cnt[j & 1][0][0];
            asm volatile("bar.sync 1, 128;" ::: "memory");
            // lane e: expert e's rows before this warp's (earlier blocks and quarters), and in the block
            int pre = run, tot = 0;
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) {
                const int c = lane < CM_MAX_E ? cb[qq * CM_MAX_E + lane] : 0;
                if (qq < q) pre += c;
                tot += c;
            }
            run += tot;
            const int base = __shfl_sync(0xffffffffu, pre, (esel >= 0 && esel < E) ? esel : 0);
            if (ok && valid) {
                if (a.tinfo != a.idx) a.idx[row] = esel;
                a.tinfo[row] = esel < E ? esel | ((base + rk) << 8) : E;
            }
        }
        if (q == 0 && lane < E) a.cta_counts[(size_t)blockIdx.x * CM_MAX_E + lane] = run;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 5) tmem_dealloc(tmem, RTC_TMEM_COLS);
}

// ------------------------------------------------------------------ fp32 router
constexpr int RT_THREADS = 256;  // 8 warps
constexpr size_t RT_F32_SMEM_MAX = 220 * 1024;

// Dynamic shared memory: [W_g as fp32] [per-row word: expert | local rank << 8, when chunk words
// fit; else that word lives in idx in global memory (the CTA's own rows, visible block-wide after
// __syncthreads) until the finalize kernel rewrites idx with the expert alone], so the footprint
// does not grow with T.
struct RouteF32Layout {
    size_t sidx, total;
    bool sidx_in_smem;
};
__host__ __device__ inline RouteF32Layout route_f32_layout(int d, int E, int chunk) {
    RouteF32Layout L;
    L.sidx = ((size_t)E * d * 4 + 127) & ~(size_t)127;
    L.sidx_in_smem = L.sidx + (size_t)chunk * 4 <= RT_F32_SMEM_MAX;
    L.total = L.sidx + (L.sidx_in_smem ? (size_t)chunk * 4 : 0);
    return L;
}

__global__ void __launch_bounds__(RT_THREADS) route_f32_kernel(const RouteArgs a, const int chunk) {
    constexpr int NTHREADS = RT_THREADS;
    constexpr int NWARPS = NTHREADS / 32;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ int s_count[CM_MAX_E];
    __shared__ int s_run[CM_MAX_E];
    __shared__ int s_wc[NWARPS][CM_MAX_E];

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int E = a.E, d = a.d;
    const int64_t row0 = (int64_t)blockIdx.x * chunk;
    const int nrows = (int)max((int64_t)0, min((int64_t)chunk, a.T - row0));
    const RouteF32Layout lay = route_f32_layout(d, E, chunk);
    // per-row expert after the first pass: in shared memory when it fits, else read back from idx
    uint32_t* sinfo = lay.sidx_in_smem ? reinterpret_cast<uint32_t*>(smem + lay.sidx) : nullptr;
    auto info_of = [&](int i) -> uint32_t { return sinfo ? sinfo[i] : (uint32_t)__ldcg(a.idx + row0 + i); };
    auto record = [&](int i, int e) {  // first-pass result of row i: idx, its word, histogram
        a.idx[row0 + i] = e;
        if (sinfo) sinfo[i] = (uint32_t)e;
        if (e < E) atomicAdd(&s_count[e], 1);  // e == E: a class token
    };
    if (tid < CM_MAX_E) s_count[tid] = 0;

    // ---------------- router logits + argmax for this CTA's rows
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
    // Lanes per row: with few rows per CTA (small T), each row is split over tpr lanes (a power of
    // two, tpr x rows <= the CTA's threads), which take its float4 columns in turn and add their
    // partial logits by shuffles; with many rows, one row per lane (tpr = 1), fp32 FMA in k order
    // and no cross-lane step. W_g is broadcast from shared memory (d % 4 == 0).
    int tpr = 1;
    while (tpr < 32 && nrows * tpr * 2 <= NTHREADS) tpr *= 2;
    const int rpw = 32 / tpr;  // rows per warp per pass
    const int sub = lane & (tpr - 1);
    const float* X = static_cast<const float*>(a.x);
    const int d4 = d / 4;
    for (int b0 = warp * rpw; b0 < nrows; b0 += NWARPS * rpw) {
        const int i = b0 + lane / tpr;
        const bool valid = i < nrows;
        const float4* xr = reinterpret_cast<const float4*>(X + (row0 + (valid ? i : 0)) * d);
        float acc[CM_MAX_E];
#pragma unroll
        for (int e = 0; e < CM_MAX_E; ++e) acc[e] = 0.f;
        for (int k4 = sub; k4 < d4; k4 += 4 * tpr) {
            float4 xv[4];
#pragma unroll
            for (int j = 0; j < 4; ++j)
                xv[j] = (k4 + j * tpr < d4) ? xr[k4 + j * tpr] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int kk = k4 + j * tpr;
                if (kk < d4) {
#pragma unroll
                    for (int e = 0; e < CM_MAX_E; ++e) {
                        if (e < E) {
                            const float4 w = reinterpret_cast<const float4*>(Wf + (size_t)e * d)[kk];
                            acc[e] = fmaf(xv[j].x, w.x, acc[e]);
                            acc[e] = fmaf(xv[j].y, w.y, acc[e]);
                            acc[e] = fmaf(xv[j].z, w.z, acc[e]);
                            acc[e] = fmaf(xv[j].w, w.w, acc[e]);
                        }
                    }
                }
            }
        }
        for (int off = tpr >> 1; off > 0; off >>= 1) {  // every lane of the row ends with the sums
#pragma unroll
            for (int e = 0; e < CM_MAX_E; ++e)
                if (e < E) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], off);
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
        if (valid && sub == 0) record(i, be);
    }
    __syncthreads();

    // ---------------- this CTA's histogram, and each row's rank among the CTA's earlier rows of
    // its expert (warp match masks, then a per-expert prefix over warps and over passes), which
    // makes the final order stable.
    if (tid < E) a.cta_counts[(size_t)blockIdx.x * CM_MAX_E + tid] = s_count[tid];
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
    // equal ranges over all CTAs (a range's last block may be partial)
    int64_t ch = (T + want - 1) / want;
    // the shared-memory attribute belongs to a device: set once per device
    if (smem_attr_once((const void*)route_tc_kernel, (int)RTC_SMEM_CAP) != cudaSuccess ||
        smem_attr_once((const void*)route_f32_kernel, (int)RT_F32_SMEM_MAX) != cudaSuccess) {
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
        const size_t smem = bf16 ? route_tc_layout(d).total : route_f32_layout(d, E, (int)ch).total;
        occ = -1;
        for (int i = 0; i < ncache; ++i)
            if (cache[i].dev == dev && cache[i].dtype == dtype && cache[i].d == d && cache[i].E == E &&
                cache[i].smem == smem)
                occ = cache[i].occ;
        if (occ < 0) {
            const void* fn = bf16 ? (const void*)route_tc_kernel : (const void*)route_f32_kernel;
            cudaError_t err = cudaOccupancyMaxActiveBlocksPerMultiprocessorWithFlags(
                &occ, fn, bf16 ? RTC_THREADS : RT_THREADS, smem, cudaOccupancyDefault);
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
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (!bf16) {  // the attribute is set by route_grid
        cfg.blockDim = dim3(RT_THREADS);
        cfg.dynamicSmemBytes = route_f32_layout(a.d, a.E, chunk).total;
        return cudaLaunchKernelEx(&cfg, route_f32_kernel, a, chunk);
    }
    if (a.d % RTC_BK != 0 || a.E > CM_MAX_E || a.T > ((int64_t)1 << 30)) return cudaErrorInvalidValue;
    RouteTcArgs t;
    t.r = a;
    t.chunk = chunk;
    if (encode_tmap_bf16_chunks(&t.tmX, a.x, a.T, a.d, RTC_BOX_ROWS, route_tc_layout(a.d).nkc) ||
        encode_tmap_bf16(&t.tmW, a.Wg, a.E, a.d, 16))
        return cudaErrorInvalidValue;
    cfg.blockDim = dim3(RTC_THREADS);
    cfg.dynamicSmemBytes = route_tc_layout(a.d).total;
    return cudaLaunchKernelEx(&cfg, route_tc_kernel, t);
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
