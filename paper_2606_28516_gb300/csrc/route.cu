// Fused routing kernel of the CLEAR-MoE FFN (Algorithm 3, steps 3-4):
//   logits = W_g x + b_g (linear router), a = argmax (lowest index on ties),
//   per-expert histogram, exclusive prefix sum, and the stable permutation perm[slot] = token.
//
// One cooperative launch of co-resident CTAs; CTA b owns a contiguous range of `chunk` tokens.
//   phase 1: stream x once from HBM, router logits and argmax per token, local histogram.
//            bf16: one CTA per SM; a producer thread copies the CTA's rows, 16 at a time, into a
//            ring of shared-memory stages with 1-D bulk copies (mbarrier-tracked, so the bytes in
//            flight cost no registers) and eight consumer warps take one 16-row stage each;
//   grid-wide wait (bounded, on a monotone arrival counter);
//   phase 2: each CTA sums the histograms of the CTAs before it and writes its tokens' slots in
//            token order (ranks from warp match masks), which makes the sort stable.
// bf16 tokens: the d x E contraction runs on the legacy warp MMA (m16n8k16, fp32 accumulate)
// straight from registers: the 16-byte loads of x are coalesced, and the K order of each
// fragment is permuted identically for x and W_g, which leaves every dot product unchanged.
// fp32 tokens: fp32 FMA on the CUDA cores (an fp32 router decision needs fp32 products).
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace cm {

constexpr int RT_THREADS = 256;                 // fp32 router: 8 warps
constexpr int RT_BF16_THREADS = 288;            // bf16 router: 8 consumer warps + 1 producer warp
constexpr int RT_MAX_WARPS = RT_BF16_THREADS / 32;
constexpr int RT_STAGE_ROWS = 16;               // rows per ring stage (one MMA row group)
constexpr int RT_RING_BYTES = 192 * 1024;       // shared-memory ring budget (bf16 router)

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

__host__ __device__ inline size_t frag_bytes(int dtype, int d, int E) {
    if (dtype == CLEARMOE_BF16) return (size_t)((E + 7) / 8) * (d / 32) * 32 * 16;
    return (size_t)E * d * 4;
}

// Dynamic shared memory: [router weights] [bf16: ring of S stages] [bf16: 2 S mbarriers]. The
// chosen expert of each row goes to idx in global memory and is read back from there (the CTA's
// own writes, visible block-wide after __syncthreads), so the footprint does not grow with T.
// The ring has one slot per consumer warp (S = 8, or 4 when eight stages do not fit): consumer
// warp w alone reads slot w, for stages w, w + S, ..., so each of its mbarrier waits is for the
// phase right after the one it last consumed (a parity wait cannot tell phases two apart).
struct RouteLayout {
    size_t ring, bars, sidx, total;
    int S, stage_bytes;
    bool sidx_in_smem;
};
constexpr size_t RT_SMEM_MAX = 220 * 1024;
__host__ __device__ inline RouteLayout route_layout(int dtype, int d, int E, int chunk) {
    RouteLayout L;
    const size_t frag = (frag_bytes(dtype, d, E) + 127) & ~(size_t)127;
    L.stage_bytes = RT_STAGE_ROWS * d * 2;
    L.S = 0;
    L.ring = frag;
    if (dtype == CLEARMOE_BF16) L.S = (8 * L.stage_bytes <= RT_RING_BYTES) ? 8 : 4;
    L.bars = (L.ring + (size_t)L.S * L.stage_bytes + 15) & ~(size_t)15;
    L.sidx = L.bars + (size_t)2 * L.S * 8;
    // expert ids of the CTA's rows: in shared memory when they fit, else read back from idx
    L.sidx_in_smem = L.sidx + (size_t)chunk <= RT_SMEM_MAX;
    L.total = L.sidx + (L.sidx_in_smem ? (size_t)chunk : 0);
    return L;
}
static size_t route_smem(int dtype, int d, int E, int chunk) { return route_layout(dtype, d, E, chunk).total; }

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

template <bool BF16>
__global__ void __launch_bounds__(BF16 ? RT_BF16_THREADS : RT_THREADS) route_kernel(const RouteArgs a, const int chunk) {
    constexpr int NTHREADS = BF16 ? RT_BF16_THREADS : RT_THREADS;
    constexpr int NWARPS = NTHREADS / 32;
    constexpr int NCONS_MAX = 8;  // warps computing logits (bf16: the first S warps)
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ int s_count[CM_MAX_E];
    __shared__ int s_base[CM_MAX_E];
    __shared__ int s_tot[CM_MAX_E];
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
    uint8_t* sidx = lay.sidx_in_smem ? smem + lay.sidx : nullptr;
    auto expert_of = [&](int i) -> int { return sidx ? (int)sidx[i] : __ldcg(a.idx + row0 + i); };
    auto record = [&](int i, int e) {  // phase 1 result of row i: idx, local id copy, histogram
        a.idx[row0 + i] = e;
        if (sidx) sidx[i] = (uint8_t)e;
        atomicAdd(&s_count[e], 1);
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
        if (tid == 0) {
            for (int s = 0; s < S; ++s) {
                mbar_init(full_bar(s), 1);
                mbar_init(empty_bar(s), 1);
            }
            mbar_fence_init();
        }
        // B fragments of W_g: [n-tile][32-column chunk][lane] -> 8 consecutive bf16 of row
        // nt*8 + lane/4, columns chunk*32 + (lane%4)*8.
        uint4* bfrag = reinterpret_cast<uint4*>(smem);
        const uint16_t* W = static_cast<const uint16_t*>(a.Wg);
        for (int i = tid; i < NT * nchunk * 32; i += NTHREADS) {
            const int l = i & 31, c = (i >> 5) % nchunk, nt = (i >> 5) / nchunk;
            const int e = nt * 8 + (l >> 2);
            uint4 v = make_uint4(0, 0, 0, 0);
            if (e < E) v = *reinterpret_cast<const uint4*>(W + (size_t)e * d + c * 32 + (l & 3) * 8);
            bfrag[i] = v;
        }
        __syncthreads();
        if (warp == NCONS_MAX) {
            // ---- producer: stage k = rows [16 k, 16 k + 16) of this CTA, ring slot k % S
            if (lane == 0) {
                const unsigned char* xb = static_cast<const unsigned char*>(a.x) + row0 * d * 2;
                int k = 0;
                for (; k < nstages; ++k) {
                    const int s = k % S;
                    if (!mbar_wait(empty_bar(s), ((k / S) & 1) ^ 1, abort_flag, a.status, (uint64_t)a.wait_limit_ns))
                        break;
                    const int rows = min(RT_STAGE_ROWS, nrows - k * RT_STAGE_ROWS);
                    const uint32_t bytes = (uint32_t)rows * d * 2;
                    mbar_arrive_expect_tx(full_bar(s), bytes);
                    bulk_g2s(ring + s * SB, xb + (size_t)k * SB, bytes, full_bar(s));
                }
                if (k < nstages) {  // gave up: let the copies in flight land before moving on
                    for (int j = max(0, k - S); j < k; ++j)
                        mbar_wait(full_bar(j % S), (j / S) & 1, nullptr, a.status, 10000000ull);
                }
            }
        } else if (warp < S) {
            // ---- consumers: warp w owns slot w and takes stages w, w + S, w + 2 S, ...
            const uint16_t* bgp = static_cast<const uint16_t*>(a.bg);
            const int g = lane >> 2, tig = lane & 3;
            const uint4 zero = make_uint4(0, 0, 0, 0);
            for (int k = warp; k < nstages; k += S) {
                const int s = warp;
                if (!mbar_wait(full_bar(s), (k / S) & 1, abort_flag, a.status, (uint64_t)a.wait_limit_ns)) break;
                const int rows = min(RT_STAGE_ROWS, nrows - k * RT_STAGE_ROWS);
                const bool vA = g < rows, vB = g + 8 < rows;
                const unsigned char* st = smem + lay.ring + (size_t)s * SB;
                const uint4* pA = reinterpret_cast<const uint4*>(st + (size_t)g * d * 2) + tig;
                const uint4* pB = reinterpret_cast<const uint4*>(st + (size_t)(g + 8) * d * 2) + tig;
                float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
                for (int c = 0; c < nchunk; ++c) {
                    const uint4 xa = vA ? pA[4 * c] : zero;
                    const uint4 xb = vB ? pB[4 * c] : zero;
#pragma unroll
                    for (int nt = 0; nt < 2; ++nt) {
                        if (nt < NT) {
                            const uint4 w = bfrag[(nt * nchunk + c) * 32 + lane];
                            mma_bf16_16816(acc[nt], xa.x, xb.x, xa.y, xb.y, w.x, w.y);
                            mma_bf16_16816(acc[nt], xa.z, xb.z, xa.w, xb.w, w.z, w.w);
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(empty_bar(s));  // the stage's rows are in registers now
                // D fragment: acc[nt][0..1] = row g, experts nt*8 + 2*tig + {0,1}; [2..3] = row g+8
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
                            arg_better(bA, eA, acc[nt][j] + bias, e);
                            arg_better(bB, eB, acc[nt][2 + j] + bias, e);
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
                if (tig == 0) {
                    const int iA = k * RT_STAGE_ROWS + g, iB = iA + 8;
                    if (vA) record(iA, eA);
                    if (vB) record(iB, eB);
                }
            }
        }
    } else {
        float* Wf = reinterpret_cast<float*>(smem);
        const float* W = static_cast<const float*>(a.Wg);
        for (int i = tid; i < E * d; i += NTHREADS) Wf[i] = W[i];
        __syncthreads();
        const float* bgp = static_cast<const float*>(a.bg);
        const float* X = static_cast<const float*>(a.x);
        for (int i = warp; i < nrows; i += NWARPS) {
            const float* xr = X + (row0 + i) * d;
            float acc[CM_MAX_E];
#pragma unroll
            for (int e = 0; e < CM_MAX_E; ++e) acc[e] = 0.f;
            for (int k = lane; k < d; k += 32) {
                const float xv = xr[k];
#pragma unroll
                for (int e = 0; e < CM_MAX_E; ++e)
                    if (e < E) acc[e] = fmaf(xv, Wf[e * d + k], acc[e]);
            }
            float bv = -INFINITY;
            int be = 0x7fffffff;
#pragma unroll
            for (int e = 0; e < CM_MAX_E; ++e) {
                if (e < E) {
                    float v = acc[e];
#pragma unroll
                    for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
                    arg_better(bv, be, v + bgp[e], e);
                }
            }
            if (be > E - 1) be = 0;
            if (lane == 0) record(i, be);
        }
    }
    __syncthreads();

    // ---------------- the local histogram (built in phase 1), published for the other CTAs by the
    // thread that arrives at the grid barrier

    // ---------------- grid-wide wait (bounded), self-resetting: the last of `arrivals` CTAs zeroes
    // the arrival count and bumps the generation that the others wait on, so nothing carries over
    // to the next launch and the host keeps no barrier state.
    if (tid == 0) {
        unsigned int* arrived = a.barrier;
        unsigned int* generation = a.barrier + 1;
        for (int e = 0; e < E; ++e) a.cta_counts[(size_t)blockIdx.x * CM_MAX_E + e] = s_count[e];
        const unsigned int gen0 = ld_acquire_u32(generation);
        __threadfence();  // the histogram is visible before this CTA's arrival
        unsigned int prev;
        asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(prev) : "l"(arrived) : "memory");
        if (prev == a.arrivals - 1) {
            st_release_u32(generation, gen0 + 1);  // release everyone, then reset for the next launch
            atomicExch(arrived, 0u);
        } else {
            const uint64_t t0 = globaltimer();
            while (ld_acquire_u32(generation) == gen0) {
                if (globaltimer() - t0 > (uint64_t)a.wait_limit_ns) {
                    s_abort = 1;
                    set_status(a.status, CLEARMOE_ETIMEOUT);
                    break;
                }
                __nanosleep(64);
            }
        }
    }
    __syncthreads();
    if (s_abort) return;

    // ---------------- phase 2: global offsets, then this CTA's slots in token order
    for (int e = warp; e < E; e += NWARPS) {
        int before = 0, total = 0;
        for (int b = lane; b < (int)gridDim.x; b += 32) {
            const int c = __ldcg(&a.cta_counts[(size_t)b * CM_MAX_E + e]);
            total += c;
            if (b < (int)blockIdx.x) before += c;
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) {
            before += __shfl_xor_sync(0xffffffffu, before, off);
            total += __shfl_xor_sync(0xffffffffu, total, off);
        }
        if (lane == 0) {
            s_base[e] = before;
            s_tot[e] = total;
        }
    }
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int e = 0; e < E; ++e) {
            const int t = s_tot[e];
            s_base[e] += run;
            if (blockIdx.x == 0) {
                a.counts[e] = t;
                a.offsets[e] = run;
            }
            run += t;
            s_run[e] = 0;
        }
        if (blockIdx.x == 0) a.offsets[E] = run;
    }
    const unsigned lt = (1u << lane) - 1u;
    for (int i0 = 0; i0 < nrows; i0 += NTHREADS) {
        if (tid < NWARPS * CM_MAX_E) (&s_wc[0][0])[tid] = 0;
        __syncthreads();
        const int i = i0 + tid;
        const bool valid = i < nrows;
        const int e = valid ? expert_of(i) : CM_MAX_E + 1;
        const unsigned same = __match_any_sync(0xffffffffu, e);
        const int rank = __popc(same & lt);
        if (valid && rank == 0) s_wc[warp][e] = __popc(same);
        __syncthreads();
        if (tid < E) {
            int run = s_run[tid];
            for (int w = 0; w < NWARPS; ++w) {
                const int c = s_wc[w][tid];
                s_wc[w][tid] = run;
                run += c;
            }
            s_run[tid] = run;
        }
        __syncthreads();
        if (valid) {
            const int slot = s_base[e] + s_wc[warp][e] + rank;
            a.perm[slot] = (int32_t)(row0 + i);
            if (a.inv) a.inv[row0 + i] = slot;
        }
        __syncthreads();
    }
}

int route_max_ctas(int num_sms, int, int, int) { return num_sms * 8; }

int route_grid(int64_t T, int d, int E, int dtype, int num_sms, int* grid, int* chunk) {
    const bool bf16 = dtype == CLEARMOE_BF16;
    int occ = 0;
    int64_t want = (int64_t)num_sms * (bf16 ? 1 : 2);  // bf16: one CTA per SM owns the ring
    int64_t ch = ((T + want - 1) / want + 15) / 16 * 16;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    static bool attr_set = false;
    if (!attr_set) {
            if (cudaFuncSetAttribute((const void*)route_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 220 * 1024) != cudaSuccess ||
            cudaFuncSetAttribute((const void*)route_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 220 * 1024) != cudaSuccess)
            return -1;
        attr_set = true;
    }
    // occupancy queries are cached: (dtype, d, E, shared-memory bytes) -> CTAs per SM
    static struct { int dtype, d, E; size_t smem; int occ; } cache[32];
    static int ncache = 0;
    for (int iter = 0; iter < 4; ++iter) {
        const size_t smem = route_smem(dtype, d, E, (int)ch);
        occ = -1;
        for (int i = 0; i < ncache; ++i)
            if (cache[i].dtype == dtype && cache[i].d == d && cache[i].E == E && cache[i].smem == smem) occ = cache[i].occ;
        if (occ < 0) {
            cudaError_t err = cudaOccupancyMaxActiveBlocksPerMultiprocessorWithFlags(
                &occ, bf16 ? (const void*)route_kernel<true> : (const void*)route_kernel<false>,
                bf16 ? RT_BF16_THREADS : RT_THREADS, smem, cudaOccupancyDefault);
            if (err != cudaSuccess) return -1;
            if (ncache < 32) cache[ncache++] = {dtype, d, E, smem, occ};
        }
        if (occ <= 0) return -2;
        const int64_t maxg = (int64_t)occ * num_sms;
        if (want <= maxg) break;
        want = maxg;
        ch = ((T + want - 1) / want + 15) / 16 * 16;
    }
    if (ch < 16) ch = 16;
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
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (bf16) return cudaLaunchKernelEx(&cfg, route_kernel<true>, a, chunk);
    return cudaLaunchKernelEx(&cfg, route_kernel<false>, a, chunk);
}

}  // namespace cm
