// Exact-fp32 GEMM of the CLEAR-MoE FFN (fp32 layers) and the LayerNorm between stacked sublayers.
//
// The fp32 forward's GEMMs run on the tensor cores (three TF32 products per step, tc_gemm.cu) where
// the shapes allow; this CUDA-core kernel keeps exact fp32 products for the rest: the folded
// LayerNorm, the scaled-residual form, the MLP router's hidden layer, and widths that are not
// multiples of 16. One tiled kernel covers every product of the layer:
//   C[m, n] = epi( sum_k A0[rowA(m), k] B0[n, k]  +  sum_k A1[m, k] B1_e[n, k] )
// with an optional row gather of A0 (fc1 on tokens in expert order), an optional second K
// segment with a per-expert B (the grouped residual GEMM, Algorithm 3 step 5; with dense_last the
// last group is the class tokens' dense path, second segment only), an epilogue of
// bias, GELU or ReLU, per-column scale and per-row scale, and an optional row scatter of C (the
// unshuffle, step 6). With the LayerNorm folded into A0 (rows of the un-normalised stream y) the
// epilogue first forms rstd (acc - mean c_n), c_n = sum_k B0[n, k], since W LN(y) = rstd (W y - mean W 1).
// Launches with too few tiles to fill the GPU split each tile's K chain over several blocks, whose
// partial sums the tile's last block adds in a fixed order: results are deterministic for a given
// shape, and the order of the fp32 sum depends on the number of tiles (so on T).
#include "common.cuh"
#include "internal.h"

namespace cm {

constexpr int SG_K = 64;  // K per shared-memory step (each thread keeps one k column of it)

// TM x TM output tiles (64, or 32 when 64-wide tiles would leave most SMs idle), 256 threads, each
// thread an (TM / 16) x (TM / 16) block of outputs.
template <int TM>
__global__ void __launch_bounds__(256) simt_gemm_kernel(const SimtGemmArgs a, const int n_tiles_n) {
    constexpr int SG_M = TM, SG_N = TM, R = TM / 16, LD = TM * SG_K / 256;
    __shared__ float As[SG_K][SG_M + 1];  // +1: the per-step stores (one k per thread) hit distinct banks
    __shared__ float Bs[SG_K][SG_N + 1];
    const int tid = threadIdx.x;
    const int nt = blockIdx.x % n_tiles_n;
    const int mt = blockIdx.x / n_tiles_n;
    // Launched with programmatic dependent launch: the next kernel may be scheduled once every block
    // of this one has started, and this one reads nothing (offsets, operands, the split-K workspace
    // and counters) before the previous kernel has completed.
    pdl_launch_dependents();
    pdl_wait();
    int64_t m_lo, m_hi;
    int e = 0;
    if (a.offsets) {
        int acc = 0;
        bool found = false;
        for (e = 0; e < a.E; ++e) {
            const int lo = a.offsets[e], hi = a.offsets[e + 1];
            const int tiles = (hi - lo + SG_M - 1) / SG_M;
            if (mt < acc + tiles) {
                m_lo = lo + (int64_t)(mt - acc) * SG_M;
                m_hi = min((int64_t)hi, m_lo + SG_M);
                found = true;
                break;
            }
            acc += tiles;
        }
        if (!found) return;
    } else {
        m_lo = (int64_t)mt * SG_M;
        if (m_lo >= a.M) return;
        m_hi = min(a.M, m_lo + SG_M);
    }
    const int n0 = nt * SG_N;
    const float* B1 = a.B1[a.offsets ? e : 0];
    const int tx = tid & 15, ty = tid >> 4;
    float acc[R][R];
#pragma unroll
    for (int i = 0; i < R; ++i)
#pragma unroll
        for (int j = 0; j < R; ++j) acc[i][j] = 0.f;

    // Thread tid loads column kk = tid % SG_K of rows tid / SG_K + (256 / SG_K) i (i < LD) of both
    // operand tiles; the next step's values are loaded into registers while this step computes.
    const int kk = tid % SG_K, r0 = tid / SG_K;
    constexpr int RS = 256 / SG_K;
    // the tile's K chain in SG_K steps (the dense path's group has no first segment), and this
    // block's range of it: split blockIdx.y of gridDim.y equal parts
    const bool seg0_on = a.A0 != nullptr && a.K0 > 0 && !(a.offsets && a.dense_last && e == a.E - 1);
    const int st0 = seg0_on ? (a.K0 + SG_K - 1) / SG_K : 0;
    const int st1 = (a.A1 != nullptr && a.K1 > 0) ? (a.K1 + SG_K - 1) / SG_K : 0;
    const int nsplit = gridDim.y, split = blockIdx.y;
    const int s_lo = (int)((int64_t)(st0 + st1) * split / nsplit), s_hi = (int)((int64_t)(st0 + st1) * (split + 1) / nsplit);
    for (int seg = 0; seg < 2; ++seg) {
        const float* A = seg == 0 ? a.A0 : a.A1;
        const float* B = seg == 0 ? a.B0 : B1;
        const int K = seg == 0 ? a.K0 : a.K1;
        const int64_t lda = seg == 0 ? a.lda0 : a.lda1;
        const int seg_st = seg == 0 ? st0 : st1, seg_base = seg == 0 ? 0 : st0;
        const int lo = max(s_lo - seg_base, 0), hi = min(s_hi - seg_base, seg_st);
        if (lo >= hi) continue;
        const int k_begin = lo * SG_K, k_end = min(hi * SG_K, K);
        int arow[LD];  // this thread's A rows (gathered for fc1), -1 outside the tile
#pragma unroll
        for (int i = 0; i < LD; ++i) {
            const int64_t m = m_lo + r0 + RS * i;
            arow[i] = -1;
            if (m < m_hi) {
                const int64_t ar = (seg == 0 && a.a_rows) ? (int64_t)a.a_rows[m] : m;
                if ((uint64_t)ar < (uint64_t)a.M) arow[i] = (int)ar;  // M < 2^31
            }
        }
        float ra[LD], rb[LD];
        auto gload = [&](int k0) {
            const int k = k0 + kk;
#pragma unroll
            for (int i = 0; i < LD; ++i) {
                const int n = n0 + r0 + RS * i;
                ra[i] = (arow[i] >= 0 && k < K) ? A[(int64_t)arow[i] * lda + k] : 0.f;
                rb[i] = (n < a.N && k < K) ? B[(int64_t)n * K + k] : 0.f;
            }
        };
        gload(k_begin);
        for (int k0 = k_begin; k0 < k_end; k0 += SG_K) {
#pragma unroll
            for (int i = 0; i < LD; ++i) {
                As[kk][r0 + RS * i] = ra[i];
                Bs[kk][r0 + RS * i] = rb[i];
            }
            __syncthreads();
            if (k0 + SG_K < k_end) gload(k0 + SG_K);
#pragma unroll 8
            for (int k = 0; k < SG_K; ++k) {
                float av[R], bv[R];
#pragma unroll
                for (int i = 0; i < R; ++i) av[i] = As[k][ty * R + i];
#pragma unroll
                for (int j = 0; j < R; ++j) bv[j] = Bs[k][tx * R + j];
#pragma unroll
                for (int i = 0; i < R; ++i)
#pragma unroll
                    for (int j = 0; j < R; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
            }
            __syncthreads();
        }
    }
    if (nsplit > 1) {
        // this split's partial tile to the workspace; the tile's last block adds all of them in
        // split order (a fixed order: deterministic) and runs the epilogue, then clears the counter
        float* part = a.ws + (int64_t)blockIdx.x * nsplit * (TM * TM);
#pragma unroll
        for (int i = 0; i < R; ++i)
#pragma unroll
            for (int j = 0; j < R; ++j) part[(int64_t)split * (TM * TM) + (ty * R + i) * TM + tx * R + j] = acc[i][j];
        __threadfence();
        __syncthreads();
        __shared__ int s_last;
        if (tid == 0) s_last = atomicAdd(a.cnt + blockIdx.x, 1) == nsplit - 1;
        __syncthreads();
        if (!s_last) return;
        __threadfence();
#pragma unroll
        for (int i = 0; i < R; ++i)
#pragma unroll
            for (int j = 0; j < R; ++j) {
                float v = 0.f;
                for (int p = 0; p < nsplit; ++p) v += __ldcg(part + (int64_t)p * (TM * TM) + (ty * R + i) * TM + tx * R + j);
                acc[i][j] = v;
            }
        if (tid == 0) a.cnt[blockIdx.x] = 0;
    }
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const int64_t m = m_lo + ty * R + i;
        if (m >= m_hi) continue;
        const int64_t orow = a.c_rows ? (int64_t)a.c_rows[m] : m;
        if ((uint64_t)orow >= (uint64_t)a.M) continue;  // only a launch that gave up leaves such rows
        float2 ln = make_float2(0.f, 1.f);  // the LayerNorm folded into A0: (mean, rstd) of its row
        if (a.ln_stats) {
            const int64_t ar = a.a_rows ? (int64_t)a.a_rows[m] : m;
            if ((uint64_t)ar < (uint64_t)a.M) ln = a.ln_stats[ar];
        }
#pragma unroll
        for (int j = 0; j < R; ++j) {
            const int n = n0 + tx * R + j;
            if (n >= a.N) continue;
            float v = acc[i][j];
            if (a.ln_stats) v = ln.y * fmaf(-ln.x, a.ln_colsum[n], v);  // W LN(y) = rstd (W y - mean c)
            if (a.bias) v += a.bias[n];
            if (a.gelu) v = gelu_erf(v);
            if (a.relu) v = fmaxf(v, 0.f);
            if (a.scale) v *= a.scale[n];
            if (a.group_scale) {
                const int g = a.row_group[m];
                if ((unsigned)g < (unsigned)a.scale_groups) v = a.row_scale_inv ? v / a.group_scale[g] : v * a.group_scale[g];
            }
            a.C[orow * a.ldc + n] = v;
        }
    }
}

template <int TM>
static int64_t simt_blocks(const SimtGemmArgs& a, int* n_tiles_n) {
    *n_tiles_n = (a.N + TM - 1) / TM;
    int64_t m_tiles = (a.M + TM - 1) / TM;
    if (a.offsets) m_tiles += a.E;  // each expert adds at most one ragged tile
    return m_tiles * *n_tiles_n;
}

cudaError_t launch_simt_gemm(const SimtGemmArgs& a, cudaStream_t s) {
    int num_sms = current_device_sms();  // per device, cached
    if (num_sms <= 0) num_sms = 1;
    int n64 = 0, n32 = 0;
    const int64_t b64 = simt_blocks<64>(a, &n64), b32 = simt_blocks<32>(a, &n32);
    if (b64 <= 0) return cudaSuccess;
    const bool t32 = b64 < 2 * (int64_t)num_sms;  // too few 64-wide tiles to fill the GPU: 32-wide ones
    const int64_t blocks = t32 ? b32 : b64;
    const int tm = t32 ? 32 : 64;
    // split K while the tiles alone would give fewer than four blocks per SM, each part at least two
    // SG_K steps, within the workspace
    const int steps = (a.K0 + SG_K - 1) / SG_K + (a.A1 ? (a.K1 + SG_K - 1) / SG_K : 0);
    int64_t nsplit = 1;
    if (a.ws && a.cnt && blocks <= a.cnt_len) {
        nsplit = (4 * (int64_t)num_sms) / blocks;
        if (nsplit > SIMT_MAX_SPLIT) nsplit = SIMT_MAX_SPLIT;
        if (nsplit > steps / 2) nsplit = steps / 2;
        while (nsplit > 1 && nsplit * blocks * tm * tm > a.ws_floats) --nsplit;
        if (nsplit < 1) nsplit = 1;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks, (unsigned)nsplit);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (t32) return cudaLaunchKernelEx(&cfg, simt_gemm_kernel<32>, a, n32);
    return cudaLaunchKernelEx(&cfg, simt_gemm_kernel<64>, a, n64);
}

// ------------------------------------------------------------------ LayerNorm (no affine)
// v = h + m + l with h, m, l bf16: each the nearest bf16 of what the previous parts leave over (the
// remainders are exact in fp32), so that the three carry v's 24 significant bits.
__device__ __forceinline__ void split3_bf16(float v, uint16_t* p) {
    p[0] = f32_to_bf16(v);
    const float r1 = v - bf16_to_f32(p[0]);
    p[1] = f32_to_bf16(r1);
    p[2] = f32_to_bf16(r1 - bf16_to_f32(p[1]));
}
// Lane j < LN_AUG_K / 8 of a warp writes columns 8 j .. 8 j + 7 of an augmentation row: v0..v8 in
// columns 0..8, zeros after them.
__device__ __forceinline__ void store_aug_row(uint16_t* row, int lane, uint16_t v0, uint16_t v1, uint16_t v2,
                                              uint16_t v3, uint16_t v4, uint16_t v5, uint16_t v6, uint16_t v7,
                                              uint16_t v8) {
    uint4 u = make_uint4(0, 0, 0, 0);
    if (lane == 0)
        u = make_uint4((uint32_t)v0 | ((uint32_t)v1 << 16), (uint32_t)v2 | ((uint32_t)v3 << 16),
                       (uint32_t)v4 | ((uint32_t)v5 << 16), (uint32_t)v6 | ((uint32_t)v7 << 16));
    else if (lane == 1)
        u.x = v8;
    reinterpret_cast<uint4*>(row)[lane] = u;
}

// One warp per token row; fp32 statistics in two passes over registers (mean, then the biased
// variance of the centred values); x = (y - mean) / sqrt(var + 1e-6).
// STATS (the LayerNorm folded into its consumers): warp rows [0, T) write (mean, 1 / sqrt(var +
// 1e-6)) of row `row` of y to x as float2; the warp rows after them sum the rows of the weight
// matrices in w (c[n] = sum_k W[n, k], d columns each), in the same chunk order and warp tree.
template <bool BF16, bool STATS>
__global__ void __launch_bounds__(256) layer_norm_kernel(const void* y, void* x, int64_t T, int d, const LnSums w) {
    pdl_wait();  // y is the previous kernel's output; the sums' buffers may still be read by it
    pdl_launch_dependents();  // the next sublayer's first kernel may set itself up meanwhile
    const int lane = threadIdx.x & 31;
    int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    const void* src = y;
    float* csum = nullptr;  // a weight row: its sum goes to csum[row]
    if (row >= T) {
        if constexpr (!STATS) return;
        int64_t wr = row - T;
        int m = 0;
        while (m < 2 && wr >= w.rows[m]) wr -= w.rows[m++];
        if (m == 2) return;
        src = w.W[m];
        csum = w.c[m];
        row = wr;
    }
    constexpr int VEC = BF16 ? 8 : 4;  // elements per 16-byte chunk
    constexpr int MAXC = 4;            // chunks per lane: d <= 32 * MAXC * VEC
    float v[MAXC][VEC];
    const int nch = d / VEC;
    float sum = 0.f;
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
        const int ch = lane + 32 * c;
        if (ch < nch) {
            const uint4 u = reinterpret_cast<const uint4*>(
                static_cast<const unsigned char*>(src) + (row * d + (int64_t)ch * VEC) * (BF16 ? 2 : 4))[0];
            if constexpr (BF16) {
                const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    v[c][2 * j] = bf16_lo(w[j]);
                    v[c][2 * j + 1] = bf16_hi(w[j]);
                }
            } else {
                v[c][0] = __uint_as_float(u.x);
                v[c][1] = __uint_as_float(u.y);
                v[c][2] = __uint_as_float(u.z);
                v[c][3] = __uint_as_float(u.w);
            }
#pragma unroll
            for (int j = 0; j < VEC; ++j) sum += v[c][j];
        }
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
    if (STATS && csum) {
        if (lane == 0) csum[row] = sum;
        if (csum == w.c[0] && w.aug_w0 && lane < LN_AUG_K / 8) {  // W[0]'s augmentation row
            uint16_t p[3];
            split3_bf16(sum, p);
            store_aug_row(w.aug_w0 + row * LN_AUG_K, lane, p[0], p[1], p[2], p[0], p[1], p[2], p[0], p[1], p[2]);
        }
        return;
    }
    const float mean = sum / (float)d;
    float sq = 0.f;
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
        if (lane + 32 * c < nch) {
#pragma unroll
            for (int j = 0; j < VEC; ++j) {
                const float t = v[c][j] - mean;
                sq += t * t;
            }
        }
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
    const float inv = 1.0f / sqrtf(sq / (float)d + 1e-6f);
    if constexpr (STATS) {
        if (lane == 0) static_cast<float2*>(x)[row] = make_float2(mean, inv);
        if (w.aug_tok && lane < LN_AUG_K / 8) {  // the token's augmentation row: -mean in 3 parts
            uint16_t p[3];
            split3_bf16(-mean, p);
            store_aug_row(w.aug_tok + row * LN_AUG_K, lane, p[0], p[0], p[0], p[1], p[1], p[1], p[2], p[2], p[2]);
        }
        return;
    }
#pragma unroll
    for (int c = 0; c < MAXC; ++c) {
        const int ch = lane + 32 * c;
        if (ch < nch) {
            uint4 u;
            if constexpr (BF16) {
                uint32_t w[4];
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    w[j] = pack_bf16((v[c][2 * j] - mean) * inv, (v[c][2 * j + 1] - mean) * inv);
                u = make_uint4(w[0], w[1], w[2], w[3]);
            } else {
                u = make_uint4(__float_as_uint((v[c][0] - mean) * inv), __float_as_uint((v[c][1] - mean) * inv),
                               __float_as_uint((v[c][2] - mean) * inv), __float_as_uint((v[c][3] - mean) * inv));
            }
            reinterpret_cast<uint4*>(static_cast<unsigned char*>(x) +
                                     (row * d + (int64_t)ch * VEC) * (BF16 ? 2 : 4))[0] = u;
        }
    }
}

static void pdl_config(cudaLaunchConfig_t& cfg, cudaLaunchAttribute* attr, unsigned grid, cudaStream_t s) {
    cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
}

cudaError_t launch_layer_norm(const void* y, void* x, int64_t T, int d, int dtype, cudaStream_t s) {
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr[1];
    pdl_config(cfg, attr, (unsigned)((T + 7) / 8), s);
    const LnSums none = {};
    if (dtype == CLEARMOE_BF16) return cudaLaunchKernelEx(&cfg, layer_norm_kernel<true, false>, y, x, T, d, none);
    return cudaLaunchKernelEx(&cfg, layer_norm_kernel<false, false>, y, x, T, d, none);
}

cudaError_t launch_ln_prep(const void* y, float2* stats, int64_t T, int d, const LnSums& w, int dtype, cudaStream_t s) {
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr[1];
    pdl_config(cfg, attr, (unsigned)((T + w.rows[0] + w.rows[1] + 7) / 8), s);
    void* out = stats;
    if (dtype == CLEARMOE_BF16) return cudaLaunchKernelEx(&cfg, layer_norm_kernel<true, true>, y, out, T, d, w);
    return cudaLaunchKernelEx(&cfg, layer_norm_kernel<false, true>, y, out, T, d, w);
}

}  // namespace cm
