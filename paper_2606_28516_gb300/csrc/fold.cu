// Folding the shared basis into the residual experts: W_e^comb = U_r diag(S_r) V_r^T + W_e^res.
//
// Eq. 2 sums a shared and a per-expert term on the same hidden state, y = W_shared z + W_e^res z,
// so y = W_e^comb z with W_e^comb = W_shared + W_e^res, which turns the forward into one grouped
// GEMM over z (the dense FFN's arithmetic) with no basis step. This kernel forms the combined
// weights once per weight set: each CTA computes a 64 x 64 tile of W_shared = U_r diag(S_r) Vh_r in
// fp32 (products S_r[k] Vh_r[k][h] in fp32, fma over k ascending), then adds it to the same tile of
// every expert's residual (none when res[e] is null: W_shared materialised alone) and rounds once
// to the layer dtype.
#include "common.cuh"
#include "internal.h"

namespace cm {
namespace {

constexpr int FT = 64;  // output tile (rows of d x columns of H)
constexpr int FK = 16;  // k step

template <bool BF16>
__device__ __forceinline__ float load_elem(const void* p, int64_t i) {
    if constexpr (BF16)
        return bf16_to_f32(static_cast<const uint16_t*>(p)[i]);
    else
        return static_cast<const float*>(p)[i];
}

template <bool BF16>
__global__ void __launch_bounds__(256) fold_basis_kernel(const FoldArgs a) {
    __shared__ float Us[FK][FT + 1];  // U_r[i0 + i][k0 + k] at [k][i]
    __shared__ float Vs[FK][FT + 1];  // S_r[k0 + k] Vh_r[k0 + k][h0 + h] at [k][h]
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int i0 = blockIdx.y * FT, h0 = blockIdx.x * FT;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < a.r; k0 += FK) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int idx = tid + 256 * q;
            const int ii = idx >> 4, kk = idx & 15;  // U: 64 rows x 16 k
            const int i = i0 + ii, k = k0 + kk;
            Us[kk][ii] = (i < a.d && k < a.r) ? load_elem<BF16>(a.U, (int64_t)i * a.r + k) : 0.f;
            const int kv = idx >> 6, hh = idx & 63;  // Vh: 16 k x 64 columns
            const int kr = k0 + kv, h = h0 + hh;
            Vs[kv][hh] = (kr < a.r && h < a.H) ? a.S[kr] * load_elem<BF16>(a.Vh, (int64_t)kr * a.H + h) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < FK; ++kk) {
            float av[4], bv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) av[i] = Us[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) bv[j] = Vs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }
    for (int e = 0; e < a.E; ++e) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int row = i0 + ty * 4 + i;
            if (row >= a.d) continue;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int col = h0 + tx * 4 + j;
                if (col >= a.H) continue;
                const int64_t off = (int64_t)row * a.H + col;
                const float v = a.res[e] ? acc[i][j] + load_elem<BF16>(a.res[e], off) : acc[i][j];
                if constexpr (BF16)
                    static_cast<uint16_t*>(a.out[e])[off] = f32_to_bf16(v);
                else
                    static_cast<float*>(a.out[e])[off] = v;
            }
        }
    }
}

}  // namespace

cudaError_t launch_fold_basis(const FoldArgs& a, int dtype, cudaStream_t s) {
    const dim3 grid((unsigned)((a.H + FT - 1) / FT), (unsigned)((a.d + FT - 1) / FT));
    if (dtype == CLEARMOE_BF16)
        fold_basis_kernel<true><<<grid, 256, 0, s>>>(a);
    else
        fold_basis_kernel<false><<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace cm
