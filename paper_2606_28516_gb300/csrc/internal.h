// Host-side launchers shared between the translation units of the library (not part of the ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace cm {

struct RouteArgs {
    const void* x;
    int64_t T;
    int d;
    int E;
    int dtype;  // clearmoe_dtype
    const void* Wg;
    const void* bg;
    int32_t* idx;
    int32_t* perm;
    int32_t* inv;                  // nullable: inv[token] = slot, the inverse of perm
    int32_t* counts;
    int32_t* offsets;
    int32_t* cta_counts;           // [grid x CM_MAX_E] per-CTA-range expert counts
    int32_t* tinfo;                // [T] per token: expert | rank within its CTA range << 8 (may be idx)
    int debug_skip;                // fault injection: CTA 0 withholds this stage (-1: none)
    int64_t wait_limit_ns;
    int32_t* status;
    // > 0: token t with t % cls_stride == 0 is a class token: it skips the router and forms group
    // E (idx = E), the dense path, whose slots follow every expert's: T - n_cls + t / cls_stride
    int64_t cls_stride;
    int w_bf16;  // fp32 tokens (the MLP router's hidden layer) with bf16 W_g and b_g
    // x is the un-normalised stream y (nullable = x is the router's input as is): logits
    // rstd_t (W_g y_t - mean_t g) + b_g with (mean_t, rstd_t) = ln_stats[t], g_e = ln_wsum[e] = sum_k W_g[e, k]
    const float2* ln_stats;
    const float* ln_wsum;
};
// Class tokens of T: every cls_stride-th from token 0 (none when cls_stride is 0).
__host__ __device__ inline int64_t n_class_tokens(int64_t T, int64_t cls_stride) {
    return cls_stride > 0 ? (T + cls_stride - 1) / cls_stride : 0;
}

// Grid of the routing kernel for T tokens (one or two CTAs per SM); chunk = rows per CTA (a
// routing range). Returns 0, -1 on a CUDA error, -2 when no launch shape fits.
int route_grid(int64_t T, int d, int E, int dtype, int num_sms, int* grid, int* chunk);
int route_max_ctas(int num_sms, int dtype, int d, int E);
// Phase 1 of the routing: idx, cta_counts and tinfo (no grid-wide step).
cudaError_t launch_route(const RouteArgs& a, int grid, int chunk, cudaStream_t s);
// The slots from the routing's output: counts, offsets, perm, inv (if set); unpacks idx when
// tinfo == idx. Same grid and chunk as the routing launch.
cudaError_t launch_route_finalize(const RouteArgs& a, int grid, int chunk, cudaStream_t s);

// ---- folding the shared basis into the experts: out[e] = U diag(S) Vh + res[e] ----
struct FoldArgs {
    const void* U;      // [d x r] layer dtype
    const float* S;     // [r]
    const void* Vh;     // [r x H] layer dtype
    const void* res[16];
    void* out[16];      // [d x H] each, layer dtype
    int d, H, r, E;
};
cudaError_t launch_fold_basis(const FoldArgs& a, int dtype, cudaStream_t s);

// ---- exact-fp32 SIMT GEMMs (fp32 layer) ----
struct SimtGemmArgs {
    // C[m, n] = epi(sum_k A0[rowA(m), k] B0[n, k] + sum_k A1[m, k] B1_e[n, k])
    const float* A0;
    int64_t lda0;
    int K0;
    const float* B0;
    const int32_t* a_rows;  // gather rows of A0 (nullable)
    const float* A1;
    int64_t lda1;
    int K1;
    const float* B1[16];     // grouped: per-expert B of the second segment; else B1[0]
    int64_t M;
    int N;
    const float* bias;   // + bias[n]
    int gelu;            // GELU after bias
    int relu;            // max(., 0) after bias
    const float* scale;  // * scale[n]
    float* C;
    int64_t ldc;
    const int32_t* c_rows;   // scatter rows of C (nullable)
    const int32_t* offsets;  // grouped: expert boundaries [E + 1] (nullable = not grouped)
    int E;
    int dense_last;          // grouped: the last group (the dense path) has no first K segment
    // row scale: C[m, :] *= group_scale[row_group[m]] (1 / that with row_scale_inv), m < M
    const int32_t* row_group;
    const float* group_scale;
    int scale_groups;
    int row_scale_inv;
    // the LayerNorm folded into A0 (A0 = un-normalised rows y): acc <- rstd (acc - mean c_n) before
    // the bias, with (mean, rstd) = ln_stats[A0's row] and c_n = ln_colsum[n] = sum_k B0[n, k]
    const float2* ln_stats;
    const float* ln_colsum;
    // split K for launches with too few tiles to fill the GPU: the K chain of each tile is cut into
    // up to SIMT_MAX_SPLIT ranges run by separate blocks, which write fp32 partial tiles to ws
    // (ws_floats floats); the last block of a tile (counter cnt[tile], cnt_len counters, zero
    // between launches) adds them in split order and runs the epilogue. Nullable: no split.
    float* ws;
    int64_t ws_floats;
    int* cnt;
    int cnt_len;
};
constexpr int SIMT_MAX_SPLIT = 8;
// Workspace of the split K: partial tiles of up to 4 blocks per SM of 64 x 64 outputs, and counters.
inline int64_t simt_ws_floats(int num_sms) { return (int64_t)4 * num_sms * 64 * 64; }
inline int simt_cnt_len(int num_sms) { return 4 * num_sms; }
cudaError_t launch_simt_gemm(const SimtGemmArgs& a, cudaStream_t s);

cudaError_t launch_layer_norm(const void* y, void* x, int64_t T, int d, int dtype, cudaStream_t s);
// Row sums of up to two weight matrices of d columns (layer dtype): c[m][n] = sum_k W[m][n, k], fp32.
// aug_tok / aug_w0 (nullable, bf16, LN_AUG_K columns per row): the augmentation K block of a GEMM
// whose A rows are the un-normalised tokens and whose B rows are W[0]'s. With mean = h + m + l and
// c = h' + m' + l' split into bf16 parts (each the rounded remainder of the previous), a token row
// holds (-h, -h, -h, -m, -m, -m, -l, -l, -l, 0, ...) and a weight row (h', m', l', h', m', l', h', m',
// l', 0, ...), so that their 9 exact products sum to -mean c in the tensor cores' fp32 accumulator.
constexpr int LN_AUG_K = 64;
struct LnSums {
    const void* W[2];
    float* c[2];
    int64_t rows[2];
    uint16_t* aug_tok;
    uint16_t* aug_w0;
};
// The LayerNorm folded into its consumers, one launch: stats[t] = (mean, 1 / sqrt(var + 1e-6)) of
// every row of y [T x d], and the row sums w of the weights that multiply the normalised rows.
cudaError_t launch_ln_prep(const void* y, float2* stats, int64_t T, int d, const LnSums& w, int dtype, cudaStream_t s);

// ---- tcgen05 bf16 GEMMs ----
enum TcEpi { TC_EPI_BIAS_GELU = 0, TC_EPI_SCALE = 1, TC_EPI_STORE = 2, TC_EPI_SCATTER = 3, TC_EPI_BIAS_RELU = 4 };
enum TcMode { TC_DENSE = 0, TC_GATHER = 1, TC_GROUPED = 2 };

struct TcGemmArgs {
    int mode;  // TcMode
    int epi;   // TcEpi
    int64_t M;
    int N;
    int K0;
    int K1;  // second K segment (grouped only)
    CUtensorMap tmA0, tmA1, tmB0;
    CUtensorMap tmB1[16];
    const void* gather_src;    // gather: rows of A0 read directly (bf16 [.. x K0])
    int64_t gather_ld;         // elements
    const int32_t* rows;       // gather: A row of output row m; scatter (the 2-SM kernel: whenever
                               // set): C row of output row m
    const int32_t* offsets;    // grouped: [E + 1]
    int E;
    const void* bias;          // bf16 [N]
    const float* scale;        // fp32 [N]
    void* C;                   // bf16
    int64_t ldc;
    int32_t* status;
    int64_t wait_limit_ns;
    // 2-SM dense kernel only: output row m (a token) goes to its routing slot offsets[e] +
    // (tokens of e in ranges before m's) + rank, with (e, rank) = rt_info[m] packed as e | rank << 8
    // and m's range m / rt_chunk; the kernel forms the prefix table from rt_counts ([rt_ctas x
    // CM_MAX_E], rt_ctas <= 256, rt_ctas * rt_E <= TC2_TAB_CAP) and writes perm, counts, offsets.
    const int32_t* rt_info;
    const int32_t* rt_counts;
    int rt_ctas, rt_chunk, rt_E;
    int32_t* rt_perm;
    int32_t* rt_out_counts;
    int32_t* rt_out_offsets;
    // store / scatter epilogues: + out_bias[n] (bf16 [N], nullable; the 2-SM kernel stages it in
    // shared memory, N <= TC2_BIAS_CAP)
    const void* out_bias;
    // grouped: the last of the E groups is the dense path (class tokens), whose K chain is the
    // z x B1 segment alone
    int dense_last;
    // fused fc1: class tokens (t % rt_cls_stride == 0) go to slot M - n_cls + t / rt_cls_stride
    int64_t rt_cls_stride;
    // C is fp32 (stored as computed, no rounding): the MLP router's hidden layer
    int c_f32;
    // row scale applied last: output row m (before any scatter) times group_scale[row_group[m]]
    // (its reciprocal with row_scale_inv); a group index outside [0, scale_groups) scales by 1.
    // Grouped mode with offsets == nullptr is a single group [0, M).
    const int32_t* row_group;
    const float* group_scale;
    int scale_groups;
    int row_scale_inv;
    // 2-SM kernel, launch overlap with the previous kernel (programmatic dependent launch):
    // pdl_wait_role 0: every thread waits for it after the setup; 1: only the epilogue warps wait
    // (their routing table and slots are its results; the operand loads and MMAs start at once);
    // 2: only the producer waits, before its first load of the K0 (t) segment (the z segment and the
    // epilogue need nothing from it). pdl_trigger_late: release the next kernel only after the wait,
    // so that it starts once this kernel's own predecessors have completed.
    int pdl_wait_role;
    int pdl_trigger_late;
    // 2-SM kernel: A tiles loaded with the L2 evict-first policy (a stream read once), so that they
    // displace one another rather than lines the next reads are still to find in L2
    int a_evict_first;
    // The LayerNorm folded into A (A = un-normalised rows y; single-segment modes): the accumulator
    // becomes rstd (acc - mean c_n) before the epilogue, with (mean, rstd) = ln_stats[A's row] (the
    // gathered row in TC_GATHER) and c_n = ln_colsum[n] = sum_k B[n, k]; nullable
    const float2* ln_stats;
    const float* ln_colsum;
    // TC_DENSE: one more K block after K0, A from tmA1 and B from tmB1[0] (the LayerNorm
    // augmentation blocks of LnSums, 16 useful columns), which adds -mean c to the accumulator;
    // with ln_stats set and ln_colsum null the epilogue then only scales by rstd, inside the bias
    // add (BIAS_GELU / BIAS_RELU)
    int ln_aug;
    // 2-SM dense kernel: the linear router inside fc1 (fr_E > 0, E <= 16). Every 256-row pair tile
    // gets one more unit whose B is W_g (tmR: [E x K0], boxes of 16 rows, rows past E read as zero)
    // and whose MMA is 256 x 32 over the same A tiles; its epilogue adds b_g (fr_bias, bf16), takes
    // the argmax (lowest index on ties) and writes, per token t, fr_idx[t] = e and fr_info[t] =
    // e | rank << 8 (rank among the earlier tokens of e in t's 128-row range t / 128), and per range
    // c the expert counts fr_counts[c * CM_MAX_E + e] (ranges c < ceil(M / 128)).
    CUtensorMap tmR;
    int fr_E;
    const void* fr_bias;
    int32_t* fr_idx;
    int32_t* fr_info;
    int32_t* fr_counts;
    // grouped mode: the z segment's A rows gathered by slot, A row of slot m = a1_rows[m] (perm),
    // by tile::gather4 loads of four rows each; tmA1 then has boxes one row high
    const int32_t* a1_rows;
    // 2-SM dense mode at 256-wide tiles: 12 epilogue warps (three per TMEM lane quarter) and a 160 KB
    // operand ring instead of 8 warps and 192 KB, for short K where the epilogue bounds a tile
    int epi12;
    // 1-SM kernel, dense and grouped modes: fp32 operands (tensor maps from encode_tmap_f32) on the
    // TF32 tensor cores with three products per K step (hi hi + hi lo + lo hi, each fp32 operand split
    // into a TF32 part and its remainder in shared memory); bias, out_bias and C are fp32 (c_f32
    // set), GELU is gelu_erf; no LayerNorm fold
    int tf32;
    // fp32 (TF32) variant: each tile's K blocks split into ksplit ranges (> 1 when tiles alone leave
    // SMs idle), one unit each; a unit stores its fp32 partial tile in ws ([tiles x ksplit x 128 x BN]),
    // and the tile's last unit (cnt[tile] counts arrivals and is reset by it) adds the partials in
    // split order and runs the epilogue: deterministic for a given shape
    int ksplit;
    int bn_tf32;  // the N tile the B maps were encoded for (tc_plan_tf32)
    float* ws;
    int64_t ws_floats;
    int* cnt;
    int cnt_len;
};
// fc1 takes the 12-epilogue-warp kernel up to this K (d): there a 256 x 256 tile's MMAs are short
// beside its bias + GELU epilogue
constexpr int TC2_EPI12_MAX_K = 512;
// Rows of one routing range of the router inside fc1 (a CTA's half of a pair tile).
constexpr int FR_RANGE = 128;
// Boundary e of a grouped GEMM's groups: offsets[e], or the single group [0, M) without offsets.
__host__ __device__ inline int64_t tc_group_off(const TcGemmArgs& a, int e) {
    return a.offsets ? (int64_t)a.offsets[e] : (e == 0 ? 0 : a.M);
}
#ifdef __CUDACC__
// The row scale of output row m (1 without group_scale or for an out-of-range group index).
__device__ __forceinline__ float tc_row_scale(const TcGemmArgs& a, int64_t m) {
    if (!a.group_scale) return 1.f;
    const int g = a.row_group[m];
    if ((unsigned)g >= (unsigned)a.scale_groups) return 1.f;
    const float s = a.group_scale[g];
    return a.row_scale_inv ? 1.f / s : s;
}
#endif
int tc_pick_bn(int mode, int N);
// N tile and K split of the 1-SM kernel's fp32 (TF32) variant for an [m_tiles x 128] x N x K
// product: of the widths 128, 64, 32, 16 dividing N, the one (with the K split that fills the SMs,
// at most 8 ways, at least 4 K blocks each, within ws_floats and cnt_len) whose busiest SM moves
// the fewest bytes; bn = 0 if none divides N
struct TcTf32Plan {
    int bn;
    int ksplit;
};
TcTf32Plan tc_plan_tf32(int N, int K, int64_t m_tiles, int num_sms, int64_t ws_floats, int cnt_len);
// 2-SM (cta_group::2) variant for the dense and grouped modes: 256 x BN tiles per CTA pair, BN =
// tc2_pick_bn(mode, N) (256, 192 or 128; 0 = shape not supported; each CTA's B box is BN / 2 rows).
// Its bias + GELU and column-scale epilogues stage the vector in shared memory (N <= TC2_BIAS_CAP).
constexpr int TC2_BIAS_CAP = 4096;
constexpr int TC2_TAB_CAP = 2432;  // routing prefix table entries (ranges x experts)
int tc2_pick_bn(int mode, int N);
cudaError_t launch_tc_gemm2(const TcGemmArgs& a, int num_sms, cudaStream_t s);
cudaError_t launch_tc_gemm(const TcGemmArgs& a, int num_sms, cudaStream_t s);

// cudaFuncSetAttribute(fn, MaxDynamicSharedMemorySize, bytes) once per (current device, fn): the
// attribute belongs to a device, so a process that launches on several GPUs sets it on each.
cudaError_t smem_attr_once(const void* fn, int bytes);
// SM count of the current device, queried once per device (0 on a CUDA error).
int current_device_sms();

// Encode a 2-D bf16 row-major [rows x cols] tensor map, box {64, box_rows}, 128-byte swizzle.
int encode_tmap_bf16(CUtensorMap* map, const void* base, int64_t rows, int64_t cols,
                     int box_rows);
// The same [rows x cols] matrix (cols % 64 == 0) viewed as {64 columns, rows, cols / 64 chunks}
// with boxes of 64 x box_rows x box_chunks, 128-byte swizzle: a box lands in shared memory as
// box_chunks consecutive [box_rows x 64] tiles (one K block each) and reads box_chunks x 128
// contiguous bytes of each of its rows.
int encode_tmap_bf16_chunks(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows,
                            int box_chunks);
// Encode a 2-D fp32 row-major [rows x cols] tensor map (cols % 4 == 0), box {32, box_rows}
// (128-byte rows), 128-byte swizzle.
int encode_tmap_f32(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows);

}  // namespace cm
