// C ABI of the CLEAR-MoE FFN layer (include/clearmoe.h): handle, workspace, argument checks, and
// the launch sequence of each call. No compute happens here; every step runs in a kernel.
#include <cstdio>
#include <cstring>
#include <new>

#include "common.cuh"
#include "internal.h"

struct clearmoe_layer {
    clearmoe_layer_desc desc;
    int device;
    int num_sms;
    size_t esz;
    // workspace (device)
    void* z;            // [max_tokens x hidden]  hidden states, expert-sorted order
    void* t;            // [max_tokens x max_r]   shared-basis coefficients
    int32_t* idx;       // [max_tokens]
    int32_t* perm;      // [max_tokens]  perm[slot] = token
    int32_t* inv;       // [max_tokens]  inv[token] = slot
    int32_t* counts;    // [CM_MAX_E]
    int32_t* offsets;   // [CM_MAX_E + 1]
    int32_t* cta_counts;  // [route_max_ctas x CM_MAX_E] the routing kernel's per-range histograms
    int32_t* tinfo;       // [max_tokens] per token: expert | rank within its routing range << 8
    int32_t* status;
    float2* ln_stats;  // [max_tokens]  (mean, rstd) per token when the input LayerNorm is folded
    float* ln_sums;    // [2 hidden + CM_MAX_E]  row sums of W1, then of the router's first matrix
    uint16_t* ln_aug_x;  // bf16 layers: [max_tokens x LN_AUG_K]  fc1's augmentation block, token side
    uint16_t* ln_aug_w;  // bf16 layers: [hidden x LN_AUG_K]      and W1's side
    float* simt_ws;      // fp32 layers: the SIMT GEMMs' split-K partial tiles [simt_ws_floats]
    int* simt_cnt;       // fp32 layers: their per-tile counters [simt_cnt_len], zero between launches
    int64_t wait_limit_ns;
    int32_t phantom;  // fault injection: > 0 makes the routing withhold one stage copy
    cm::RouteArgs rt;  // the last routing launch (its consumers reuse the shape)
    int rt_grid, rt_chunk;
    int64_t last_T;
    int32_t last_E;
    int32_t last_groups;  // last_E, + 1 when class tokens formed the dense path's group
    cudaEvent_t prof[8];
    int32_t prof_n;
};

namespace {

using cm::encode_tmap_bf16;
using cm::encode_tmap_f32;

inline bool misaligned(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; }

int cuda_fail(cudaError_t e) {
    if (e == cudaSuccess) return CLEARMOE_OK;
    (void)cudaGetLastError();
    return CLEARMOE_ECUDA;
}

// The fp32 layers' SIMT GEMMs, with the handle's split-K workspace.
// The fp32 tensor-core GEMMs' tiling: N tile and K split for an [M x N] x K product (row tiles:
// ceil(M / 128) + extra), with the handle's split workspace and counters (fp32 layers own them).
cm::TcTf32Plan tf32_plan(const clearmoe_layer* L, cm::TcGemmArgs& g, int N, int K, int64_t M, int extra_tiles) {
    g.tf32 = 1;
    g.c_f32 = 1;
    g.ws = L->simt_ws;
    g.ws_floats = L->simt_ws ? cm::simt_ws_floats(L->num_sms) : 0;
    g.cnt = L->simt_cnt;
    g.cnt_len = L->simt_cnt ? cm::simt_cnt_len(L->num_sms) : 0;
    const cm::TcTf32Plan p = cm::tc_plan_tf32(N, K, (M + 127) / 128 + extra_tiles, L->num_sms, g.ws_floats, g.cnt_len);
    g.bn_tf32 = p.bn;
    g.ksplit = p.ksplit;
    return p;
}

int launch_simt(clearmoe_layer* L, cm::SimtGemmArgs& g, cudaStream_t s) {
    g.ws = L->simt_ws;
    g.ws_floats = L->simt_ws ? cm::simt_ws_floats(L->num_sms) : 0;
    g.cnt = L->simt_cnt;
    g.cnt_len = L->simt_cnt ? cm::simt_cnt_len(L->num_sms) : 0;
    return cuda_fail(cm::launch_simt_gemm(g, s));
}

void free_ws(clearmoe_layer* L) {
    void* ptrs[] = {L->z,     L->t,          L->idx,   L->perm,   L->inv,     L->counts,
                    L->offsets, L->cta_counts, L->tinfo, L->status, L->ln_stats, L->ln_sums,
                    L->ln_aug_x, L->ln_aug_w, L->simt_ws, L->simt_cnt};
    for (void* p : ptrs)
        if (p) cudaFree(p);
}

int check_common(const clearmoe_layer* L, const void* x, int64_t T) {
    if (!L || !x) return CLEARMOE_EINVAL;
    if (T < 1 || T > L->desc.max_tokens) return CLEARMOE_EINVAL;
    if (misaligned(x)) return CLEARMOE_EINVAL;
    return CLEARMOE_OK;
}

// The MLP router's hidden layer h = act(W_in x + b_in) [T x hidden], fp32, into the hidden-state
// workspace (free until fc1 runs): the tensor-core GEMM with an fp32-store epilogue, or the fp32
// SIMT GEMM on the fp32 layer.
// ln: x is the un-normalised stream; its LayerNorm is folded in (stats and W_in's row sums from ln_prep)
int mlp_hidden(clearmoe_layer* L, const void* x, int64_t T, const clearmoe_mlp_router* m, bool ln, cudaStream_t s) {
    const int d = L->desc.d, nh = m->hidden;
    const float2* lns = ln ? L->ln_stats : nullptr;
    const float* lnc = ln ? L->ln_sums + L->desc.hidden : nullptr;
    if (L->desc.dtype == CLEARMOE_F32) {
        cm::SimtGemmArgs g;
        std::memset(&g, 0, sizeof(g));
        g.A0 = static_cast<const float*>(x);
        g.lda0 = d;
        g.K0 = d;
        g.B0 = static_cast<const float*>(m->W_in);
        g.M = T;
        g.N = nh;
        g.bias = static_cast<const float*>(m->b_in);
        g.gelu = m->act == CLEARMOE_ACT_GELU;
        g.relu = m->act == CLEARMOE_ACT_RELU;
        g.C = static_cast<float*>(L->z);
        g.ldc = nh;
        g.ln_stats = lns;
        g.ln_colsum = lnc;
        return launch_simt(L, g, s);
    }
    cm::TcGemmArgs g;
    std::memset(&g, 0, sizeof(g));
    g.status = L->status;
    g.wait_limit_ns = L->wait_limit_ns;
    const int p = nh <= cm::TC2_BIAS_CAP ? cm::tc2_pick_bn(cm::TC_DENSE, nh) : 0;
    const int bn = cm::tc_pick_bn(cm::TC_DENSE, nh);
    if (!p && !bn) return CLEARMOE_EUNSUPPORTED;
    if (encode_tmap_bf16(&g.tmA0, x, T, d, 128) || encode_tmap_bf16(&g.tmB0, m->W_in, nh, d, p ? p / 2 : bn))
        return CLEARMOE_ECUDA;
    g.mode = cm::TC_DENSE;
    g.epi = m->act == CLEARMOE_ACT_GELU ? cm::TC_EPI_BIAS_GELU : cm::TC_EPI_BIAS_RELU;
    g.M = T;
    g.N = nh;
    g.K0 = d;
    g.bias = m->b_in;
    g.C = L->z;
    g.ldc = nh;
    g.c_f32 = 1;
    g.ln_stats = lns;
    g.ln_colsum = lnc;
    return cuda_fail(p ? cm::launch_tc_gemm2(g, L->num_sms, s) : cm::launch_tc_gemm(g, L->num_sms, s));
}

int check_mlp(const clearmoe_layer* L, const clearmoe_mlp_router* m, int E) {
    if (!m || !m->W_in || !m->b_in || !m->W_out || !m->b_out) return CLEARMOE_EINVAL;
    if (misaligned(m->W_in) || misaligned(m->b_in) || misaligned(m->W_out)) return CLEARMOE_EINVAL;
    if (m->act != CLEARMOE_ACT_RELU && m->act != CLEARMOE_ACT_GELU) return CLEARMOE_EINVAL;
    if (E < 1 || E > L->desc.max_E) return CLEARMOE_EINVAL;
    const bool bf16 = L->desc.dtype == CLEARMOE_BF16;
    if (m->hidden < 1 || m->hidden % (bf16 ? 16 : 4)) return CLEARMOE_EINVAL;
    if ((int64_t)m->hidden * 4 > (int64_t)L->esz * L->desc.hidden) return CLEARMOE_EINVAL;  // fits in z
    return CLEARMOE_OK;
}

int check_router(const clearmoe_layer* L, const clearmoe_router* router, int E);

// The router (linear, or the MLP router of the options) and the deployment options of a forward.
int check_router_and_options(const clearmoe_layer* L, const clearmoe_router* router, const clearmoe_ffn_options* opt,
                             int E) {
    const int rc = (opt && opt->mlp_router) ? check_mlp(L, opt->mlp_router, E) : check_router(L, router, E);
    if (rc) return rc;
    if (opt) {
        if (opt->cls_stride < 0 || opt->cls_stride > ((int64_t)1 << 30)) return CLEARMOE_EINVAL;
        if (opt->b2 && misaligned(opt->b2)) return CLEARMOE_EINVAL;
        if (opt->cls_stride > 0) {
            if (!opt->W2 || misaligned(opt->W2)) return CLEARMOE_EINVAL;
            if (E + 1 > CM_MAX_E) return CLEARMOE_EUNSUPPORTED;  // the dense path takes a group
        }
    }
    return CLEARMOE_OK;
}

// The LayerNorm of x folded into its consumers (input_layernorm): (mean, rstd) of every token row,
// the row sums of W1 and those of the router's matrix applied to x (W_g, or the MLP router's W_in),
// and in bf16 layers the augmentation block that carries -mean W1 1 into fc1's MMAs, in one launch
// ahead of the routing.
int ln_prep(clearmoe_layer* L, const void* y, int64_t T, const void* W1, const void* Wr, int rows_r, cudaStream_t s) {
    cm::LnSums w = {};
    w.W[0] = W1;
    w.c[0] = L->ln_sums;
    w.rows[0] = W1 ? L->desc.hidden : 0;
    w.W[1] = Wr;
    w.c[1] = L->ln_sums + L->desc.hidden;
    w.rows[1] = Wr ? rows_r : 0;
    w.aug_tok = L->ln_aug_x;  // null in fp32 layers
    w.aug_w0 = W1 ? L->ln_aug_w : nullptr;
    return cuda_fail(cm::launch_ln_prep(y, L->ln_stats, T, L->desc.d, w, L->desc.dtype, s));
}

// A 2-SM fc1 (or the dense FFN's) with the LayerNorm folded: the mean term enters as one more K
// block (LnSums' augmentation rows), and the epilogue scales by rstd inside its bias add.
int ln_fc1_aug(clearmoe_layer* L, cm::TcGemmArgs& g, int64_t T, int b_box) {
    g.ln_stats = L->ln_stats;
    g.ln_colsum = nullptr;
    g.ln_aug = 1;
    if (encode_tmap_bf16(&g.tmA1, L->ln_aug_x, T, cm::LN_AUG_K, 128) ||
        encode_tmap_bf16(&g.tmB1[0], L->ln_aug_w, L->desc.hidden, cm::LN_AUG_K, b_box))
        return CLEARMOE_ECUDA;
    return CLEARMOE_OK;
}

int do_route(clearmoe_layer* L, const void* x, int64_t T, const clearmoe_router* router,
             const clearmoe_mlp_router* mlp, int E, int64_t cls_stride, cudaStream_t s, bool ln = false) {
    // the MLP router: its hidden layer first, then the routing kernel on it (fp32 tokens)
    const int rd = mlp ? mlp->hidden : L->desc.d;
    const int rdtype = mlp ? CLEARMOE_F32 : L->desc.dtype;
    int grid = 0, chunk = 0;
    const int g = cm::route_grid(T, rd, E, rdtype, L->num_sms, &grid, &chunk);
    if (g) return g == -2 ? CLEARMOE_EUNSUPPORTED : CLEARMOE_ECUDA;
    if (grid > cm::route_max_ctas(L->num_sms, rdtype, rd, E)) return CLEARMOE_EUNSUPPORTED;
    if (mlp) {
        const int rc = mlp_hidden(L, x, T, mlp, ln, s);
        if (rc) return rc;
    }
    cm::RouteArgs& a = L->rt;
    std::memset(&a, 0, sizeof(a));
    a.x = mlp ? L->z : x;
    a.T = T;
    a.d = rd;
    a.E = E;
    a.dtype = rdtype;
    a.Wg = mlp ? mlp->W_out : router->W;
    a.bg = mlp ? mlp->b_out : router->b;
    a.w_bf16 = mlp && L->desc.dtype == CLEARMOE_BF16;
    a.idx = L->idx;
    a.perm = L->perm;
    a.inv = L->inv;
    a.counts = L->counts;
    a.offsets = L->offsets;
    a.cta_counts = L->cta_counts;
    a.tinfo = L->tinfo;
    a.debug_skip = L->phantom > 0 ? 0 : -1;
    a.wait_limit_ns = L->wait_limit_ns;
    a.status = L->status;
    a.cls_stride = cls_stride;
    if (ln && !mlp) {  // the MLP router folds it into its hidden layer instead
        a.ln_stats = L->ln_stats;
        a.ln_wsum = L->ln_sums + L->desc.hidden;
    }
    L->rt_grid = grid;
    L->rt_chunk = chunk;
    const int rc = cuda_fail(cm::launch_route(a, grid, chunk, s));
    if (rc == CLEARMOE_OK) {
        L->last_T = T;
        L->last_E = E;
        L->last_groups = E + (cls_stride > 0 ? 1 : 0);
    }
    return rc;
}

// counts, offsets, perm and inv from the last routing launch
int do_finalize(clearmoe_layer* L, cudaStream_t s) {
    return cuda_fail(cm::launch_route_finalize(L->rt, L->rt_grid, L->rt_chunk, s));
}

inline void mark(const clearmoe_layer* L, int i, cudaStream_t s) {
    if (i < L->prof_n && L->prof[i]) cudaEventRecord(L->prof[i], s);
}

int check_router(const clearmoe_layer* L, const clearmoe_router* router, int E) {
    if (!router || !router->W || !router->b) return CLEARMOE_EINVAL;
    if (misaligned(router->W)) return CLEARMOE_EINVAL;
    if (E < 1 || E > L->desc.max_E) return CLEARMOE_EINVAL;
    return CLEARMOE_OK;
}

}  // namespace

extern "C" {

const char* clearmoe_strerror(int status) {
    switch (status) {
        case CLEARMOE_OK: return "ok";
        case CLEARMOE_EINVAL: return "invalid argument";
        case CLEARMOE_EUNSUPPORTED: return "shape not supported by this build";
        case CLEARMOE_ECUDA: return "CUDA error";
        case CLEARMOE_ENOMEM: return "out of device memory";
        case CLEARMOE_ETIMEOUT: return "a bounded device-side wait timed out";
        default: return "unknown status";
    }
}

int clearmoe_version(void) { return 100; }

int clearmoe_layer_create(const clearmoe_layer_desc* desc, clearmoe_layer** out) {
    if (!desc || !out) return CLEARMOE_EINVAL;
    *out = nullptr;
    const clearmoe_layer_desc& D = *desc;
    if (D.max_tokens < 1 || D.d < 1 || D.hidden < 1 || D.max_E < 1 || D.max_r < 1) return CLEARMOE_EINVAL;
    if (D.dtype != CLEARMOE_F32 && D.dtype != CLEARMOE_BF16) return CLEARMOE_EINVAL;
    if (D.max_E > CM_MAX_E || D.max_r > CM_MAX_R) return CLEARMOE_EUNSUPPORTED;
    if (D.max_tokens > (int64_t)1 << 30) return CLEARMOE_EUNSUPPORTED;
    if (D.dtype == CLEARMOE_BF16) {
        if (D.d % 64 || D.hidden % 64 || D.d > 1024) return CLEARMOE_EUNSUPPORTED;
    } else {
        if (D.d % 4 || D.hidden % 4 || D.d > 512) return CLEARMOE_EUNSUPPORTED;
    }
    clearmoe_layer* L = new (std::nothrow) clearmoe_layer();
    if (!L) return CLEARMOE_ENOMEM;
    std::memset(L, 0, sizeof(*L));
    L->desc = D;
    L->esz = D.dtype == CLEARMOE_BF16 ? 2 : 4;
    L->wait_limit_ns = 1000000000LL;
    if (cudaGetDevice(&L->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&L->num_sms, cudaDevAttrMultiProcessorCount, L->device) != cudaSuccess) {
        delete L;
        (void)cudaGetLastError();
        return CLEARMOE_ECUDA;
    }
    const size_t T = (size_t)D.max_tokens;
    // per-range histograms: the routing kernel's ranges, or the 128-row ranges of the router
    // inside fc1, whichever are more
    size_t ncta = (size_t)cm::route_max_ctas(L->num_sms, D.dtype, D.d, D.max_E);
    const size_t nfr = (T + cm::FR_RANGE - 1) / cm::FR_RANGE;
    if (nfr > ncta) ncta = nfr;
    bool ok = cudaMalloc(&L->z, T * D.hidden * L->esz) == cudaSuccess &&
              cudaMalloc(&L->t, T * D.max_r * L->esz) == cudaSuccess &&
              cudaMalloc((void**)&L->idx, T * 4) == cudaSuccess &&
              cudaMalloc((void**)&L->perm, T * 4) == cudaSuccess &&
              cudaMalloc((void**)&L->inv, T * 4) == cudaSuccess &&
              cudaMalloc((void**)&L->counts, CM_MAX_E * 4) == cudaSuccess &&
              cudaMalloc((void**)&L->offsets, (CM_MAX_E + 1) * 4) == cudaSuccess &&
              cudaMalloc((void**)&L->cta_counts, ncta * CM_MAX_E * 4) == cudaSuccess &&
              cudaMalloc((void**)&L->tinfo, T * 4) == cudaSuccess &&
              cudaMalloc((void**)&L->status, 4) == cudaSuccess &&
              cudaMalloc((void**)&L->ln_stats, T * sizeof(float2)) == cudaSuccess &&
              cudaMalloc((void**)&L->ln_sums, (2 * (size_t)D.hidden + CM_MAX_E) * 4) == cudaSuccess &&
              (D.dtype != CLEARMOE_BF16 ||
               (cudaMalloc((void**)&L->ln_aug_x, T * cm::LN_AUG_K * 2) == cudaSuccess &&
                cudaMalloc((void**)&L->ln_aug_w, (size_t)D.hidden * cm::LN_AUG_K * 2) == cudaSuccess)) &&
              (D.dtype != CLEARMOE_F32 ||
               (cudaMalloc((void**)&L->simt_ws, (size_t)cm::simt_ws_floats(L->num_sms) * 4) == cudaSuccess &&
                cudaMalloc((void**)&L->simt_cnt, (size_t)cm::simt_cnt_len(L->num_sms) * 4) == cudaSuccess &&
                cudaMemset(L->simt_cnt, 0, (size_t)cm::simt_cnt_len(L->num_sms) * 4) == cudaSuccess));
    if (ok) {
        // index workspaces start at zero (valid rows), so no launch ever reads garbage indices
        ok = cudaMemset(L->status, 0, 4) == cudaSuccess && cudaMemset(L->perm, 0, T * 4) == cudaSuccess &&
             cudaMemset(L->inv, 0, T * 4) == cudaSuccess && cudaMemset(L->tinfo, 0, T * 4) == cudaSuccess &&
             cudaMemset(L->idx, 0, T * 4) == cudaSuccess &&
             cudaDeviceSynchronize() == cudaSuccess;
    }
    if (!ok) {
        const cudaError_t e = cudaGetLastError();
        free_ws(L);
        delete L;
        return e == cudaErrorMemoryAllocation ? CLEARMOE_ENOMEM : CLEARMOE_ECUDA;
    }
    *out = L;
    return CLEARMOE_OK;
}

int clearmoe_layer_destroy(clearmoe_layer* L) {
    if (!L) return CLEARMOE_OK;
    const cudaError_t e = cudaDeviceSynchronize();
    free_ws(L);
    delete L;
    return cuda_fail(e);
}

int clearmoe_route(clearmoe_layer* L, const void* x, int64_t T, const clearmoe_router* router, int32_t E,
                   void* stream) {
    int rc = check_common(L, x, T);
    if (rc) return rc;
    if ((rc = check_router(L, router, E))) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if ((rc = do_route(L, x, T, router, nullptr, E, 0, s))) return rc;
    return do_finalize(L, s);
}

int clearmoe_route_mlp(clearmoe_layer* L, const void* x, int64_t T, const clearmoe_mlp_router* mlp, int32_t E,
                       void* stream) {
    int rc = check_common(L, x, T);
    if (rc) return rc;
    if ((rc = check_mlp(L, mlp, E))) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if ((rc = do_route(L, x, T, nullptr, mlp, E, 0, s))) return rc;
    return do_finalize(L, s);
}

// The router inside fc1 (clearmoe_ffn_options.router_in_fc1), bf16 layers: fc1 runs in token
// order and every 256-row pair tile gets one more unit that multiplies the same x tiles by W_g, so
// the tokens are read once for both; its epilogue writes idx, each token's rank within its 128-row
// range and every range's expert counts. The slot kernel (route_finalize_kernel over those ranges)
// forms counts, offsets, perm and inv; the basis factor reads z in token order and stores each t
// row at its token's slot; the grouped GEMM gathers each expert's z rows by perm (four rows per TMA
// gather) and scatters its output rows back to token order, as in the default path.
static int ffn_router_in_fc1(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                             const void* U_r, const float* S_r, const void* Vh_r, const void* const* residual_e,
                             const clearmoe_router* router, int E, int r, const void* b2, void* out,
                             cudaStream_t s) {
    const bool factored = U_r != nullptr;
    const int d = L->desc.d, H = L->desc.hidden;
    const int p1 = H <= cm::TC2_BIAS_CAP ? cm::tc2_pick_bn(cm::TC_DENSE, H) : 0;
    const int p3 = cm::tc2_pick_bn(cm::TC_GROUPED, d);
    const int p2 = factored ? cm::tc2_pick_bn(cm::TC_DENSE, r) : 0;
    const int bn2 = factored ? cm::tc_pick_bn(cm::TC_DENSE, r) : 1;
    if (L->desc.dtype != CLEARMOE_BF16 || !p1 || !p3 || !bn2) return CLEARMOE_EUNSUPPORTED;
    const int G = (int)((T + cm::FR_RANGE - 1) / cm::FR_RANGE);  // 128-row ranges
    int rc;
    mark(L, 0, s);
    cm::TcGemmArgs g;
    std::memset(&g, 0, sizeof(g));
    g.status = L->status;
    g.wait_limit_ns = L->wait_limit_ns;
    if (encode_tmap_bf16(&g.tmA0, x, T, d, 128) || encode_tmap_bf16(&g.tmB0, W1, H, d, p1 / 2) ||
        encode_tmap_bf16(&g.tmR, router->W, E, d, 16))
        return CLEARMOE_ECUDA;
    g.mode = cm::TC_DENSE;
    g.epi = cm::TC_EPI_BIAS_GELU;
    g.M = T;
    g.N = H;
    g.K0 = d;
    g.bias = b1;
    g.C = L->z;  // token order
    g.ldc = H;
    g.fr_E = E;
    g.fr_bias = router->b;
    g.fr_idx = L->idx;
    g.fr_info = L->tinfo;
    g.fr_counts = L->cta_counts;
    g.pdl_wait_role = 0;  // x may be the previous kernel's output
    if ((rc = cuda_fail(cm::launch_tc_gemm2(g, L->num_sms, s)))) return rc;
    mark(L, 1, s);
    cm::RouteArgs& a = L->rt;  // the slots from the 128-row ranges
    std::memset(&a, 0, sizeof(a));
    a.T = T;
    a.d = d;
    a.E = E;
    a.dtype = CLEARMOE_BF16;
    a.idx = L->idx;
    a.perm = L->perm;
    a.inv = L->inv;
    a.counts = L->counts;
    a.offsets = L->offsets;
    a.cta_counts = L->cta_counts;
    a.tinfo = L->tinfo;
    a.debug_skip = -1;
    a.wait_limit_ns = L->wait_limit_ns;
    a.status = L->status;
    L->rt_grid = G;
    L->rt_chunk = cm::FR_RANGE;
    if ((rc = cuda_fail(cm::launch_route_finalize(a, G, cm::FR_RANGE, s)))) return rc;
    L->last_T = T;
    L->last_E = E;
    L->last_groups = E;
    mark(L, 2, s);
    if (factored) {  // t = diag(S_r) Vh_r z, z in token order, each t row stored at its slot (inv)
        cm::TcGemmArgs g2;
        std::memset(&g2, 0, sizeof(g2));
        g2.status = L->status;
        g2.wait_limit_ns = L->wait_limit_ns;
        if (encode_tmap_bf16(&g2.tmA0, L->z, T, H, 128) || encode_tmap_bf16(&g2.tmB0, Vh_r, r, H, p2 ? p2 / 2 : bn2))
            return CLEARMOE_ECUDA;
        g2.mode = cm::TC_DENSE;
        g2.epi = cm::TC_EPI_SCALE;
        g2.M = T;
        g2.N = r;
        g2.K0 = H;
        g2.scale = S_r;
        g2.C = L->t;
        g2.ldc = r;
        g2.rows = L->inv;
        g2.a_evict_first = 1;
        // z is complete once the slot kernel releases this one (it waits for fc1 first): the loads
        // and MMAs start at once, the epilogue waits for the slots
        g2.pdl_wait_role = 1;
        g2.pdl_trigger_late = 1;
        rc = cuda_fail(p2 ? cm::launch_tc_gemm2(g2, L->num_sms, s) : cm::launch_tc_gemm(g2, L->num_sms, s));
        if (rc) return rc;
    }
    mark(L, 3, s);
    cm::TcGemmArgs g3;
    std::memset(&g3, 0, sizeof(g3));
    g3.status = L->status;
    g3.wait_limit_ns = L->wait_limit_ns;
    const int box3 = p3 / 2;
    if ((factored && (encode_tmap_bf16(&g3.tmA0, L->t, T, r, 128) || encode_tmap_bf16(&g3.tmB0, U_r, d, r, box3))) ||
        encode_tmap_bf16(&g3.tmA1, L->z, T, H, 1))  // one-row boxes: the z rows are gathered
        return CLEARMOE_ECUDA;
    for (int e = 0; e < E; ++e)
        if (encode_tmap_bf16(&g3.tmB1[e], residual_e[e], d, H, box3)) return CLEARMOE_ECUDA;
    g3.out_bias = b2;
    // after the basis kernel (released once the slots exist) the z segments may start at once; with
    // no basis kernel the slot kernel precedes this one and every thread waits for it
    g3.pdl_wait_role = factored ? 2 : 0;
    g3.mode = cm::TC_GROUPED;
    g3.epi = cm::TC_EPI_SCATTER;
    g3.M = T;
    g3.N = d;
    g3.K0 = factored ? r : 0;
    g3.K1 = H;
    g3.offsets = L->offsets;
    g3.E = E;
    g3.rows = L->perm;
    g3.a1_rows = L->perm;
    g3.C = out;
    g3.ldc = d;
    rc = cuda_fail(cm::launch_tc_gemm2(g3, L->num_sms, s));
    mark(L, 4, s);
    return rc;
}

// fp32 layers on the tensor cores (the 1-SM kernel's TF32 variant: three TF32 products per K step,
// their accuracy stated at the head of tc_gemm.cu), after the routing:
//   fc1: z[slot(t)] = GELU(W1 x_t + b1), x read in token order, each row stored at its slot (formed
//   in the epilogue from the routing's per-range counts and ranks when `fused`, else inv[t] from
//   the finalize kernel);
//   basis (factorised): t = diag(S_r) Vh_r z over the routed slots;
//   grouped: out[perm[slot]] = [t | z] [U_r | W_e^res]^T + b2 per group (materialised: [z | z] x
//   [W_sh | W_e^res]; folded: z x W_e^comb alone; class tokens: z x W2 alone).
// Needs d, H (and r when factorised) multiples of 16; the caller falls back to the SIMT kernels
// otherwise.
static bool f32_tc_ok(int d, int H, int r, bool factored) {
    return d % 16 == 0 && H % 16 == 0 && (!factored || r % 16 == 0);
}

static int ffn_f32_tc(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1, const void* U_r,
                      const float* S_r, const void* Vh_r, const void* W_sh, const void* const* residual_e, int E,
                      int r, int64_t n_cls, int64_t cls_stride, int G, const void* b2, const void* W2, bool fused,
                      void* out, cudaStream_t s) {
    const bool factored = U_r != nullptr;
    const bool materialized = !factored && W_sh != nullptr;
    const int d = L->desc.d, H = L->desc.hidden;
    int rc;
    cm::TcGemmArgs g;
    std::memset(&g, 0, sizeof(g));
    g.status = L->status;
    g.wait_limit_ns = L->wait_limit_ns;
    const int bn1 = tf32_plan(L, g, H, d, T, 0).bn;
    if (encode_tmap_f32(&g.tmA0, x, T, d, 128) || encode_tmap_f32(&g.tmB0, W1, H, d, bn1)) return CLEARMOE_ECUDA;
    g.mode = cm::TC_DENSE;
    g.epi = cm::TC_EPI_BIAS_GELU;
    g.M = T;
    g.N = H;
    g.K0 = d;
    g.bias = b1;
    if (fused) {  // slots from the routing's per-range counts and ranks; writes perm, counts, offsets
        g.rt_info = L->tinfo;
        g.rt_counts = L->cta_counts;
        g.rt_ctas = L->rt_grid;
        g.rt_chunk = L->rt_chunk;
        g.rt_E = E;
        g.rt_perm = L->perm;
        g.rt_out_counts = L->counts;
        g.rt_out_offsets = L->offsets;
        g.rt_cls_stride = cls_stride;
    } else {
        g.rows = L->inv;  // token t's row goes to its slot (the finalize kernel's inverse permutation)
    }
    g.C = L->z;
    g.ldc = H;
    if ((rc = cuda_fail(cm::launch_tc_gemm(g, L->num_sms, s)))) return rc;
    mark(L, 2, s);
    if (factored && T - n_cls > 0) {
        cm::TcGemmArgs g2;
        std::memset(&g2, 0, sizeof(g2));
        g2.status = L->status;
        g2.wait_limit_ns = L->wait_limit_ns;
        const int64_t M2 = T - n_cls;  // the routed slots (class tokens' follow them)
        const int bn2 = tf32_plan(L, g2, r, H, M2, 0).bn;
        if (encode_tmap_f32(&g2.tmA0, L->z, M2, H, 128) || encode_tmap_f32(&g2.tmB0, Vh_r, r, H, bn2))
            return CLEARMOE_ECUDA;
        g2.mode = cm::TC_DENSE;
        g2.epi = cm::TC_EPI_SCALE;
        g2.M = M2;
        g2.N = r;
        g2.K0 = H;
        g2.scale = S_r;
        g2.C = L->t;
        g2.ldc = r;
        if ((rc = cuda_fail(cm::launch_tc_gemm(g2, L->num_sms, s)))) return rc;
    }
    mark(L, 3, s);
    cm::TcGemmArgs g3;
    std::memset(&g3, 0, sizeof(g3));
    g3.status = L->status;
    g3.wait_limit_ns = L->wait_limit_ns;
    const int bn3 = tf32_plan(L, g3, d, (factored ? r : materialized ? H : 0) + H, T, G).bn;
    if ((factored && (encode_tmap_f32(&g3.tmA0, L->t, T, r, 128) || encode_tmap_f32(&g3.tmB0, U_r, d, r, bn3))) ||
        (materialized && (encode_tmap_f32(&g3.tmA0, L->z, T, H, 128) || encode_tmap_f32(&g3.tmB0, W_sh, d, H, bn3))) ||
        encode_tmap_f32(&g3.tmA1, L->z, T, H, 128))
        return CLEARMOE_ECUDA;
    for (int e = 0; e < E; ++e)
        if (encode_tmap_f32(&g3.tmB1[e], residual_e[e], d, H, bn3)) return CLEARMOE_ECUDA;
    if (n_cls > 0) {  // the dense path's group: W2
        if (encode_tmap_f32(&g3.tmB1[E], W2, d, H, bn3)) return CLEARMOE_ECUDA;
        g3.dense_last = 1;
    }
    g3.mode = cm::TC_GROUPED;
    g3.epi = cm::TC_EPI_SCATTER;
    g3.M = T;
    g3.N = d;
    g3.K0 = factored ? r : materialized ? H : 0;  // folded: the K chain is z x W_e^comb alone
    g3.K1 = H;
    g3.offsets = L->offsets;
    g3.E = G;
    g3.rows = L->perm;
    g3.out_bias = b2;
    g3.C = out;
    g3.ldc = d;
    rc = cuda_fail(cm::launch_tc_gemm(g3, L->num_sms, s));
    mark(L, 4, s);
    return rc;
}

static int ffn_impl(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                    const void* U_r, const float* S_r, const void* Vh_r, const void* W_sh,
                    const void* const* residual_e, const clearmoe_router* router, int E, int r,
                    const clearmoe_ffn_options* opt, void* out, cudaStream_t s) {
    // Basis forms: factorised (U_r set: t = diag(S_r) Vh_r z, then U_r t), materialised (W_sh
    // set: the K chain [z | z] x [W_e^res | W_sh]), folded (neither: residual_e holds W_comb, no
    // basis step, no first K segment).
    const bool factored = U_r != nullptr;
    const bool materialized = !factored && W_sh != nullptr;
    const int d = L->desc.d, H = L->desc.hidden;
    const bool bf16 = L->desc.dtype == CLEARMOE_BF16;
    // class tokens: group E after the experts (slots [T - n_cls, T)), K chain z x W2 alone
    const int64_t cls_stride = opt ? opt->cls_stride : 0;
    const int64_t n_cls = cm::n_class_tokens(T, cls_stride);
    const int G = E + (cls_stride > 0 ? 1 : 0);  // groups of the grouped GEMM
    const void* b2 = opt ? opt->b2 : nullptr;
    const clearmoe_mlp_router* mlp = opt ? opt->mlp_router : nullptr;
    const bool ln = opt && opt->input_layernorm;  // x is y: LN(y) folded into the router and fc1
    if (opt && opt->router_in_fc1) {  // the linear router only, no class tokens, no folded LayerNorm
        if (mlp || cls_stride > 0 || ln || materialized) return CLEARMOE_EUNSUPPORTED;
        return ffn_router_in_fc1(L, x, T, W1, b1, U_r, S_r, Vh_r, residual_e, router, E, r, b2, out, s);
    }
    int rc;
    mark(L, 0, s);
    if (ln && (rc = ln_prep(L, x, T, W1, mlp ? mlp->W_in : router->W, mlp ? mlp->hidden : E, s))) return rc;
    if ((rc = do_route(L, x, T, router, mlp, E, cls_stride, s, ln))) return rc;
    // bf16 with the 2-SM fc1, or fp32 on the tensor cores: the fc1 epilogue assigns the slots
    // itself (no finalize launch)
    const int p1 = bf16 && H <= cm::TC2_BIAS_CAP ? cm::tc2_pick_bn(cm::TC_DENSE, H) : 0;
    const bool f32_tc = !bf16 && !ln && f32_tc_ok(d, H, r, factored);
    const bool fused = (p1 || f32_tc) && L->rt_grid <= 256 && L->rt_grid * E <= cm::TC2_TAB_CAP;
    if (!fused && (rc = do_finalize(L, s))) return rc;
    mark(L, 1, s);

    if (f32_tc)
        return ffn_f32_tc(L, x, T, W1, b1, U_r, S_r, Vh_r, W_sh, residual_e, E, r, n_cls, cls_stride, G, b2,
                          opt ? opt->W2 : nullptr, fused, out, s);
    if (!bf16) {
        cm::SimtGemmArgs g;
        std::memset(&g, 0, sizeof(g));
        // fc1 + bias + GELU on tokens gathered in expert order
        g.A0 = static_cast<const float*>(x);
        g.lda0 = d;
        g.K0 = d;
        g.B0 = static_cast<const float*>(W1);
        g.a_rows = L->perm;
        g.M = T;
        g.N = H;
        g.bias = static_cast<const float*>(b1);
        g.gelu = 1;
        g.C = static_cast<float*>(L->z);
        g.ldc = H;
        if (ln) {
            g.ln_stats = L->ln_stats;
            g.ln_colsum = L->ln_sums;
        }
        if ((rc = launch_simt(L, g, s))) return rc;
        mark(L, 2, s);
        if (factored) {  // t = diag(S_r) Vh_r z
            std::memset(&g, 0, sizeof(g));
            g.A0 = static_cast<const float*>(L->z);
            g.lda0 = H;
            g.K0 = H;
            g.B0 = static_cast<const float*>(Vh_r);
            g.M = T - n_cls;  // the routed slots (class tokens' follow them)
            g.N = r;
            g.scale = S_r;
            g.C = static_cast<float*>(L->t);
            g.ldc = r;
            if ((rc = launch_simt(L, g, s))) return rc;
        }
        mark(L, 3, s);
        // out[perm[slot]] = U_r t + W_e^res z per expert sub-batch (folded: W_e^comb z)
        std::memset(&g, 0, sizeof(g));
        if (factored) {
            g.A0 = static_cast<const float*>(L->t);
            g.lda0 = r;
            g.K0 = r;
            g.B0 = static_cast<const float*>(U_r);
        } else if (materialized) {
            g.A0 = static_cast<const float*>(L->z);
            g.lda0 = H;
            g.K0 = H;
            g.B0 = static_cast<const float*>(W_sh);
        }
        g.A1 = static_cast<const float*>(L->z);
        g.lda1 = H;
        g.K1 = H;
        for (int e = 0; e < E; ++e) g.B1[e] = static_cast<const float*>(residual_e[e]);
        if (n_cls > 0) {
            g.B1[E] = static_cast<const float*>(opt->W2);
            g.dense_last = 1;
        }
        g.bias = static_cast<const float*>(b2);
        g.M = T;
        g.N = d;
        g.C = static_cast<float*>(out);
        g.ldc = d;
        g.c_rows = L->perm;
        g.offsets = L->offsets;
        g.E = G;
        rc = launch_simt(L, g, s);
        mark(L, 4, s);
        return rc;
    }

    // ---- bf16: tcgen05 GEMMs
    const int bn1 = cm::tc_pick_bn(cm::TC_GATHER, H);
    const int bn2 = factored ? cm::tc_pick_bn(cm::TC_DENSE, r) : 1;
    const int bn3 = cm::tc_pick_bn(cm::TC_GROUPED, d);
    if (!bn1 || !bn2 || !bn3) return CLEARMOE_EUNSUPPORTED;
    cm::TcGemmArgs g;
    std::memset(&g, 0, sizeof(g));
    g.status = L->status;
    g.wait_limit_ns = L->wait_limit_ns;
    // fc1 + b1 + GELU into z in expert order. 2-SM kernel: x read in token order by TMA, each
    // output row stored at its slot (formed in the epilogue, or inv[token] after the finalize
    // kernel); otherwise A rows are gathered by perm.
    g.epi = cm::TC_EPI_BIAS_GELU;
    g.M = T;
    g.N = H;
    g.K0 = d;
    g.bias = b1;
    g.C = L->z;
    g.ldc = H;
    if (ln) {
        g.ln_stats = L->ln_stats;
        g.ln_colsum = L->ln_sums;
    }
    if (p1) {
        if (encode_tmap_bf16(&g.tmA0, x, T, d, 128) || encode_tmap_bf16(&g.tmB0, W1, H, d, p1 / 2))
            return CLEARMOE_ECUDA;
        if (ln && (rc = ln_fc1_aug(L, g, T, p1 / 2))) return rc;
        g.mode = cm::TC_DENSE;
        if (fused) {  // slots from the routing's per-range counts and ranks; writes perm, counts, offsets
            g.rt_info = L->tinfo;
            g.rt_counts = L->cta_counts;
            g.rt_ctas = L->rt_grid;
            g.rt_chunk = L->rt_chunk;
            g.rt_E = E;
            g.rt_perm = L->perm;
            g.rt_out_counts = L->counts;
            g.rt_out_offsets = L->offsets;
            g.rt_cls_stride = cls_stride;
        } else {
            g.rows = L->inv;
        }
        // x and W1 are ready before the routing (which releases fc1 only after its own wait): the
        // operand loads and MMAs start at once; the epilogue waits for the routing's results
        g.pdl_wait_role = 1;
        g.epi12 = p1 == 256 && d <= cm::TC2_EPI12_MAX_K;  // short K: the GELU epilogue bounds a tile
        rc = cuda_fail(cm::launch_tc_gemm2(g, L->num_sms, s));
    } else {
        if (encode_tmap_bf16(&g.tmB0, W1, H, d, bn1)) return CLEARMOE_ECUDA;
        g.mode = cm::TC_GATHER;
        g.gather_src = x;
        g.gather_ld = d;
        g.rows = L->perm;
        rc = cuda_fail(cm::launch_tc_gemm(g, L->num_sms, s));
    }
    if (rc) return rc;
    mark(L, 2, s);
    if (factored) {  // t = diag(S_r) Vh_r z (2-SM kernel when r is a multiple of 128)
        cm::TcGemmArgs g2;
        std::memset(&g2, 0, sizeof(g2));
        g2.status = L->status;
        g2.wait_limit_ns = L->wait_limit_ns;
        const int p2 = cm::tc2_pick_bn(cm::TC_DENSE, r);
        if (encode_tmap_bf16(&g2.tmA0, L->z, T, H, 128) ||
            encode_tmap_bf16(&g2.tmB0, Vh_r, r, H, p2 ? p2 / 2 : bn2))
            return CLEARMOE_ECUDA;
        g2.mode = cm::TC_DENSE;
        g2.epi = cm::TC_EPI_SCALE;
        g2.M = T - n_cls;  // the routed slots (class tokens' follow them)
        g2.N = r;
        g2.K0 = H;
        g2.scale = S_r;
        g2.C = L->t;
        g2.ldc = r;
        g2.a_evict_first = 1;  // z is streamed once here; its rows still in L2 from fc1 stay there
        g2.pdl_trigger_late = 1;  // the grouped GEMM may start once fc1 has completed
        rc = cuda_fail(p2 ? cm::launch_tc_gemm2(g2, L->num_sms, s) : cm::launch_tc_gemm(g2, L->num_sms, s));
        if (rc) return rc;
    }
    mark(L, 3, s);
    // out[perm[slot]] = [t | z] [U_r | W_e^res]^T per expert sub-batch
    cm::TcGemmArgs g3;
    std::memset(&g3, 0, sizeof(g3));
    g3.status = L->status;
    g3.wait_limit_ns = L->wait_limit_ns;
    // The 2-SM kernel loads half of each pair tile's B rows per CTA: boxes of p3 / 2 rows.
    const int p3 = cm::tc2_pick_bn(cm::TC_GROUPED, d);
    const int box3 = p3 ? p3 / 2 : bn3;
    if ((factored && (encode_tmap_bf16(&g3.tmA0, L->t, T, r, 128) || encode_tmap_bf16(&g3.tmB0, U_r, d, r, box3))) ||
        (materialized &&
         (encode_tmap_bf16(&g3.tmA0, L->z, T, H, 128) || encode_tmap_bf16(&g3.tmB0, W_sh, d, H, box3))) ||
        encode_tmap_bf16(&g3.tmA1, L->z, T, H, 128))
        return CLEARMOE_ECUDA;
    for (int e = 0; e < E; ++e)
        if (encode_tmap_bf16(&g3.tmB1[e], residual_e[e], d, H, box3)) return CLEARMOE_ECUDA;
    if (n_cls > 0) {  // the dense path's group: W2
        if (encode_tmap_bf16(&g3.tmB1[E], opt->W2, d, H, box3)) return CLEARMOE_ECUDA;
        g3.dense_last = 1;
    }
    g3.out_bias = b2;
    // right after the basis kernel (which releases it only once fc1 has completed) the grouped GEMM
    // starts its z segments at once, on the SMs the basis leaves idle, and waits for the basis only
    // before its first t segment; with no routed rows no basis kernel runs, and fc1 (which releases
    // early) precedes it
    if (factored && T - n_cls > 0) g3.pdl_wait_role = 2;
    g3.mode = cm::TC_GROUPED;
    g3.epi = cm::TC_EPI_SCATTER;
    g3.M = T;
    g3.N = d;
    g3.K0 = factored ? r : materialized ? H : 0;  // folded: the K chain is z x W_e^comb alone
    g3.K1 = H;
    g3.offsets = L->offsets;
    g3.E = G;
    g3.rows = L->perm;
    g3.C = out;
    g3.ldc = d;
    rc = cuda_fail(p3 ? cm::launch_tc_gemm2(g3, L->num_sms, s) : cm::launch_tc_gemm(g3, L->num_sms, s));
    mark(L, 4, s);
    return rc;
}

int clearmoe_ffn_forward(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                         const void* U_r, const float* S_r, const void* Vh_r, const void* const* residual_e,
                         const clearmoe_router* router, int32_t E, int32_t r, void* out, void* stream) {
    return clearmoe_ffn_forward_ex(L, x, T, W1, b1, U_r, S_r, Vh_r, residual_e, router, E, r, nullptr, out, stream);
}

int clearmoe_ffn_forward_ex(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                            const void* U_r, const float* S_r, const void* Vh_r, const void* const* residual_e,
                            const clearmoe_router* router, int32_t E, int32_t r, const clearmoe_ffn_options* opt,
                            void* out, void* stream) {
    int rc = check_common(L, x, T);
    if (rc) return rc;
    if ((rc = check_router_and_options(L, router, opt, E))) return rc;
    if (!W1 || !b1 || !U_r || !S_r || !Vh_r || !residual_e || !out) return CLEARMOE_EINVAL;
    const int d = L->desc.d, H = L->desc.hidden;
    if (r < 1 || r > L->desc.max_r || r > d || r > H) return CLEARMOE_EINVAL;
    for (int e = 0; e < E; ++e)
        if (!residual_e[e] || misaligned(residual_e[e])) return CLEARMOE_EINVAL;
    if (misaligned(W1) || misaligned(b1) || misaligned(U_r) || misaligned(S_r) || misaligned(Vh_r) ||
        misaligned(out))
        return CLEARMOE_EINVAL;
    const bool bf16 = L->desc.dtype == CLEARMOE_BF16;
    if (bf16 && r % 16) return CLEARMOE_EUNSUPPORTED;
    if (!bf16 && r % 4) return CLEARMOE_EUNSUPPORTED;
    return ffn_impl(L, x, T, W1, b1, U_r, S_r, Vh_r, nullptr, residual_e, router, E, r, opt, out,
                    static_cast<cudaStream_t>(stream));
}

int clearmoe_ffn_forward_folded(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                                const void* const* W_comb, const clearmoe_router* router, int32_t E, void* out,
                                void* stream) {
    return clearmoe_ffn_forward_folded_ex(L, x, T, W1, b1, W_comb, router, E, nullptr, out, stream);
}

int clearmoe_ffn_forward_folded_ex(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                                   const void* const* W_comb, const clearmoe_router* router, int32_t E,
                                   const clearmoe_ffn_options* opt, void* out, void* stream) {
    int rc = check_common(L, x, T);
    if (rc) return rc;
    if ((rc = check_router_and_options(L, router, opt, E))) return rc;
    if (!W1 || !b1 || !W_comb || !out) return CLEARMOE_EINVAL;
    for (int e = 0; e < E; ++e)
        if (!W_comb[e] || misaligned(W_comb[e])) return CLEARMOE_EINVAL;
    if (misaligned(W1) || misaligned(b1) || misaligned(out)) return CLEARMOE_EINVAL;
    return ffn_impl(L, x, T, W1, b1, nullptr, nullptr, nullptr, nullptr, W_comb, router, E, 0, opt, out,
                    static_cast<cudaStream_t>(stream));
}

int clearmoe_ffn_forward_materialized(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                                      const void* W_sh, const void* const* residual_e, const clearmoe_router* router,
                                      int32_t E, void* out, void* stream) {
    return clearmoe_ffn_forward_materialized_ex(L, x, T, W1, b1, W_sh, residual_e, router, E, nullptr, out, stream);
}

int clearmoe_ffn_forward_materialized_ex(clearmoe_layer* L, const void* x, int64_t T, const void* W1,
                                         const void* b1, const void* W_sh, const void* const* residual_e,
                                         const clearmoe_router* router, int32_t E, const clearmoe_ffn_options* opt,
                                         void* out, void* stream) {
    int rc = check_common(L, x, T);
    if (rc) return rc;
    if ((rc = check_router_and_options(L, router, opt, E))) return rc;
    if (!W1 || !b1 || !W_sh || !residual_e || !out) return CLEARMOE_EINVAL;
    for (int e = 0; e < E; ++e)
        if (!residual_e[e] || misaligned(residual_e[e])) return CLEARMOE_EINVAL;
    if (misaligned(W1) || misaligned(b1) || misaligned(W_sh) || misaligned(out)) return CLEARMOE_EINVAL;
    return ffn_impl(L, x, T, W1, b1, nullptr, nullptr, nullptr, W_sh, residual_e, router, E, 0, opt, out,
                    static_cast<cudaStream_t>(stream));
}

// Algorithm 2's residuals are scaled copies of one matrix, W_e^res = s_e R with R = W2 - W_shared,
// so y = W_shared z + s_a R z = s_a (U_r t' + R z) with t' = diag(S_r) Vh_r z / s_a: every GEMM
// runs in token order (no sort, no scatter) and the router's choice enters as a row scale only.
int clearmoe_ffn_forward_scaled(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                                const void* U_r, const float* S_r, const void* Vh_r, const void* R,
                                const float* s_e, const clearmoe_router* router, int32_t E, int32_t r, void* out,
                                void* stream) {
    int rc = check_common(L, x, T);
    if (rc) return rc;
    if ((rc = check_router(L, router, E))) return rc;
    if (!W1 || !b1 || !U_r || !S_r || !Vh_r || !R || !s_e || !out) return CLEARMOE_EINVAL;
    const int d = L->desc.d, H = L->desc.hidden;
    if (r < 1 || r > L->desc.max_r || r > d || r > H) return CLEARMOE_EINVAL;
    if (misaligned(W1) || misaligned(b1) || misaligned(U_r) || misaligned(S_r) || misaligned(Vh_r) ||
        misaligned(R) || misaligned(out))
        return CLEARMOE_EINVAL;
    const bool bf16 = L->desc.dtype == CLEARMOE_BF16;
    if (r % (bf16 ? 16 : 4)) return CLEARMOE_EUNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    mark(L, 0, s);
    if ((rc = do_route(L, x, T, router, nullptr, E, 0, s))) return rc;  // idx, in token order
    mark(L, 1, s);
    if (!bf16) {
        cm::SimtGemmArgs g;
        std::memset(&g, 0, sizeof(g));
        g.A0 = static_cast<const float*>(x);  // z = GELU(W1 x + b1), token order
        g.lda0 = d;
        g.K0 = d;
        g.B0 = static_cast<const float*>(W1);
        g.M = T;
        g.N = H;
        g.bias = static_cast<const float*>(b1);
        g.gelu = 1;
        g.C = static_cast<float*>(L->z);
        g.ldc = H;
        if ((rc = launch_simt(L, g, s))) return rc;
        mark(L, 2, s);
        std::memset(&g, 0, sizeof(g));  // t' = diag(S_r) Vh_r z / s_a
        g.A0 = static_cast<const float*>(L->z);
        g.lda0 = H;
        g.K0 = H;
        g.B0 = static_cast<const float*>(Vh_r);
        g.M = T;
        g.N = r;
        g.scale = S_r;
        g.row_group = L->idx;
        g.group_scale = s_e;
        g.scale_groups = E;
        g.row_scale_inv = 1;
        g.C = static_cast<float*>(L->t);
        g.ldc = r;
        if ((rc = launch_simt(L, g, s))) return rc;
        mark(L, 3, s);
        std::memset(&g, 0, sizeof(g));  // out = s_a (U_r t' + R z)
        g.A0 = static_cast<const float*>(L->t);
        g.lda0 = r;
        g.K0 = r;
        g.B0 = static_cast<const float*>(U_r);
        g.A1 = static_cast<const float*>(L->z);
        g.lda1 = H;
        g.K1 = H;
        g.B1[0] = static_cast<const float*>(R);
        g.M = T;
        g.N = d;
        g.row_group = L->idx;
        g.group_scale = s_e;
        g.scale_groups = E;
        g.C = static_cast<float*>(out);
        g.ldc = d;
        rc = launch_simt(L, g, s);
    } else {
        const int p1 = H <= cm::TC2_BIAS_CAP ? cm::tc2_pick_bn(cm::TC_DENSE, H) : 0;
        const int p2 = cm::tc2_pick_bn(cm::TC_DENSE, r), p3 = cm::tc2_pick_bn(cm::TC_GROUPED, d);
        const int b1n = cm::tc_pick_bn(cm::TC_DENSE, H), b2n = cm::tc_pick_bn(cm::TC_DENSE, r);
        const int b3n = cm::tc_pick_bn(cm::TC_GROUPED, d);
        if ((!p1 && !b1n) || (!p2 && !b2n) || (!p3 && !b3n)) return CLEARMOE_EUNSUPPORTED;
        cm::TcGemmArgs g;
        std::memset(&g, 0, sizeof(g));
        g.status = L->status;
        g.wait_limit_ns = L->wait_limit_ns;
        if (encode_tmap_bf16(&g.tmA0, x, T, d, 128) || encode_tmap_bf16(&g.tmB0, W1, H, d, p1 ? p1 / 2 : b1n))
            return CLEARMOE_ECUDA;
        g.mode = cm::TC_DENSE;
        g.epi = cm::TC_EPI_BIAS_GELU;
        g.M = T;
        g.N = H;
        g.K0 = d;
        g.bias = b1;
        g.C = L->z;
        g.ldc = H;
        g.epi12 = p1 == 256 && d <= cm::TC2_EPI12_MAX_K;  // short K: the GELU epilogue bounds a tile
        if ((rc = cuda_fail(p1 ? cm::launch_tc_gemm2(g, L->num_sms, s) : cm::launch_tc_gemm(g, L->num_sms, s))))
            return rc;
        mark(L, 2, s);
        cm::TcGemmArgs g2;
        std::memset(&g2, 0, sizeof(g2));
        g2.status = L->status;
        g2.wait_limit_ns = L->wait_limit_ns;
        if (encode_tmap_bf16(&g2.tmA0, L->z, T, H, 128) || encode_tmap_bf16(&g2.tmB0, Vh_r, r, H, p2 ? p2 / 2 : b2n))
            return CLEARMOE_ECUDA;
        g2.mode = cm::TC_DENSE;
        g2.epi = cm::TC_EPI_SCALE;
        g2.M = T;
        g2.N = r;
        g2.K0 = H;
        g2.scale = S_r;
        g2.row_group = L->idx;
        g2.group_scale = s_e;
        g2.scale_groups = E;
        g2.row_scale_inv = 1;
        g2.C = L->t;
        g2.ldc = r;
        g2.a_evict_first = 1;
        if ((rc = cuda_fail(p2 ? cm::launch_tc_gemm2(g2, L->num_sms, s) : cm::launch_tc_gemm(g2, L->num_sms, s))))
            return rc;
        mark(L, 3, s);
        cm::TcGemmArgs g3;
        std::memset(&g3, 0, sizeof(g3));
        g3.status = L->status;
        g3.wait_limit_ns = L->wait_limit_ns;
        const int box3 = p3 ? p3 / 2 : b3n;
        if (encode_tmap_bf16(&g3.tmA0, L->t, T, r, 128) || encode_tmap_bf16(&g3.tmB0, U_r, d, r, box3) ||
            encode_tmap_bf16(&g3.tmA1, L->z, T, H, 128) || encode_tmap_bf16(&g3.tmB1[0], R, d, H, box3))
            return CLEARMOE_ECUDA;
        g3.mode = cm::TC_GROUPED;  // one group over all tokens (no offsets): [z | t'] x [R | U_r]
        g3.epi = cm::TC_EPI_STORE;
        g3.M = T;
        g3.N = d;
        g3.K0 = r;
        g3.K1 = H;
        g3.E = 1;
        g3.row_group = L->idx;
        g3.group_scale = s_e;
        g3.scale_groups = E;
        g3.C = out;
        g3.ldc = d;
        rc = cuda_fail(p3 ? cm::launch_tc_gemm2(g3, L->num_sms, s) : cm::launch_tc_gemm(g3, L->num_sms, s));
    }
    mark(L, 4, s);
    if (rc) return rc;
    return do_finalize(L, s);  // counts, offsets, perm for clearmoe_get_routing (off the path)
}

int clearmoe_materialize_basis(clearmoe_layer* L, const void* U_r, const float* S_r, const void* Vh_r, int32_t r,
                               void* W_sh, void* stream) {
    if (!L || !U_r || !S_r || !Vh_r || !W_sh) return CLEARMOE_EINVAL;
    const int d = L->desc.d, H = L->desc.hidden;
    if (r < 1 || r > L->desc.max_r || r > d || r > H) return CLEARMOE_EINVAL;
    cm::FoldArgs f;
    std::memset(&f, 0, sizeof(f));
    f.U = U_r;
    f.S = S_r;
    f.Vh = Vh_r;
    f.out[0] = W_sh;  // res[0] == nullptr: W_shared alone
    f.d = d;
    f.H = H;
    f.r = r;
    f.E = 1;
    return cuda_fail(cm::launch_fold_basis(f, L->desc.dtype, static_cast<cudaStream_t>(stream)));
}

int clearmoe_fold_basis(clearmoe_layer* L, const void* U_r, const float* S_r, const void* Vh_r,
                        const void* const* residual_e, int32_t E, int32_t r, void* const* W_comb, void* stream) {
    if (!L || !U_r || !S_r || !Vh_r || !residual_e || !W_comb) return CLEARMOE_EINVAL;
    const int d = L->desc.d, H = L->desc.hidden;
    if (E < 1 || E > L->desc.max_E) return CLEARMOE_EINVAL;
    if (r < 1 || r > L->desc.max_r || r > d || r > H) return CLEARMOE_EINVAL;
    cm::FoldArgs f;
    std::memset(&f, 0, sizeof(f));
    f.U = U_r;
    f.S = S_r;
    f.Vh = Vh_r;
    for (int e = 0; e < E; ++e) {
        if (!residual_e[e] || !W_comb[e]) return CLEARMOE_EINVAL;
        f.res[e] = residual_e[e];
        f.out[e] = W_comb[e];
    }
    f.d = d;
    f.H = H;
    f.r = r;
    f.E = E;
    return cuda_fail(cm::launch_fold_basis(f, L->desc.dtype, static_cast<cudaStream_t>(stream)));
}

int clearmoe_dense_ffn_forward(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                               const void* W2, void* out, void* stream) {
    return clearmoe_dense_ffn_forward_ex(L, x, T, W1, b1, W2, nullptr, out, stream);
}

static int dense_impl(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1, const void* W2,
                      const void* b2, bool ln, void* out, cudaStream_t s) {
    int rc = check_common(L, x, T);
    if (rc) return rc;
    if (!W1 || !b1 || !W2 || !out) return CLEARMOE_EINVAL;
    if (misaligned(W1) || misaligned(b1) || misaligned(W2) || misaligned(out) || misaligned(b2))
        return CLEARMOE_EINVAL;
    const int d = L->desc.d, H = L->desc.hidden;
    mark(L, 0, s);
    if (ln && (rc = ln_prep(L, x, T, W1, nullptr, 0, s))) return rc;  // x is y: LN(y) folded into fc1
    const float2* lns = ln ? L->ln_stats : nullptr;
    const float* lnc = ln ? L->ln_sums : nullptr;
    if (L->desc.dtype == CLEARMOE_F32 && !ln && f32_tc_ok(d, H, 0, false)) {  // TF32 tensor cores
        cm::TcGemmArgs g;
        std::memset(&g, 0, sizeof(g));
        g.status = L->status;
        g.wait_limit_ns = L->wait_limit_ns;
        const int bn1 = tf32_plan(L, g, H, d, T, 0).bn;
        if (encode_tmap_f32(&g.tmA0, x, T, d, 128) || encode_tmap_f32(&g.tmB0, W1, H, d, bn1)) return CLEARMOE_ECUDA;
        g.mode = cm::TC_DENSE;
        g.epi = cm::TC_EPI_BIAS_GELU;
        g.M = T;
        g.N = H;
        g.K0 = d;
        g.bias = b1;
        g.C = L->z;
        g.ldc = H;
        if ((rc = cuda_fail(cm::launch_tc_gemm(g, L->num_sms, s)))) return rc;
        mark(L, 1, s);
        cm::TcGemmArgs g2;
        std::memset(&g2, 0, sizeof(g2));
        g2.status = L->status;
        g2.wait_limit_ns = L->wait_limit_ns;
        const int bn2 = tf32_plan(L, g2, d, H, T, 0).bn;
        if (encode_tmap_f32(&g2.tmA0, L->z, T, H, 128) || encode_tmap_f32(&g2.tmB0, W2, d, H, bn2))
            return CLEARMOE_ECUDA;
        g2.mode = cm::TC_DENSE;
        g2.epi = cm::TC_EPI_STORE;
        g2.out_bias = b2;
        g2.M = T;
        g2.N = d;
        g2.K0 = H;
        g2.C = out;
        g2.ldc = d;
        rc = cuda_fail(cm::launch_tc_gemm(g2, L->num_sms, s));
        mark(L, 2, s);
        return rc;
    }
    if (L->desc.dtype == CLEARMOE_F32) {
        cm::SimtGemmArgs g;
        std::memset(&g, 0, sizeof(g));
        g.A0 = static_cast<const float*>(x);
        g.lda0 = d;
        g.K0 = d;
        g.B0 = static_cast<const float*>(W1);
        g.M = T;
        g.N = H;
        g.bias = static_cast<const float*>(b1);
        g.gelu = 1;
        g.C = static_cast<float*>(L->z);
        g.ldc = H;
        g.ln_stats = lns;
        g.ln_colsum = lnc;
        if ((rc = launch_simt(L, g, s))) return rc;
        mark(L, 1, s);
        std::memset(&g, 0, sizeof(g));
        g.A0 = static_cast<const float*>(L->z);
        g.lda0 = H;
        g.K0 = H;
        g.B0 = static_cast<const float*>(W2);
        g.bias = static_cast<const float*>(b2);
        g.M = T;
        g.N = d;
        g.C = static_cast<float*>(out);
        g.ldc = d;
        rc = launch_simt(L, g, s);
        mark(L, 2, s);
        return rc;
    }
    const int bn1 = cm::tc_pick_bn(cm::TC_DENSE, H);
    const int bn2 = cm::tc_pick_bn(cm::TC_DENSE, d);
    cm::TcGemmArgs g;
    std::memset(&g, 0, sizeof(g));
    g.status = L->status;
    g.wait_limit_ns = L->wait_limit_ns;
    const int pair1 = H <= cm::TC2_BIAS_CAP ? cm::tc2_pick_bn(cm::TC_DENSE, H) : 0;  // 2-SM tile widths
    const int pair2 = cm::tc2_pick_bn(cm::TC_DENSE, d);
    if (encode_tmap_bf16(&g.tmA0, x, T, d, 128) || encode_tmap_bf16(&g.tmB0, W1, H, d, pair1 ? pair1 / 2 : bn1))
        return CLEARMOE_ECUDA;
    g.mode = cm::TC_DENSE;
    g.epi = cm::TC_EPI_BIAS_GELU;
    g.M = T;
    g.N = H;
    g.K0 = d;
    g.bias = b1;
    g.C = L->z;
    g.ldc = H;
    g.ln_stats = lns;
    g.ln_colsum = lnc;  // the 1-SM kernel: the column sums in the epilogue
    if (ln && pair1 && (rc = ln_fc1_aug(L, g, T, pair1 / 2))) return rc;  // 2-SM: the augmentation block
    g.epi12 = pair1 == 256 && d <= cm::TC2_EPI12_MAX_K;  // short K: the GELU epilogue bounds a tile
    if ((rc = cuda_fail(pair1 ? cm::launch_tc_gemm2(g, L->num_sms, s) : cm::launch_tc_gemm(g, L->num_sms, s))))
        return rc;
    mark(L, 1, s);
    cm::TcGemmArgs g2;
    std::memset(&g2, 0, sizeof(g2));
    g2.status = L->status;
    g2.wait_limit_ns = L->wait_limit_ns;
    if (encode_tmap_bf16(&g2.tmA0, L->z, T, H, 128) || encode_tmap_bf16(&g2.tmB0, W2, d, H, pair2 ? pair2 / 2 : bn2))
        return CLEARMOE_ECUDA;
    g2.mode = cm::TC_DENSE;
    g2.epi = cm::TC_EPI_STORE;
    g2.out_bias = b2;
    g2.M = T;
    g2.N = d;
    g2.K0 = H;
    g2.C = out;
    g2.ldc = d;
    rc = cuda_fail(pair2 ? cm::launch_tc_gemm2(g2, L->num_sms, s) : cm::launch_tc_gemm(g2, L->num_sms, s));
    mark(L, 2, s);
    return rc;
}

int clearmoe_dense_ffn_forward_ex(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                                  const void* W2, const void* b2, void* out, void* stream) {
    return dense_impl(L, x, T, W1, b1, W2, b2, false, out, static_cast<cudaStream_t>(stream));
}

int clearmoe_dense_ffn_forward_opt(clearmoe_layer* L, const void* x, int64_t T, const void* W1, const void* b1,
                                   const void* W2, const clearmoe_ffn_options* opt, void* out, void* stream) {
    if (opt && (opt->cls_stride != 0 || opt->mlp_router)) return CLEARMOE_EINVAL;
    return dense_impl(L, x, T, W1, b1, W2, opt ? opt->b2 : nullptr, opt && opt->input_layernorm, out,
                      static_cast<cudaStream_t>(stream));
}

int clearmoe_layer_norm(clearmoe_layer* L, const void* y, int64_t T, void* x_out, void* stream) {
    int rc = check_common(L, y, T);
    if (rc) return rc;
    if (!x_out || misaligned(x_out)) return CLEARMOE_EINVAL;
    return cuda_fail(cm::launch_layer_norm(y, x_out, T, L->desc.d, L->desc.dtype, static_cast<cudaStream_t>(stream)));
}

int clearmoe_get_routing(clearmoe_layer* L, int32_t* idx, int32_t* counts, int32_t* offsets, int32_t* perm,
                         void* stream) {
    if (!L) return CLEARMOE_EINVAL;
    if (L->last_T < 1) return CLEARMOE_EINVAL;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t T = (size_t)L->last_T, E = (size_t)L->last_groups;
    cudaError_t e = cudaSuccess;
    if (idx && e == cudaSuccess) e = cudaMemcpyAsync(idx, L->idx, T * 4, cudaMemcpyDeviceToDevice, s);
    if (counts && e == cudaSuccess) e = cudaMemcpyAsync(counts, L->counts, E * 4, cudaMemcpyDeviceToDevice, s);
    if (offsets && e == cudaSuccess) e = cudaMemcpyAsync(offsets, L->offsets, (E + 1) * 4, cudaMemcpyDeviceToDevice, s);
    if (perm && e == cudaSuccess) e = cudaMemcpyAsync(perm, L->perm, T * 4, cudaMemcpyDeviceToDevice, s);
    return cuda_fail(e);
}

int clearmoe_layer_status(clearmoe_layer* L) {
    if (!L) return CLEARMOE_EINVAL;
    if (cudaDeviceSynchronize() != cudaSuccess) {
        (void)cudaGetLastError();
        return CLEARMOE_ECUDA;
    }
    int32_t st = 0;
    if (cudaMemcpy(&st, L->status, 4, cudaMemcpyDeviceToHost) != cudaSuccess) return CLEARMOE_ECUDA;
    if (st != 0) {
        // A GEMM whose waits gave up may leave K-split arrival counters part-counted: clear them so
        // that the next calls start from zero (a routing launch that gave up has already retired its
        // tag: nothing else to reset).
        if (cudaMemset(L->status, 0, 4) != cudaSuccess) return CLEARMOE_ECUDA;
        if (L->simt_cnt && cudaMemset(L->simt_cnt, 0, sizeof(int) * cm::simt_cnt_len(L->num_sms)) != cudaSuccess)
            return CLEARMOE_ECUDA;
        if (cudaDeviceSynchronize() != cudaSuccess) return CLEARMOE_ECUDA;
    }
    return st;
}

int clearmoe_set_profile_events(clearmoe_layer* L, void* const* events, int32_t n) {
    if (!L || n < 0 || n > 8 || (n > 0 && !events)) return CLEARMOE_EINVAL;
    for (int i = 0; i < 8; ++i) L->prof[i] = (i < n) ? static_cast<cudaEvent_t>(events[i]) : nullptr;
    L->prof_n = n;
    return CLEARMOE_OK;
}

int clearmoe_debug_set_wait(clearmoe_layer* L, int64_t wait_limit_ns, int32_t phantom_arrivals) {
    if (!L || wait_limit_ns < 1000 || phantom_arrivals < 0) return CLEARMOE_EINVAL;
    L->wait_limit_ns = wait_limit_ns;
    L->phantom = phantom_arrivals;
    return CLEARMOE_OK;
}

}  // extern "C"
