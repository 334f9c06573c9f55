/*
 * clearmoe.h -- C ABI of the GB300 (sm_103a) CLEAR-MoE FFN layer.
 *
 * CLEAR-MoE (arxiv 2606.28516) converts a frozen ViT FFN into a shared fc1, a shared truncated-SVD
 * fc2 basis and per-cluster residual fc2 experts chosen by a top-1 router (Eq. 2, Algorithms 2-3):
 *
 *     z = GELU(W1 x + b1)                       (fc1 shared by every expert, exact-erf GELU)
 *     a = argmax_e (W_g x + b_g)_e              (linear router, lowest index on ties)
 *     y = U_r diag(S_r) Vh_r z + W_a^res z      (shared SVD basis + residual expert of token a)
 *
 * Shapes (row-major, element type "D" = the layer's dtype unless stated):
 *   x [T x d], W1 [H x d], b1 [H], U_r [d x r], S_r [r] (always float32), Vh_r = V_r^T [r x H],
 *   residual_e[e] [d x H] for e < E, W_g [E x d], b_g [E], W2 [d x H], out [T x d].
 *
 * Conventions for every call below:
 *   - Every pointer named as a tensor is a DEVICE pointer owned by the caller, 16-byte aligned,
 *     to a dense row-major array of the stated shape. The library never frees caller memory.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream). Calls only enqueue work and
 *     return; they never synchronise, except clearmoe_layer_status and clearmoe_layer_destroy.
 *   - One handle may be used by one stream at a time: its workspace holds the hidden states and
 *     routing of the last forward.
 *   - Kernels are launched with programmatic dependent launch: the first kernel of a call may start,
 *     and read the weights (every tensor argument except x), while the kernel enqueued just before it
 *     on the same stream is finishing; x is read only after that kernel has completed. So weights
 *     must not be written by the kernel immediately before the call (any later-enqueued work in
 *     between, or a synchronisation, is enough).
 *   - Arguments are validated on the host first; on a validation error (EINVAL, EUNSUPPORTED)
 *     nothing is enqueued and the outputs are untouched. CLEARMOE_ECUDA can also come from a
 *     launch after earlier kernels of the same call were enqueued; the outputs are then
 *     undefined. Return values are clearmoe_status codes.
 *   - Device-side waits are bounded. A wait that runs out writes CLEARMOE_ETIMEOUT into the
 *     handle's device status word (read by clearmoe_layer_status); the outputs of that call are
 *     then undefined, and the handle stays usable.
 */
#ifndef CLEARMOE_H
#define CLEARMOE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CLEARMOE_OK = 0,
    CLEARMOE_EINVAL = -1,       /* bad argument: null pointer, size out of range, misalignment */
    CLEARMOE_EUNSUPPORTED = -2, /* valid but not tiled by this build (see clearmoe_layer_create) */
    CLEARMOE_ECUDA = -3,        /* a CUDA runtime/driver call failed */
    CLEARMOE_ENOMEM = -4,       /* workspace allocation failed */
    CLEARMOE_ETIMEOUT = -5      /* a bounded device-side wait ran out */
} clearmoe_status;

typedef enum { CLEARMOE_F32 = 0, CLEARMOE_BF16 = 1 } clearmoe_dtype;

/* Capacity of a layer handle. d and hidden are fixed per handle; T, E and r are per call and
 * bounded by max_tokens, max_E and max_r. dtype selects the arithmetic:
 *   CLEARMOE_BF16: bf16 storage, fp32 accumulation on the tcgen05 tensor cores; z, the shared-
 *                  basis coefficients t = diag(S_r) Vh_r z and out are stored in bf16.
 *   CLEARMOE_F32:  fp32 storage; the routing logits in fp32 FMA on the CUDA cores. The GEMMs of
 *                  the forward and of the dense FFN run on the TF32 tensor cores with each fp32
 *                  operand split into a TF32 part and its remainder and three products per term
 *                  (relative error near 2^-21 per product) when d, hidden and r are multiples
 *                  of 16 and the LayerNorm is not folded; otherwise, and in the other fp32 calls,
 *                  in exact fp32 FMA on the CUDA cores.
 * Tiling limits (else CLEARMOE_EUNSUPPORTED): bf16 needs d % 64 == 0, d <= 1024, hidden % 64 == 0
 * and r % 16 == 0 per call; fp32 needs d % 4 == 0, d <= 512, hidden % 4 == 0 and r % 4 == 0.
 * max_E <= 16, max_r <= 256, max_tokens <= 2^30. */
typedef struct {
    int64_t max_tokens;
    int32_t d;
    int32_t hidden;
    int32_t max_E;
    int32_t max_r;
    int32_t dtype; /* clearmoe_dtype */
} clearmoe_layer_desc;

/* Linear router (Phase 4, "Linear": d x E weights and a bias per expert): W [E x d], b [E],
 * both device pointers in the layer's dtype. */
typedef struct {
    const void* W;
    const void* b;
} clearmoe_router;

/* MLP router (Phase 4, "MLP": one hidden layer of d/6 units; the paper does not name its
 * activation, so both are offered): logits = W_out act(W_in x + b_in) + b_out with W_in
 * [hidden x d], b_in [hidden], W_out [E x hidden], b_out [E], device pointers in the layer's dtype.
 * The hidden layer runs on the tensor-core GEMM (fp32 on the fp32 layer) and is kept in fp32; the
 * output layer and the argmax run in fp32 on the routing kernel, so the decision is taken on fp32
 * logits as for the linear router. hidden: a multiple of 16 (bf16) or 4 (fp32), at most H / 2
 * (bf16) or H (fp32): the hidden layer lives in the hidden-state workspace before fc1 runs. */
typedef enum { CLEARMOE_ACT_RELU = 0, CLEARMOE_ACT_GELU = 1 } clearmoe_act;
typedef struct {
    const void* W_in;
    const void* b_in;
    const void* W_out;
    const void* b_out;
    int32_t hidden;
    int32_t act; /* clearmoe_act */
} clearmoe_mlp_router;

typedef struct clearmoe_layer clearmoe_layer;

/* Allocates the handle and its device workspace on the current device (hidden states
 * [max_tokens x hidden], basis coefficients [max_tokens x max_r], routing arrays, status word,
 * and for the folded LayerNorm 8 bytes per token of statistics, fp32 row sums [2 hidden + 16] and,
 * in bf16 layers, 128 bytes per token and per hidden unit of fc1's augmentation block).
 * Returns EINVAL for a null/invalid desc, EUNSUPPORTED per the tiling limits above, ENOMEM or
 * ECUDA if allocation fails (nothing is leaked). */
int clearmoe_layer_create(const clearmoe_layer_desc* desc, clearmoe_layer** out);

/* Synchronises the device, frees the workspace and the handle. NULL is accepted. */
int clearmoe_layer_destroy(clearmoe_layer* layer);

/* Routing only (Algorithm 3, steps 3-4): for every token t, a_t = the lowest e maximising
 * the fp32 logit W_g x_t + b_g; counts_e, offsets = exclusive prefix sum of counts (E + 1
 * entries), and perm[slot] = token with the tokens of expert e in slots
 * [offsets_e, offsets_{e+1}) in increasing id order (a stable sort by expert). One fused
 * kernel (logits, argmax, per-range histograms and ranks) and a slot kernel; results stay in
 * the handle (read them with clearmoe_get_routing).
 * 1 <= T <= max_tokens, 1 <= E <= max_E. */
int clearmoe_route(clearmoe_layer* layer, const void* x, int64_t T, const clearmoe_router* router,
                   int32_t E, void* stream);

/* Routing only with the MLP router: its hidden layer (one GEMM launch), then the routing kernel on
 * the fp32 hidden layer with W_out, b_out as the router, then the slot kernel. Same outputs and
 * errors as clearmoe_route; EINVAL for a NULL or misaligned weight, an unknown act or a hidden
 * width outside the limits above. */
int clearmoe_route_mlp(clearmoe_layer* layer, const void* x, int64_t T, const clearmoe_mlp_router* mlp,
                       int32_t E, void* stream);

/* The CLEAR-MoE FFN forward (Eq. 2 with Algorithm 3): routes (as clearmoe_route), computes
 * z = GELU(W1 x + b1) for every token in expert-sorted order (fc1 reads x in token order and its
 * epilogue stores each row at the token's slot), the shared basis through its factors,
 * t = diag(S_r) Vh_r z, and then, per expert sub-batch, out[perm[slot]] = U_r t + residual_e[e] z
 * (the scatter and the sum of the shared and residual terms are folded into the epilogue; each
 * row is written once).
 * residual_e is a HOST array of E device pointers, each to a [d x H] matrix.
 * 1 <= T <= max_tokens, 1 <= E <= max_E, 1 <= r <= min(max_r, d, H). out [T x d] must not
 * alias any input. */
int clearmoe_ffn_forward(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                         const void* b1, const void* U_r, const float* S_r, const void* Vh_r,
                         const void* const* residual_e, const clearmoe_router* router,
                         int32_t E, int32_t r, void* out, void* stream);

/* Deployment options of clearmoe_ffn_forward_ex (zero-initialise, then set the fields used).
 *  b2          fc2's bias [d] in the layer dtype (device), added once to every output row; NULL:
 *              none (Eq. 2 as printed has no fc2 bias; a pretrained ViT layer has one).
 *  cls_stride  > 0: token t with t % cls_stride == 0 is a class token (cls_stride = tokens per
 *              image, 197 for a 224 px ViT at patch 16, the class token first): it skips the router
 *              and takes the dense path out_t = W2 z_t (+ b2), as the dispatch benchmark keeps the
 *              class token out of expert dispatch. The class tokens form group E after the experts:
 *              idx = E, counts[E] = n_cls = ceil(T / cls_stride), slots [T - n_cls, T) in token
 *              order. Requires W2 and E + 1 <= 16 (EUNSUPPORTED otherwise). 0: every token routed.
 *  W2          the layer's dense fc2 [d x H] row-major (device), read for class tokens only.
 *  mlp_router  the MLP router in place of the linear one (see clearmoe_mlp_router).
 *  input_layernorm  non-zero: x is the un-normalised residual stream y of a ViT block, and the
 *              sublayer's input is its per-token LayerNorm without affine, LN(y) = (y - mean) /
 *              sqrt(biased variance + 1e-6), as clearmoe_layer_norm computes it (a pretrained
 *              block's LN affine folds into W1, b1 and the router offline). LN(y) is never
 *              written: one launch forms (mean, rstd) per token and the row sums c = W 1 of W1 and
 *              of the router's first matrix (W_g, or the MLP router's W_in), and the router and fc1
 *              use W LN(y) = rstd (W y - mean c) on their fp32 accumulators. 0: x is the input.
 *  router_in_fc1  non-zero: the linear router's logits (Phase 4 "Linear", Algorithm 3 step 3) are
 *              computed inside fc1 from the token tiles fc1 has already loaded (one more 256 x 32
 *              MMA unit per 256-token tile, W_g as its B operand), so the tokens are read from HBM
 *              once for both; fc1 stores z in token order, a slot kernel forms counts, offsets,
 *              perm and inv from per-128-token-range counts and ranks, the basis factor stores t at
 *              each token's slot, and the grouped GEMM gathers z rows by perm (TMA four-row
 *              gathers). Same results as the default path (expert indices bit-exact outside near
 *              ties, outputs within the tolerance). bf16 layers with the 2-SM kernels only (H a
 *              multiple of 128 and <= 4096, d a multiple of 128), the linear router, and neither
 *              class tokens, the MLP router, input_layernorm nor the materialised basis:
 *              EUNSUPPORTED otherwise. Works with clearmoe_ffn_forward_ex (factorised basis) and
 *              clearmoe_ffn_forward_folded_ex. */
typedef struct {
    const void* b2;
    int64_t cls_stride;
    const void* W2;
    const clearmoe_mlp_router* mlp_router; /* non-NULL: routes with it (router may then be NULL) */
    int32_t input_layernorm;
    int32_t router_in_fc1;
} clearmoe_ffn_options;

/* clearmoe_ffn_forward with deployment options (opt may be NULL: then identical to it). With
 * class tokens the basis step covers the routed slots only and the grouped GEMM has E + 1 groups,
 * the last one z x W2^T alone. EINVAL for cls_stride < 0 or > 2^30, a misaligned b2 or W2, or a
 * NULL W2 with cls_stride > 0. */
int clearmoe_ffn_forward_ex(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                            const void* b1, const void* U_r, const float* S_r, const void* Vh_r,
                            const void* const* residual_e, const clearmoe_router* router,
                            int32_t E, int32_t r, const clearmoe_ffn_options* opt, void* out,
                            void* stream);

/* The shared basis folded into the experts (Eq. 2 regrouped; the paper materialises W_shared in
 * Phase 3): W_comb[e] = U_r diag(S_r) Vh_r + residual_e[e] for e < E, so that the layer output is
 * y_t = W_comb[a_t] GELU(W1 x_t + b1). W_shared is formed in fp32 (products in fp32, summed over
 * k ascending) and each sum is rounded once to the layer dtype. W_comb is a HOST array of E
 * caller-owned device buffers, each [d x H] row-major like residual_e; computed once per weight
 * set, it replaces the basis step of every later forward. Arguments as clearmoe_ffn_forward. */
int clearmoe_fold_basis(clearmoe_layer* layer, const void* U_r, const float* S_r, const void* Vh_r,
                        const void* const* residual_e, int32_t E, int32_t r, void* const* W_comb,
                        void* stream);

/* The CLEAR-MoE FFN forward on folded weights: routing and fc1 as clearmoe_ffn_forward, then per
 * expert sub-batch out[perm[slot]] = W_comb[e] z in one grouped GEMM (no basis step: the dense
 * FFN's arithmetic plus the routing). Same limits and errors as clearmoe_ffn_forward. */
int clearmoe_ffn_forward_folded(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                                const void* b1, const void* const* W_comb,
                                const clearmoe_router* router, int32_t E, void* out, void* stream);

/* clearmoe_ffn_forward_folded with the deployment options of clearmoe_ffn_forward_ex (fc2 bias,
 * class tokens on the dense path W2, the MLP router); opt may be NULL. Same errors as
 * clearmoe_ffn_forward_ex. */
int clearmoe_ffn_forward_folded_ex(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                                   const void* b1, const void* const* W_comb,
                                   const clearmoe_router* router, int32_t E,
                                   const clearmoe_ffn_options* opt, void* out, void* stream);

/* The paper's own form of the shared basis (Phase 3 text: W_shared materialised before
 * inference): W_sh = U_r diag(S_r) Vh_r as one [d x H] row-major matrix in the layer dtype, formed
 * in fp32 (products in fp32, summed over k ascending) and rounded once. W_sh is a caller-owned
 * device buffer. 1 <= r <= min(max_r, d, H). */
int clearmoe_materialize_basis(clearmoe_layer* layer, const void* U_r, const float* S_r, const void* Vh_r,
                               int32_t r, void* W_sh, void* stream);

/* The CLEAR-MoE FFN forward with the materialised basis (Eq. 2 as the paper computes it):
 * routing and fc1 as clearmoe_ffn_forward, then per expert sub-batch out[perm[slot]] =
 * W_sh z + residual_e[e] z in one grouped GEMM whose K chain is [z | z] x [W_e^res | W_sh]
 * (2 d H multiply-adds per token there, against d (H + r) + r H factorised). Same limits and
 * errors as clearmoe_ffn_forward_folded. */
int clearmoe_ffn_forward_materialized(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                                      const void* b1, const void* W_sh, const void* const* residual_e,
                                      const clearmoe_router* router, int32_t E, void* out, void* stream);

/* clearmoe_ffn_forward_materialized with the deployment options of clearmoe_ffn_forward_ex; opt
 * may be NULL. Same errors as clearmoe_ffn_forward_ex. */
int clearmoe_ffn_forward_materialized_ex(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                                         const void* b1, const void* W_sh, const void* const* residual_e,
                                         const clearmoe_router* router, int32_t E,
                                         const clearmoe_ffn_options* opt, void* out, void* stream);

/* The residual structure of Algorithm 2 exploited: its residual experts are scaled copies of one
 * matrix, W_e^res = s_e R with R = W2 - W_shared, so y_t = W_shared z_t + s_{a_t} R z_t =
 * s_{a_t} (U_r t'_t + R z_t) with t'_t = diag(S_r) Vh_r z_t / s_{a_t}. Routing (idx), fc1, the
 * basis factor (column scale S_r and row scale 1 / s_a) and one GEMM with the K chain
 * [z | t'] x [R | U_r] and row scale s_a, all in token order: no sort, no scatter, one residual
 * matrix instead of E. Exact (up to rounding) only for residuals of that form; s_e [E] fp32
 * device, every s_e finite and non-zero (Algorithm 2's are ratios of mean norms, positive), else
 * the rows of that expert are not finite. R [d x H] row-major in the layer dtype. counts, offsets
 * and perm are still produced (after the output) for clearmoe_get_routing. Errors as
 * clearmoe_ffn_forward. */
int clearmoe_ffn_forward_scaled(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                                const void* b1, const void* U_r, const float* S_r, const void* Vh_r,
                                const void* R, const float* s_e, const clearmoe_router* router,
                                int32_t E, int32_t r, void* out, void* stream);

/* The dense FFN the layer was converted from, on the same device: out = W2 GELU(W1 x + b1)
 * (the comparison path; no bias on fc2, as in Eq. 2). 1 <= T <= max_tokens. */
int clearmoe_dense_ffn_forward(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                               const void* b1, const void* W2, void* out, void* stream);

/* The dense FFN with fc2's bias: out = W2 GELU(W1 x + b1) + b2, b2 [d] in the layer dtype
 * (NULL: as clearmoe_dense_ffn_forward). */
int clearmoe_dense_ffn_forward_ex(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                                  const void* b1, const void* W2, const void* b2, void* out,
                                  void* stream);

/* The dense FFN with the options of clearmoe_ffn_forward_ex that apply to it: b2 (as
 * clearmoe_dense_ffn_forward_ex) and input_layernorm (x is y; LN(y) folded into fc1 as there).
 * opt may be NULL. EINVAL for cls_stride != 0 or a non-NULL mlp_router; opt->W2 is not read. */
int clearmoe_dense_ffn_forward_opt(clearmoe_layer* layer, const void* x, int64_t T, const void* W1,
                                   const void* b1, const void* W2, const clearmoe_ffn_options* opt,
                                   void* out, void* stream);

/* Per-token LayerNorm without affine between stacked sublayers: x_out = (y - mean(y)) /
 * sqrt(var(y) + 1e-6), biased variance, fp32 statistics; y and x_out [T x d] in the layer's
 * dtype (they may alias). 1 <= T <= max_tokens. */
int clearmoe_layer_norm(clearmoe_layer* layer, const void* y, int64_t T, void* x_out,
                        void* stream);

/* Copies (device to device, on `stream`) the routing of the last clearmoe_route /
 * clearmoe_ffn_forward on this handle: idx [T], counts [G], offsets [G + 1], perm [T], all
 * int32 device pointers, G = E (E + 1 when that forward had class tokens: group E is theirs);
 * any may be NULL to skip it. EINVAL if no forward has run yet. */
int clearmoe_get_routing(clearmoe_layer* layer, int32_t* idx, int32_t* counts, int32_t* offsets,
                         int32_t* perm, void* stream);

/* Synchronises the device, returns the handle's device status word (CLEARMOE_OK or the first
 * device-side error since the last call, e.g. CLEARMOE_ETIMEOUT) and clears it; after an error it
 * also clears the handle's split-K arrival counters, which a GEMM that gave up may have left
 * part-counted, so that the next calls run on a consistent handle. */
int clearmoe_layer_status(clearmoe_layer* layer);

/* Fault injection for tests of the bounded waits: every device-side wait of the routing kernel
 * gives up after wait_limit_ns nanoseconds (default 1e9) and, when phantom_arrivals > 0, the
 * bf16 routing withholds the copy of its first stage (the first K blocks of its first 128-row block,
 * in its first CTA), so the MMA thread's wait for it runs out and the call reports
 * CLEARMOE_ETIMEOUT through clearmoe_layer_status; the kernel lets its other copies in flight land
 * before it exits, and the layer stays usable. phantom_arrivals = 0 restores normal use. */
int clearmoe_debug_set_wait(clearmoe_layer* layer, int64_t wait_limit_ns, int32_t phantom_arrivals);

/* Per-stage timing: when n >= 5, clearmoe_ffn_forward records events[0] before its first kernel
 * and events[i] after its i-th kernel (1 routing, 2 fc1 + GELU, 3 shared-basis factor, 4 grouped
 * residual GEMM); clearmoe_dense_ffn_forward records events[0..2] around its two kernels. The
 * events are cudaEvent_t handles owned by the caller, recorded on the call's stream; n = 0 (or
 * events = NULL) turns recording off. The library never waits on them. */
int clearmoe_set_profile_events(clearmoe_layer* layer, void* const* events, int32_t n);

/* Routing without a handle, for callers that cannot allocate device memory (engines that own
 * every device byte and forbid allocation in their enqueue path, processes held to a fixed
 * memory budget, loops that cannot afford cudaMalloc's implicit device synchronisation). The
 * paper has no counterpart: this is a deployment variant of clearmoe_route, with the same results
 * (idx [T], counts [E], offsets [E + 1], perm [T]: caller-owned int32 device outputs) for tokens
 * x [T x d] of dtype `dtype` and the router W [E x d], b [E] in that dtype.
 *   - It calls no cudaMalloc, cudaFree or other allocating routine. Its scratch (per-CTA expert
 *     histograms and a spare status word) is one static device array of 65,600 bytes that every
 *     GPU loading the library holds until exit; it serves up to 1,024 routing CTAs (two per SM on
 *     GPUs with up to 512 SMs). A launch that would need more returns CLEARMOE_EUNSUPPORTED and
 *     enqueues nothing. Between its two kernels idx holds packed per-token words; the second
 *     kernel leaves the experts there.
 *   - The first call on a device looks up the array's device address (once per device, with that
 *     device current); make that first call before any stream capture.
 *   - Every call shares the array and it keeps the last call's contents; each call clears what
 *     must start at zero (the status words; the histograms are rewritten before they are read).
 *     Calls whose work overlaps on the GPU (other streams, other host threads) race on the
 *     array: serialise them.
 *   - status (optional int32 device pointer, else NULL) is set to 0 at the start of the call and
 *     receives CLEARMOE_ETIMEOUT if a bounded device-side wait (1 s) runs out, in which case the
 *     outputs are undefined.
 * Limits: 1 <= T <= 2^30, 1 <= E <= 16; bf16: d % 64 == 0, d <= 1024; fp32: d % 4 == 0, d <= 512;
 * x and W 16-byte aligned. Host-side errors return EINVAL / EUNSUPPORTED / ECUDA with nothing
 * enqueued. */
int clearmoe_route_noalloc(const void* x, int64_t T, int32_t d, int32_t dtype,
                           const clearmoe_router* router, int32_t E, int32_t* idx, int32_t* counts,
                           int32_t* offsets, int32_t* perm, int32_t* status, void* stream);

/* Static string for a status code. */
const char* clearmoe_strerror(int status);

/* Library version as MAJOR * 10000 + MINOR * 100 + PATCH. */
int clearmoe_version(void);

#ifdef __cplusplus
}
#endif

#endif /* CLEARMOE_H */
