/* Float64 oracle of one CLEAR-MoE FFN layer in plain C (arxiv 2606.28516). TEST INFRASTRUCTURE ONLY.
 *
 * A second restatement of the layer, independent of the numpy oracle beside it and of the CUDA
 * library: plain loops over row-major double arrays, every sum taken in ascending index order,
 * libm's erf for GELU. Only the tests (through oracle/ref_c.py) load it; the library never links
 * it. It follows Eq. 2 and Algorithm 3 step by step:
 *   1. z <- GELU(W1 x + b1) for every token (shared fc1)
 *   2. h_sh <- W_shared z with W_shared = U_r diag(S_r) Vh_r formed once (the paper materialises it)
 *   3. a <- argmax of the router's logits, the lowest expert index on ties
 *   4. sort the tokens by a (stable), counts and sub-batch offsets
 *   5. h_res <- W_e^res z for each expert's sub-batch
 *   6. unshuffle and add: y <- h_sh + h_res
 * plus the deployment pieces the library offers: fc2's bias b2 on every row, class tokens on the
 * dense path W2 (group E after the experts), the MLP router, and the per-token LayerNorm of the
 * stacked workload, and the folded and one-residual-matrix forms. Shapes: x [T x d], W1 [H x d],
 * b1 [H], U [d x r], S [r], Vh [r x H], residuals [E x d x H], W_g [E x d], b_g [E], W2 [d x H],
 * b2 [d], y [T x d].
 * Compile with contraction off (-ffp-contract=off) so that x86 and Arm hosts agree bit for bit. */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* v rounded to the nearest value with 8 significant bits (bf16), halves to the even neighbour:
 * v = m 2^e with 1/2 <= |m| < 1, and the result is nearbyint(m 2^8) 2^(e - 8) in the default
 * round-to-nearest-even mode. The bf16 layer's quantisation point of z. */
double cmref_round_bf16(double v) {
    if (v == 0.0 || !isfinite(v)) return v;
    int e;
    const double m = frexp(v, &e);
    return ldexp(nearbyint(ldexp(m, 8)), e - 8);
}

/* GELU(u) = u Phi(u), Phi the standard normal CDF = (1 + erf(u / sqrt 2)) / 2 (Eq. 2's activation). */
double cmref_gelu(double u) { return u * 0.5 * (1.0 + erf(u / sqrt(2.0))); }

/* The linear router's logits g(x_t)_e = sum_k W_g[e, k] x_t[k] + b_g[e] (Phase 4, linear router). */
void cmref_router_logits(const double* x, int64_t T, int d, const double* Wg, const double* bg, int E,
                         double* logits) {
    for (int64_t t = 0; t < T; ++t)
        for (int e = 0; e < E; ++e) {
            double s = 0.0;
            for (int k = 0; k < d; ++k) s += Wg[(int64_t)e * d + k] * x[t * d + k];
            logits[t * E + e] = s + bg[e];
        }
}

/* The MLP router's logits W_out act(W_in x_t + b_in) + b_out (Phase 4, "MLP"; act 0 = ReLU,
 * 1 = GELU). hidden units, W_in [hidden x d], W_out [E x hidden]. */
void cmref_mlp_router_logits(const double* x, int64_t T, int d, const double* W_in, const double* b_in, int hidden,
                             const double* W_out, const double* b_out, int E, int act, double* logits) {
    double* h = (double*)malloc(sizeof(double) * (size_t)(hidden > 0 ? hidden : 1));
    if (!h) return;
    for (int64_t t = 0; t < T; ++t) {
        for (int j = 0; j < hidden; ++j) {
            double u = 0.0;
            for (int k = 0; k < d; ++k) u += W_in[(int64_t)j * d + k] * x[t * d + k];
            u += b_in[j];
            h[j] = act == 1 ? cmref_gelu(u) : (u > 0.0 ? u : 0.0);
        }
        for (int e = 0; e < E; ++e) {
            double s = 0.0;
            for (int j = 0; j < hidden; ++j) s += W_out[(int64_t)e * hidden + j] * h[j];
            logits[t * E + e] = s + b_out[e];
        }
    }
    free(h);
}

/* Algorithm 3 step 3: a_t = the lowest e with the largest logit (a later equal logit never wins).
 * cls_stride > 0: token t with t % cls_stride == 0 is a class token and takes group E (the dense
 * path) without consulting the router. */
void cmref_argmax(const double* logits, int64_t T, int E, int64_t cls_stride, int32_t* a) {
    for (int64_t t = 0; t < T; ++t) {
        if (cls_stride > 0 && t % cls_stride == 0) {
            a[t] = E;
            continue;
        }
        int best = 0;
        for (int e = 1; e < E; ++e)
            if (logits[t * E + e] > logits[t * E + best]) best = e;
        a[t] = best;
    }
}

/* Algorithm 3 step 4, "sort z by a": counts_g = |{t : a_t = g}|, offsets = exclusive prefix sum
 * (G + 1 entries), perm[slot] = token with the tokens of group g in slots [offsets_g,
 * offsets_{g+1}) in increasing token order (a counting sort, which is stable). Returns -1 for an
 * index outside [0, G). */
int cmref_sort_by_group(const int32_t* a, int64_t T, int G, int32_t* counts, int32_t* offsets, int32_t* perm) {
    for (int g = 0; g < G; ++g) counts[g] = 0;
    for (int64_t t = 0; t < T; ++t) {
        if (a[t] < 0 || a[t] >= G) return -1;
        counts[a[t]] += 1;
    }
    offsets[0] = 0;
    for (int g = 0; g < G; ++g) offsets[g + 1] = offsets[g] + counts[g];
    int32_t* next = (int32_t*)malloc(sizeof(int32_t) * (size_t)(G > 0 ? G : 1));
    if (!next) return -1;
    for (int g = 0; g < G; ++g) next[g] = offsets[g];
    for (int64_t t = 0; t < T; ++t) perm[next[a[t]]++] = (int32_t)t;
    free(next);
    return 0;
}

/* Algorithm 3 step 1: z_t = GELU(W1 x_t + b1), stored rounded to bf16 when z_bf16 (the bf16
 * layer's hidden state). */
void cmref_fc1_gelu(const double* x, int64_t T, int d, int H, const double* W1, const double* b1, int z_bf16,
                    double* z) {
    for (int64_t t = 0; t < T; ++t)
        for (int j = 0; j < H; ++j) {
            double u = 0.0;
            for (int k = 0; k < d; ++k) u += W1[(int64_t)j * d + k] * x[t * d + k];
            const double g = cmref_gelu(u + b1[j]);
            z[t * H + j] = z_bf16 ? cmref_round_bf16(g) : g;
        }
}

/* W_shared = U_r Sigma_r V_r^T as a d x H matrix (Eq. 2; formed before inference). */
void cmref_shared_weight(const double* U, const double* S, const double* Vh, int d, int r, int H, double* Wsh) {
    for (int i = 0; i < d; ++i)
        for (int j = 0; j < H; ++j) {
            double s = 0.0;
            for (int k = 0; k < r; ++k) s += U[(int64_t)i * r + k] * S[k] * Vh[(int64_t)k * H + j];
            Wsh[(int64_t)i * H + j] = s;
        }
}

/* y_row = W z_row for W [d x H]. */
static void matvec(const double* W, const double* zr, int d, int H, double* out) {
    for (int i = 0; i < d; ++i) {
        double s = 0.0;
        for (int j = 0; j < H; ++j) s += W[(int64_t)i * H + j] * zr[j];
        out[i] = s;
    }
}

/* Algorithm 3 steps 2 and 4-6 on hidden states z [T x H] with groups a [T]: h_sh = W_shared z for
 * every routed token, the tokens sorted by group, h_res = W_e^res z per expert sub-batch, then
 * unshuffled and added. Tokens of group E (class tokens; only when W2 is given) take the dense path
 * y_t = W2 z_t instead. b2 (nullable) is added to every row. Returns -1 for a group outside
 * [0, E), or E without W2. */
int cmref_experts_forward(const double* z, int64_t T, int d, int H, const double* Wsh, const double* residuals,
                          int E, const int32_t* a, const double* W2, const double* b2, double* y) {
    const int G = E + (W2 ? 1 : 0);
    int32_t* counts = (int32_t*)malloc(sizeof(int32_t) * (size_t)G);
    int32_t* offsets = (int32_t*)malloc(sizeof(int32_t) * (size_t)(G + 1));
    int32_t* perm = (int32_t*)malloc(sizeof(int32_t) * (size_t)(T > 0 ? T : 1));
    double* hsh = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1) * (size_t)d);
    double* hres = (double*)malloc(sizeof(double) * (size_t)d);
    int rc = -1;
    if (!counts || !offsets || !perm || !hsh || !hres) goto done;
    if (cmref_sort_by_group(a, T, G, counts, offsets, perm)) goto done;  /* step 4 */
    for (int64_t t = 0; t < T; ++t)                                       /* step 2 */
        if (a[t] < E) matvec(Wsh, z + t * H, d, H, hsh + t * d);
    for (int g = 0; g < G; ++g)                                           /* steps 5, 6 */
        for (int32_t slot = offsets[g]; slot < offsets[g + 1]; ++slot) {
            const int64_t t = perm[slot];
            if (g < E) {
                matvec(residuals + (int64_t)g * d * H, z + t * H, d, H, hres);
                for (int i = 0; i < d; ++i) y[t * d + i] = hsh[t * d + i] + hres[i];
            } else {
                matvec(W2, z + t * H, d, H, y + t * d);
            }
        }
    if (b2)
        for (int64_t t = 0; t < T; ++t)
            for (int i = 0; i < d; ++i) y[t * d + i] += b2[i];
    rc = 0;
done:
    free(counts);
    free(offsets);
    free(perm);
    free(hsh);
    free(hres);
    return rc;
}

/* The CLEAR-MoE FFN forward (Eq. 2 with Algorithm 3) for a given assignment a (E + 1 = class
 * token when W2 is given): z from fc1, W_shared formed, then the experts. Returns -1 on a bad
 * group index or an allocation failure. */
int cmref_ffn_forward(const double* x, int64_t T, int d, int H, const double* W1, const double* b1,
                      const double* U, const double* S, const double* Vh, int r, const double* residuals, int E,
                      const int32_t* a, const double* W2, const double* b2, int z_bf16, double* y) {
    double* z = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1) * (size_t)H);
    double* Wsh = (double*)malloc(sizeof(double) * (size_t)d * (size_t)H);
    int rc = -1;
    if (z && Wsh) {
        cmref_fc1_gelu(x, T, d, H, W1, b1, z_bf16, z);
        cmref_shared_weight(U, S, Vh, d, r, H, Wsh);
        rc = cmref_experts_forward(z, T, d, H, Wsh, residuals, E, a, W2, b2, y);
    }
    free(z);
    free(Wsh);
    return rc;
}

/* The unconverted layer: y = W2 GELU(W1 x + b1) (+ b2). */
int cmref_dense_ffn(const double* x, int64_t T, int d, int H, const double* W1, const double* b1, const double* W2,
                    const double* b2, int z_bf16, double* y) {
    double* z = (double*)malloc(sizeof(double) * (size_t)H);
    if (!z) return -1;
    for (int64_t t = 0; t < T; ++t) {
        cmref_fc1_gelu(x + t * d, 1, d, H, W1, b1, z_bf16, z);
        matvec(W2, z, d, H, y + t * d);
        if (b2)
            for (int i = 0; i < d; ++i) y[t * d + i] += b2[i];
    }
    free(z);
    return 0;
}

/* Per-token LayerNorm without affine: x_t = (y_t - mean) / sqrt(biased variance + eps), the
 * normalisation between the stacked sublayers. */
void cmref_layer_norm(const double* y, int64_t T, int d, double eps, double* x) {
    for (int64_t t = 0; t < T; ++t) {
        const double* yr = y + t * d;
        double mean = 0.0, var = 0.0;
        for (int k = 0; k < d; ++k) mean += yr[k];
        mean /= d;
        for (int k = 0; k < d; ++k) var += (yr[k] - mean) * (yr[k] - mean);
        var /= d;
        const double inv = 1.0 / sqrt(var + eps);
        for (int k = 0; k < d; ++k) x[t * d + k] = (yr[k] - mean) * inv;
    }
}

/* Eq. 2 regrouped: both terms act on the same z, so W_shared z + W_e^res z = W_comb[e] z with
 * W_comb[e] = W_shared + W_e^res, for every expert e (W_comb [E x d x H]). */
void cmref_fold_basis(const double* U, const double* S, const double* Vh, const double* residuals, int E, int d,
                      int r, int H, double* W_comb) {
    cmref_shared_weight(U, S, Vh, d, r, H, W_comb);  /* W_shared in the first slot */
    for (int e = E - 1; e >= 0; --e)                  /* the last slot first: slot 0 is read below */
        for (int64_t i = 0; i < (int64_t)d * H; ++i) W_comb[(int64_t)e * d * H + i] = W_comb[i] + residuals[(int64_t)e * d * H + i];
}

/* Algorithm 2's residuals are scaled copies of one matrix, W_e^res = s_e R: y_t = W_shared z_t +
 * s_{a_t} R z_t, with z from fc1 as in cmref_ffn_forward. Returns -1 on a bad expert index or an
 * allocation failure. */
int cmref_ffn_forward_scaled(const double* x, int64_t T, int d, int H, const double* W1, const double* b1,
                             const double* U, const double* S, const double* Vh, int r, const double* R,
                             const double* s, int E, const int32_t* a, int z_bf16, double* y) {
    double* z = (double*)malloc(sizeof(double) * (size_t)H);
    double* Wsh = (double*)malloc(sizeof(double) * (size_t)d * (size_t)H);
    double* hsh = (double*)malloc(sizeof(double) * (size_t)d);
    double* hr = (double*)malloc(sizeof(double) * (size_t)d);
    int rc = -1;
    if (!z || !Wsh || !hsh || !hr) goto done;
    cmref_shared_weight(U, S, Vh, d, r, H, Wsh);
    for (int64_t t = 0; t < T; ++t) {
        if (a[t] < 0 || a[t] >= E) goto done;
        cmref_fc1_gelu(x + t * d, 1, d, H, W1, b1, z_bf16, z);
        matvec(Wsh, z, d, H, hsh);
        matvec(R, z, d, H, hr);
        for (int i = 0; i < d; ++i) y[t * d + i] = hsh[i] + s[a[t]] * hr[i];
    }
    rc = 0;
done:
    free(z);
    free(Wsh);
    free(hsh);
    free(hr);
    return rc;
}
