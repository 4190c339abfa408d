/*
 * xpress_oracle.c -- reference CPU oracle for the xPress refinement pass.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / --impl reference legs of bench.py may load this library.
 * The product path (libxpress.so) never links, loads or calls it, and it
 * shares no code, header, table or helper with the CUDA sources.
 *
 * Everything here follows arXiv 2608.02438 ("xPress: Parallel Refinement for
 * Diffusion Drafters in Speculative Decoding") literally, in fp64, with plain
 * loops and no blocking, fusion or reordering beyond what the paper states:
 *
 *   refiner map R_theta            Sec. 4.1, Eq. (fuse), (mix), (mlp), (read),
 *                                  (correct); g = mean of h over the block
 *   refined distribution           Sec. 4.1, Eq. (refined-dist)
 *   Jacobi refinement              Sec. 4.2, Algorithm 1, Eq. (jacobi-update)
 *   sequential decode Y*           Sec. 4.2, Theorem 1
 *   greedy acceptance              Sec. 3.1 (longest matching prefix + 1)
 *   lossless acceptance            Sec. 3.1 and Sec. 4.3 (accept w.p.
 *                                  min(1, p/q), else resample max(0, p-q))
 *   training objective             Sec. 4.3 (cross-entropy + L1 / total
 *                                  variation, position weights, drafter
 *                                  anchor, consistency forward)
 *   base logits s = W_lm h         Sec. 4.1 / Fig. 2a (the target-sized LM
 *                                  head that produces s_k; Algorithm 1's
 *                                  Y^(0) = argmax s)
 *
 * Readings of points the paper leaves open:
 *   - sigma is selectable: SiLU (default), GELU(erf), ReLU (Sec. 4.1 says only
 *     "a pointwise nonlinearity");
 *   - no biases or norms (the equations have none);
 *   - x_0 is a per-sequence anchor token id;
 *   - Y^(0) is the given draft, or argmax s when none is given (Algorithm 1);
 *   - ties in argmax go to the smallest token id (Theorem 1's "fixed rule");
 *   - T > 0 refinement (the paper defines only argmax) re-selects with a
 *     FIXED-NOISE hierarchical Gumbel-max: the vocabulary is cut into groups of
 *     XO_GROUP consecutive ids; a group is drawn with probability
 *     proportional to its mass (Gumbel-max over the group log-sum-exp), then a
 *     token inside it (Gumbel-max over the members).  The noise depends on
 *     (seed, offset, position, id) but not on the iteration, so each update is
 *     a deterministic function of the prefix and Theorem 1 still holds; the
 *     draw is an exact sample of softmax(l/T);
 *   - bf16 precision contract: weights, h, s and target logits are stored in
 *     bf16; the activations that feed a tensor-core product (c before W_1, the
 *     activation u before W_2, z before W_r) are rounded to bf16
 *     (round-to-nearest-even); everything else is exact here (fp64).  In the
 *     fp32 configuration nothing is rounded.
 *   - a decision that floating point turns into an integer (argmax, a Gumbel
 *     comparison, the accept test) is taken on values rounded to fp32, the
 *     precision the kernels decide in; ties resolve to the smallest index.
 *   - training (Sec. 4.3): lambda weighs the drafter-anchor term and beta the
 *     consistency term, as in the total-loss equation; every softmax at
 *     T = 1; the bf16 operand roundings pass the gradient straight through;
 *     sgn(0) = 0 in the L1 subgradient; the consistency forward takes the
 *     first argmax of s_{k-1} as x_k (x_0 the anchor); the target logits are
 *     those of the B positions themselves and w_k = exp(-(k-1)/gamma) for
 *     k = 1..B; the drafter's own parameters are out of scope, so L(p^b)
 *     contributes a value and no gradient.
 *
 * Random numbers: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11), written
 * here from its published definition.  key = (seed low 32, seed high 32),
 * counter = (index >> 2, position, stream, offset), output word index & 3;
 * u = ((x >> 9) + 0.5) * 2^-23, exact in fp32 and strictly inside (0, 1).
 * Streams: 0 group noise, 1 in-group noise, 2 accept uniforms,
 * 3 residual / bonus noise.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define XO_GROUP 32

enum { XO_F32 = 0, XO_BF16 = 1 };
enum { XO_SILU = 0, XO_GELU = 1, XO_RELU = 2 };
enum { XO_STREAM_GROUP = 0, XO_STREAM_ELEM = 1, XO_STREAM_ACCEPT = 2, XO_STREAM_RESID = 3 };

/* Refiner definition (Sec. 4.1).  Row-major storage:
 *   W_e  [V, r]   row x is the paper's column W_e[x] of W_e in R^{r x V}
 *   W_h  [r, H], W_g [r, H], W_in [r, 3r], L [r, B, B] (L[d][k][j] = L^(d)_{k,j}),
 *   W1   [2r, r], W2 [r, 2r], W_r [V, r].                                    */
typedef struct {
    int H, V, r, B;
    int dtype; /* XO_F32 or XO_BF16: storage of weights and of h, s, target */
    int act;   /* XO_SILU, XO_GELU, XO_RELU */
    const void *W_e, *W_h, *W_g, *W_in, *L, *W1, *W2, *W_r;
} xo_model;

/* ------------------------------------------------------------------ helpers */

static double ld(const void *p, int dtype, size_t i)
{
    if (dtype == XO_F32) return (double)((const float *)p)[i];
    uint32_t u = (uint32_t)((const uint16_t *)p)[i] << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

/* Round to the nearest bf16 value (8 significant bits, fp32 exponent range),
 * ties to even.  Used only at the tensor-core operand points. */
double xo_round_bf16(double x)
{
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    double m = frexp(fabs(x), &e);      /* |x| = m * 2^e, m in [0.5, 1) */
    double q;
    if (e - 1 < -126) {                 /* bf16 subnormal range: step 2^-133 */
        q = rint(fabs(x) * ldexp(1.0, 133)) * ldexp(1.0, -133);
    } else {
        q = ldexp(rint(m * 256.0), e - 8);
    }
    if (q > 3.3895313892515355e38) q = INFINITY;
    return x < 0 ? -q : q;
}

static double opround(const xo_model *M, double x)
{
    return M->dtype == XO_BF16 ? xo_round_bf16(x) : x;
}

static double sigma(int act, double t)
{
    switch (act) {
    case XO_RELU: return t > 0 ? t : 0.0;
    case XO_GELU: return 0.5 * t * (1.0 + erf(t / sqrt(2.0)));
    default: return t / (1.0 + exp(-t));
    }
}

/* ------------------------------------------------------------------ Philox */

void xo_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int round = 0; round < 10; ++round) {
        uint64_t p0 = (uint64_t)0xD2511F53u * c0;
        uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
        uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
        uint32_t n1 = (uint32_t)p1;
        uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
        uint32_t n3 = (uint32_t)p0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* Uniform in (0,1) for element `index` of (position, stream, offset). */
double xo_uniform(uint64_t seed, uint32_t index, uint32_t position, uint32_t stream, uint32_t offset)
{
    uint32_t ctr[4] = {index >> 2, position, stream, offset};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    xo_philox4x32_10(ctr, key, out);
    uint32_t x = out[index & 3u];
    return ((double)(x >> 9) + 0.5) * (1.0 / 8388608.0);
}

double xo_gumbel(uint64_t seed, uint32_t index, uint32_t position, uint32_t stream, uint32_t offset)
{
    double u = xo_uniform(seed, index, position, stream, offset);
    return -log(-log(u));
}

/* ------------------------------------------------------------ refiner map */

/* Token-independent part of Fuse (Eq. fuse): u_h,k = W_h h_k and u_g = W_g g
 * with g = (1/B) sum_j h_j.  Outputs uh [B, r], ug [r]. */
static void fuse_hidden(const xo_model *M, const void *h, double *uh, double *ug)
{
    const int H = M->H, r = M->r, B = M->B;
    double *g = (double *)calloc((size_t)H, sizeof(double));
    for (int j = 0; j < B; ++j)
        for (int i = 0; i < H; ++i) g[i] += ld(h, M->dtype, (size_t)j * H + i);
    for (int i = 0; i < H; ++i) g[i] /= B;
    for (int d = 0; d < r; ++d) {
        double acc = 0.0;
        for (int i = 0; i < H; ++i) acc += ld(M->W_g, M->dtype, (size_t)d * H + i) * g[i];
        ug[d] = acc;
    }
    for (int k = 0; k < B; ++k)
        for (int d = 0; d < r; ++d) {
            double acc = 0.0;
            for (int i = 0; i < H; ++i)
                acc += ld(M->W_h, M->dtype, (size_t)d * H + i) * ld(h, M->dtype, (size_t)k * H + i);
            uh[(size_t)k * r + d] = acc;
        }
    free(g);
}

/* Fuse (Eq. fuse) and Mix (Eq. mix) for positions 0..upto (0-based), given
 * x[0..B-1] = (x_0, ..., x_{B-1}).  Writes c [B, r] rows 0..upto. */
static void fuse_mix(const xo_model *M, const double *uh, const double *ug, const int32_t *x,
                     int upto, double *a, double *c)
{
    const int r = M->r, B = M->B;
    for (int k = 0; k <= upto; ++k) {
        size_t erow = (size_t)x[k] * r;
        for (int d = 0; d < r; ++d) {
            const size_t wrow = (size_t)d * 3 * r;
            double acc = 0.0;
            for (int e = 0; e < r; ++e) acc += ld(M->W_in, M->dtype, wrow + e) * uh[(size_t)k * r + e];
            for (int e = 0; e < r; ++e) acc += ld(M->W_in, M->dtype, wrow + r + e) * ug[e];
            for (int e = 0; e < r; ++e)
                acc += ld(M->W_in, M->dtype, wrow + 2 * r + e) * ld(M->W_e, M->dtype, erow + e);
            a[(size_t)k * r + d] = acc;
        }
    }
    for (int k = 0; k <= upto; ++k)
        for (int d = 0; d < r; ++d) {
            double acc = a[(size_t)k * r + d];
            for (int j = 0; j < k; ++j)
                acc += ld(M->L, M->dtype, ((size_t)d * B + k) * B + j) * a[(size_t)j * r + d];
            c[(size_t)k * r + d] = acc;
        }
}

/* Trans (Eq. mlp) for one position: z = c + W2 sigma(W1 c); returns the
 * unrounded z and the W_r operand zop (bf16-rounded in the bf16 contract). */
static void trans(const xo_model *M, const double *ck, double *zk, double *zop)
{
    const int r = M->r;
    double *cop = (double *)malloc(sizeof(double) * r);
    double *uop = (double *)malloc(sizeof(double) * 2 * r);
    for (int d = 0; d < r; ++d) cop[d] = opround(M, ck[d]);
    for (int o = 0; o < 2 * r; ++o) {
        double t = 0.0;
        for (int d = 0; d < r; ++d) t += ld(M->W1, M->dtype, (size_t)o * r + d) * cop[d];
        uop[o] = opround(M, sigma(M->act, t));
    }
    for (int d = 0; d < r; ++d) {
        double acc = 0.0;
        for (int o = 0; o < 2 * r; ++o) acc += ld(M->W2, M->dtype, (size_t)d * 2 * r + o) * uop[o];
        zk[d] = ck[d] + acc;
        zop[d] = opround(M, zk[d]);
    }
    free(cop);
    free(uop);
}

/* Read (Eq. read) and Correct (Eq. correct) for one position. */
static void read_correct(const xo_model *M, const void *s, int k, const double *zop, double *ell)
{
    const int r = M->r, V = M->V;
    for (int v = 0; v < V; ++v) {
        double acc = 0.0;
        for (int d = 0; d < r; ++d) acc += ld(M->W_r, M->dtype, (size_t)v * r + d) * zop[d];
        ell[v] = ld(s, M->dtype, (size_t)k * V + v) + acc;
    }
}

/* The refiner R_theta composed with Correct, for all B positions.
 * x[0..B-1] = (x_0 = anchor, x_1, ..., x_{B-1}).  Any output may be NULL. */
int xo_forward(const xo_model *M, const void *h, const void *s, const int32_t *x,
               double *ell, double *z, double *c_out)
{
    const int r = M->r, B = M->B, V = M->V;
    for (int k = 0; k < B; ++k)
        if (x[k] < 0 || x[k] >= V) return -1;
    double *uh = (double *)malloc(sizeof(double) * (size_t)B * r);
    double *ug = (double *)malloc(sizeof(double) * r);
    double *a = (double *)malloc(sizeof(double) * (size_t)B * r);
    double *c = (double *)malloc(sizeof(double) * (size_t)B * r);
    double *zk = (double *)malloc(sizeof(double) * r);
    double *zop = (double *)malloc(sizeof(double) * r);
    fuse_hidden(M, h, uh, ug);
    fuse_mix(M, uh, ug, x, B - 1, a, c);
    for (int k = 0; k < B; ++k) {
        trans(M, c + (size_t)k * r, zk, zop);
        if (z) memcpy(z + (size_t)k * r, zk, sizeof(double) * r);
        if (ell) read_correct(M, s, k, zop, ell + (size_t)k * V);
    }
    if (c_out) memcpy(c_out, c, sizeof(double) * (size_t)B * r);
    free(uh); free(ug); free(a); free(c); free(zk); free(zop);
    return 0;
}

/* --------------------------------------------------------------- selection */

/* First index of the maximum of fp32-rounded values; top-2 margin in fp64. */
static int argmax_f32(const double *x, int n, double *margin)
{
    int best = 0;
    float bv = (float)x[0];
    for (int i = 1; i < n; ++i)
        if ((float)x[i] > bv) { bv = (float)x[i]; best = i; }
    if (margin) {
        double second = -INFINITY;
        for (int i = 0; i < n; ++i)
            if (i != best && x[i] > second) second = x[i];
        *margin = n > 1 ? x[best] - second : INFINITY;
    }
    return best;
}

/* Re-select position k (0-based) from its corrected logits ell[0..V-1]
 * (Algorithm 1 inner loop; Eq. refined-dist for T > 0).
 * Outputs: *y; for T > 0 also *lse = log sum_v exp(ell_v / T) and
 * *sel = ell_y / T; *margin = smallest top-2 gap of the decisions taken. */
int xo_select(const double *ell, int V, double T, uint64_t seed, uint32_t offset, int k,
              int32_t *y, double *lse, double *sel, double *margin)
{
    double mg = INFINITY;
    if (T <= 0.0) {
        int v = argmax_f32(ell, V, &mg);
        *y = v;
        if (sel) *sel = ell[v];
        if (lse) *lse = NAN;
        if (margin) *margin = mg;
        return 0;
    }
    const int G = (V + XO_GROUP - 1) / XO_GROUP;
    double *x = (double *)malloc(sizeof(double) * V);
    double *score = (double *)malloc(sizeof(double) * G);
    double mx = -INFINITY;
    for (int v = 0; v < V; ++v) {
        x[v] = ell[v] / T;
        if (x[v] > mx) mx = x[v];
    }
    double tot = 0.0;
    for (int v = 0; v < V; ++v) tot += exp(x[v] - mx);
    for (int g = 0; g < G; ++g) {
        int lo = g * XO_GROUP, hi = lo + XO_GROUP < V ? lo + XO_GROUP : V;
        double gm = -INFINITY, gs = 0.0;
        for (int v = lo; v < hi; ++v) if (x[v] > gm) gm = x[v];
        for (int v = lo; v < hi; ++v) gs += exp(x[v] - gm);
        score[g] = gm + log(gs) + xo_gumbel(seed, (uint32_t)g, (uint32_t)k, XO_STREAM_GROUP, offset);
    }
    double m1;
    int gsel = argmax_f32(score, G, &m1);
    int lo = gsel * XO_GROUP, hi = lo + XO_GROUP < V ? lo + XO_GROUP : V;
    double *es = (double *)malloc(sizeof(double) * (hi - lo));
    for (int v = lo; v < hi; ++v)
        es[v - lo] = x[v] + xo_gumbel(seed, (uint32_t)v, (uint32_t)k, XO_STREAM_ELEM, offset);
    double m2;
    int vsel = lo + argmax_f32(es, hi - lo, &m2);
    *y = vsel;
    if (sel) *sel = x[vsel];
    if (lse) *lse = mx + log(tot);
    mg = m1 < m2 ? m1 : m2;
    if (margin) *margin = mg;
    free(x); free(score); free(es);
    return 0;
}

/* ------------------------------------------------------ Jacobi refinement */

/* Algorithm 1.  draft may be NULL (then Y^(0) = argmax_v s_k,v).
 * fixed_K != 0 runs exactly K_max passes (no break); converged then reports
 * whether the last pass left the block unchanged.
 * Outputs (per position, from the last executed pass): tokens [B], lse [B],
 * sel [B], z_final [B, r] (unrounded z); iters, converged; min_margin = the
 * smallest decision margin over all passes; traj [(K_max+1) * B] (optional)
 * holds Y^(0..iters) and margins [K_max * B] (optional) the per-pass margins. */
int xo_jacobi(const xo_model *M, const void *h, const void *s, int32_t anchor, const int32_t *draft,
              double T, uint64_t seed, uint32_t offset, int K_max, int fixed_K,
              int32_t *tokens, int32_t *iters, int32_t *converged, double *lse, double *sel,
              double *z_final, double *min_margin, int32_t *traj, double *margins)
{
    const int B = M->B, V = M->V, r = M->r;
    if (anchor < 0 || anchor >= V || K_max < 1) return -1;
    if (draft)
        for (int k = 0; k < B; ++k)
            if (draft[k] < 0 || draft[k] >= V) return -1;
    int32_t *Y = (int32_t *)malloc(sizeof(int32_t) * B);
    int32_t *Yn = (int32_t *)malloc(sizeof(int32_t) * B);
    int32_t *x = (int32_t *)malloc(sizeof(int32_t) * B);
    double *ell = (double *)malloc(sizeof(double) * (size_t)B * V);
    double *z = (double *)malloc(sizeof(double) * (size_t)B * r);
    double *srow = (double *)malloc(sizeof(double) * V);
    double mm = INFINITY;
    for (int k = 0; k < B; ++k) {
        if (draft) {
            Y[k] = draft[k];
        } else {
            for (int v = 0; v < V; ++v) srow[v] = ld(s, M->dtype, (size_t)k * V + v);
            Y[k] = argmax_f32(srow, V, NULL);
        }
    }
    if (traj) memcpy(traj, Y, sizeof(int32_t) * B);
    int it = 0, conv = 0;
    for (int j = 0; j < K_max; ++j) {
        x[0] = anchor;
        for (int k = 1; k < B; ++k) x[k] = Y[k - 1];
        xo_forward(M, h, s, x, ell, z, NULL);
        int same = 1;
        for (int k = 0; k < B; ++k) {
            double mg;
            xo_select(ell + (size_t)k * V, V, T, seed, offset, k, &Yn[k], lse ? &lse[k] : NULL,
                      sel ? &sel[k] : NULL, &mg);
            if (margins) margins[(size_t)j * B + k] = mg;
            if (mg < mm) mm = mg;
            if (Yn[k] != Y[k]) same = 0;
        }
        it = j + 1;
        memcpy(Y, Yn, sizeof(int32_t) * B);
        if (traj) memcpy(traj + (size_t)it * B, Y, sizeof(int32_t) * B);
        conv = same;
        if (same && !fixed_K) break;
    }
    memcpy(tokens, Y, sizeof(int32_t) * B);
    *iters = it;
    *converged = conv;
    if (z_final) memcpy(z_final, z, sizeof(double) * (size_t)B * r);
    if (min_margin) *min_margin = mm;
    free(Y); free(Yn); free(x); free(ell); free(z); free(srow);
    return 0;
}

/* Sequential decode (Theorem 1): y*_k = Select(R(y*_{<k}))_k for k = 1..B,
 * evaluating only position k at step k.  margins [B] optional. */
int xo_sequential(const xo_model *M, const void *h, const void *s, int32_t anchor, double T,
                  uint64_t seed, uint32_t offset, int32_t *ystar, double *margins)
{
    const int B = M->B, V = M->V, r = M->r;
    if (anchor < 0 || anchor >= V) return -1;
    double *uh = (double *)malloc(sizeof(double) * (size_t)B * r);
    double *ug = (double *)malloc(sizeof(double) * r);
    double *a = (double *)malloc(sizeof(double) * (size_t)B * r);
    double *c = (double *)malloc(sizeof(double) * (size_t)B * r);
    double *zk = (double *)malloc(sizeof(double) * r);
    double *zop = (double *)malloc(sizeof(double) * r);
    double *ell = (double *)malloc(sizeof(double) * V);
    int32_t *x = (int32_t *)calloc((size_t)B, sizeof(int32_t));
    fuse_hidden(M, h, uh, ug);
    x[0] = anchor;
    for (int k = 0; k < B; ++k) {
        fuse_mix(M, uh, ug, x, k, a, c);
        trans(M, c + (size_t)k * r, zk, zop);
        read_correct(M, s, k, zop, ell);
        double mg;
        xo_select(ell, V, T, seed, offset, k, &ystar[k], NULL, NULL, &mg);
        if (margins) margins[k] = mg;
        if (k + 1 < B) x[k + 1] = ystar[k];
    }
    free(uh); free(ug); free(a); free(c); free(zk); free(zop); free(ell); free(x);
    return 0;
}

/* --------------------------------------------------------------- accept */

/* Acceptance against target logits tgt [(B+1), V] (Sec. 3.1).
 * T == 0: greedy -- t_k = argmax tgt_k, n = longest prefix with y_k = t_k;
 *         emit y_1..y_n, t_{n+1}.
 * T > 0:  lossless rejection sampling.  q_k(y_k) = exp(sel_k - lse_k) from
 *         the last refinement pass; p_k = softmax(tgt_k / T).  Accept y_k if
 *         u_k q_k(y_k) < p_k(y_k) (u_k from stream 2); at the first reject
 *         sample from max(0, p_k - q_k) (q_k recomputed as softmax(l_k / T)
 *         from z_final; Gumbel-max on stream 3; if the residual has no mass,
 *         sample p_k); if all B are accepted, the bonus is a Gumbel-max draw
 *         from p_{B+1} (stream 3, position B).
 * out [B+1] = emitted tokens then -1; returns n in *accept_len.
 * margin: smallest decision margin (relative for the accept tests).
 * gaps [B+2] (optional): gaps[k] for k < B is the margin of the decision at
 * position k (T = 0: the top-2 gap of target row k, for the rows examined;
 * T > 0: |u q - p| / p of the accept test, for the positions tested), and
 * gaps[B+1] the top-2 margin of the token drawn or taken at the end; entries
 * not decided are +inf. */
int xo_accept(const xo_model *M, const void *tgt, const void *s, const int32_t *y,
              const double *lse, const double *sel, const double *z_final, double T,
              uint64_t seed, uint32_t offset, int32_t *accept_len, int32_t *out, double *margin,
              double *gaps)
{
    const int B = M->B, V = M->V, r = M->r;
    double *row = (double *)malloc(sizeof(double) * V);
    double *sc = (double *)malloc(sizeof(double) * V);
    double mg = INFINITY, m1;
    int n = 0;
    for (int k = 0; k <= B; ++k) out[k] = -1;
    if (gaps)
        for (int k = 0; k < B + 2; ++k) gaps[k] = INFINITY;
    if (T <= 0.0) {
        for (;;) {
            for (int v = 0; v < V; ++v) row[v] = ld(tgt, M->dtype, (size_t)n * V + v);
            int t = argmax_f32(row, V, &m1);
            if (m1 < mg) mg = m1;
            if (gaps) gaps[n < B ? n : B + 1] = m1;
            if (n < B && y[n] == t) { out[n] = y[n]; ++n; continue; }
            out[n] = t;
            if (gaps && n < B) gaps[B + 1] = m1;
            break;
        }
    } else {
        int rejected = 0;
        for (; n < B; ++n) {
            double mx = -INFINITY, tot = 0.0;
            for (int v = 0; v < V; ++v) {
                row[v] = ld(tgt, M->dtype, (size_t)n * V + v) / T;
                if (row[v] > mx) mx = row[v];
            }
            for (int v = 0; v < V; ++v) tot += exp(row[v] - mx);
            double lse_p = mx + log(tot);
            double p_y = exp(row[y[n]] - lse_p);
            double q_y = exp(sel[n] - lse[n]);
            double u = xo_uniform(seed, 0u, (uint32_t)n, XO_STREAM_ACCEPT, offset);
            double rel = fabs(u * q_y - p_y) / (p_y > 0 ? p_y : 1e-300);
            if (rel < mg) mg = rel;
            if (gaps) gaps[n] = rel;
            if ((float)(u * q_y) < (float)p_y) { out[n] = y[n]; continue; }
            rejected = 1;
            /* residual max(0, p - q) at position n */
            double *zop = (double *)malloc(sizeof(double) * r);
            double *ell = (double *)malloc(sizeof(double) * V);
            for (int d = 0; d < r; ++d) zop[d] = opround(M, z_final[(size_t)n * r + d]);
            read_correct(M, s, n, zop, ell);
            double qm = -INFINITY, qt = 0.0;
            for (int v = 0; v < V; ++v) { ell[v] /= T; if (ell[v] > qm) qm = ell[v]; }
            for (int v = 0; v < V; ++v) qt += exp(ell[v] - qm);
            double lse_q = qm + log(qt);
            int any = 0;
            for (int v = 0; v < V; ++v) {
                double res = exp(row[v] - lse_p) - exp(ell[v] - lse_q);
                if (res > 0) {
                    sc[v] = log(res) + xo_gumbel(seed, (uint32_t)v, (uint32_t)n, XO_STREAM_RESID, offset);
                    any = 1;
                } else {
                    sc[v] = -INFINITY;
                }
            }
            if (!any)
                for (int v = 0; v < V; ++v)
                    sc[v] = row[v] + xo_gumbel(seed, (uint32_t)v, (uint32_t)n, XO_STREAM_RESID, offset);
            out[n] = argmax_f32(sc, V, &m1);
            if (m1 < mg) mg = m1;
            if (gaps) gaps[B + 1] = m1;
            free(zop); free(ell);
            break;
        }
        if (!rejected) {
            for (int v = 0; v < V; ++v)
                sc[v] = ld(tgt, M->dtype, (size_t)B * V + v) / T +
                        xo_gumbel(seed, (uint32_t)v, (uint32_t)B, XO_STREAM_RESID, offset);
            out[B] = argmax_f32(sc, V, &m1);
            if (m1 < mg) mg = m1;
            if (gaps) gaps[B + 1] = m1;
        }
    }
    *accept_len = n;
    if (margin) *margin = mg;
    free(row); free(sc);
    return 0;
}

/* ------------------------------------------------------------ base logits */

/* s_n = W_lm h_n for N hidden states (Sec. 4.1, Fig. 2a: the LM head that
 * produces the drafter's base logits s_k), W_lm [V, H] and h [N, H] in the
 * storage dtype.  Outputs: s_exact [N, V] (fp64 sums, optional); s_store
 * [N, V] in the storage dtype (bf16 bit patterns rounded to nearest even, or
 * fp32); argmax [N] = first index of the maximum of the stored row (Algorithm
 * 1's Y^(0) = argmax_v s_k,v, taken on s as stored). */
int xo_lm_head(const void *W_lm, const void *h, int V, int H, int N, int dtype, double *s_exact, void *s_store,
               int32_t *argmax)
{
    if (V < 1 || H < 1 || N < 1) return -1;
    double *row = (double *)malloc(sizeof(double) * V);
    for (int n = 0; n < N; ++n) {
        for (int v = 0; v < V; ++v) {
            double acc = 0.0;
            for (int i = 0; i < H; ++i)
                acc += ld(W_lm, dtype, (size_t)v * H + i) * ld(h, dtype, (size_t)n * H + i);
            if (s_exact) s_exact[(size_t)n * V + v] = acc;
            if (dtype == XO_BF16) {
                const float f = (float)xo_round_bf16(acc);
                uint32_t u;
                memcpy(&u, &f, 4);
                if (s_store) ((uint16_t *)s_store)[(size_t)n * V + v] = (uint16_t)(u >> 16);
                row[v] = (double)f;
            } else {
                const float f = (float)acc;
                if (s_store) ((float *)s_store)[(size_t)n * V + v] = f;
                row[v] = (double)f;
            }
        }
        int best = 0;
        for (int v = 1; v < V; ++v)
            if (row[v] > row[best]) best = v;
        if (argmax) argmax[n] = best;
    }
    free(row);
    return 0;
}

/* ------------------------------------------------------------ training */

/* d sigma / dt for the three readings of sigma. */
static double sigma_prime(int act, double t)
{
    switch (act) {
    case XO_RELU: return t > 0 ? 1.0 : 0.0;
    case XO_GELU: return 0.5 * (1.0 + erf(t / sqrt(2.0))) + t * exp(-0.5 * t * t) / sqrt(2.0 * 3.14159265358979323846);
    default: {
        const double sg = 1.0 / (1.0 + exp(-t));
        return sg + t * sg * (1.0 - sg);
    }
    }
}

/* Gradients of the refiner weights (fp64, same shapes and layouts as xo_model's
 * tensors). */
typedef struct {
    double *W_e, *W_h, *W_g, *W_in, *L, *W1, *W2, *W_r;
} xo_grads;

/* log sum exp and softmax of row[0..n-1]. */
static double softmax_row(const double *row, int n, double *p)
{
    double mx = -INFINITY;
    for (int v = 0; v < n; ++v) if (row[v] > mx) mx = row[v];
    double tot = 0.0;
    for (int v = 0; v < n; ++v) tot += exp(row[v] - mx);
    const double lse = mx + log(tot);
    if (p) for (int v = 0; v < n; ++v) p[v] = exp(row[v] - lse);
    return lse;
}

/* The per-position loss of Sec. 4.3 for distribution p (softmax of ell) at
 * position k against the target distribution q = softmax(tgt_k) and the
 * ground-truth token y*:  a_ce (-log p(y*)) + a_l1 |p - q|_1.  With dl given,
 * also its gradient with respect to ell, times `scale`:
 *   a_ce (p_v - [v = y*]) + a_l1 p_v (sgn(p_v - q_v) - sum_u sgn(p_u - q_u) p_u). */
static double position_loss(const double *ell, const double *tgtrow, int V, int ystar, double a_ce, double a_l1,
                            double scale, double *dl, double *p, double *q)
{
    const double lse = softmax_row(ell, V, p);
    softmax_row(tgtrow, V, q);
    double l1 = 0.0, S = 0.0;
    for (int v = 0; v < V; ++v) {
        const double d = p[v] - q[v];
        l1 += fabs(d);
        S += (d > 0 ? 1.0 : (d < 0 ? -1.0 : 0.0)) * p[v];
    }
    if (dl)
        for (int v = 0; v < V; ++v) {
            const double d = p[v] - q[v];
            const double sg = d > 0 ? 1.0 : (d < 0 ? -1.0 : 0.0);
            dl[v] = scale * (a_ce * (p[v] - (v == ystar ? 1.0 : 0.0)) + a_l1 * p[v] * (sg - S));
        }
    return a_ce * (lse - ell[ystar]) + a_l1 * l1;
}

/* One refiner forward with token inputs x[0..B-1] (x_0 the anchor), the loss
 * L(p) = sum_k w_k loss_k of its refined distributions p_k = softmax(l_k)
 * (T = 1) against the ground truth ystar and the target logits, and, with g
 * given, mult * dL/dtheta added into g.  The bf16 operand roundings of the
 * forward (c before W_1, sigma(W_1 c) before W_2, z before W_r) pass the
 * gradient through unchanged (straight-through). */
static double refiner_loss(const xo_model *M, const void *h, const void *s, const void *tgt, const int32_t *x,
                           const int32_t *ystar, double a_ce, double a_l1, double gam, double mult, xo_grads *g)
{
    const int H = M->H, V = M->V, r = M->r, B = M->B, R2 = 2 * r;
    double *uh = calloc((size_t)B * r, 8), *ug = calloc(r, 8), *gm = calloc(H, 8);
    double *a = calloc((size_t)B * r, 8), *c = calloc((size_t)B * r, 8), *cop = calloc((size_t)B * r, 8);
    double *tp = calloc((size_t)B * R2, 8), *uop = calloc((size_t)B * R2, 8);
    double *z = calloc((size_t)B * r, 8), *zop = calloc((size_t)B * r, 8);
    double *ell = malloc(sizeof(double) * V), *tr = malloc(sizeof(double) * V), *dl = malloc(sizeof(double) * V);
    double *p = malloc(sizeof(double) * V), *q = malloc(sizeof(double) * V);
    double *dz = calloc((size_t)B * r, 8), *dc = calloc((size_t)B * r, 8), *da = calloc((size_t)B * r, 8);
    double *du = calloc(R2, 8), *dt = calloc(R2, 8), *dug = calloc(r, 8);
    /* Fuse: u_h,k = W_h h_k, g = mean_j h_j, u_g = W_g g, a_k = W_in [u_h,k; u_g; W_e[x_k]] */
    for (int j = 0; j < B; ++j)
        for (int i = 0; i < H; ++i) gm[i] += ld(h, M->dtype, (size_t)j * H + i);
    for (int i = 0; i < H; ++i) gm[i] /= B;
    for (int d = 0; d < r; ++d) {
        double acc = 0.0;
        for (int i = 0; i < H; ++i) acc += ld(M->W_g, M->dtype, (size_t)d * H + i) * gm[i];
        ug[d] = acc;
        for (int k = 0; k < B; ++k) {
            double ah = 0.0;
            for (int i = 0; i < H; ++i) ah += ld(M->W_h, M->dtype, (size_t)d * H + i) * ld(h, M->dtype, (size_t)k * H + i);
            uh[(size_t)k * r + d] = ah;
        }
    }
    for (int k = 0; k < B; ++k)
        for (int d = 0; d < r; ++d) {
            double acc = 0.0;
            for (int e = 0; e < r; ++e) {
                acc += ld(M->W_in, M->dtype, (size_t)d * 3 * r + e) * uh[(size_t)k * r + e];
                acc += ld(M->W_in, M->dtype, (size_t)d * 3 * r + r + e) * ug[e];
                acc += ld(M->W_in, M->dtype, (size_t)d * 3 * r + 2 * r + e) * ld(M->W_e, M->dtype, (size_t)x[k] * r + e);
            }
            a[(size_t)k * r + d] = acc;
        }
    /* Mix: c_k = a_k + sum_{j<k} L_kj a_j (per channel) */
    for (int k = 0; k < B; ++k)
        for (int d = 0; d < r; ++d) {
            double acc = a[(size_t)k * r + d];
            for (int j = 0; j < k; ++j) acc += ld(M->L, M->dtype, ((size_t)d * B + k) * B + j) * a[(size_t)j * r + d];
            c[(size_t)k * r + d] = acc;
        }
    /* Trans: z = c + W_2 sigma(W_1 c) */
    for (int k = 0; k < B; ++k) {
        for (int d = 0; d < r; ++d) cop[(size_t)k * r + d] = opround(M, c[(size_t)k * r + d]);
        for (int o = 0; o < R2; ++o) {
            double acc = 0.0;
            for (int d = 0; d < r; ++d) acc += ld(M->W1, M->dtype, (size_t)o * r + d) * cop[(size_t)k * r + d];
            tp[(size_t)k * R2 + o] = acc;
            uop[(size_t)k * R2 + o] = opround(M, sigma(M->act, acc));
        }
        for (int d = 0; d < r; ++d) {
            double acc = 0.0;
            for (int o = 0; o < R2; ++o) acc += ld(M->W2, M->dtype, (size_t)d * R2 + o) * uop[(size_t)k * R2 + o];
            z[(size_t)k * r + d] = c[(size_t)k * r + d] + acc;
            zop[(size_t)k * r + d] = opround(M, z[(size_t)k * r + d]);
        }
    }
    /* Read + Correct (Eq. read / correct), the loss, and dL/dl -> W_r, z */
    double L = 0.0;
    for (int k = 0; k < B; ++k) {
        for (int v = 0; v < V; ++v) {
            double acc = 0.0;
            for (int d = 0; d < r; ++d) acc += ld(M->W_r, M->dtype, (size_t)v * r + d) * zop[(size_t)k * r + d];
            ell[v] = ld(s, M->dtype, (size_t)k * V + v) + acc;
            tr[v] = ld(tgt, M->dtype, (size_t)k * V + v);
        }
        const double w = exp(-(double)k / gam);                    /* w_k = exp(-(k-1)/gamma), k from 1 */
        L += w * position_loss(ell, tr, V, ystar[k], a_ce, a_l1, mult * w, g ? dl : NULL, p, q);
        if (!g) continue;
        for (int v = 0; v < V; ++v)
            for (int d = 0; d < r; ++d) {
                g->W_r[(size_t)v * r + d] += dl[v] * zop[(size_t)k * r + d];
                dz[(size_t)k * r + d] += dl[v] * ld(M->W_r, M->dtype, (size_t)v * r + d);
            }
    }
    if (g) {
        /* Trans backward (Eq. mlp) */
        for (int k = 0; k < B; ++k) {
            for (int o = 0; o < R2; ++o) {
                double acc = 0.0;
                for (int d = 0; d < r; ++d) {
                    acc += ld(M->W2, M->dtype, (size_t)d * R2 + o) * dz[(size_t)k * r + d];
                    g->W2[(size_t)d * R2 + o] += dz[(size_t)k * r + d] * uop[(size_t)k * R2 + o];
                }
                du[o] = acc;
                dt[o] = acc * sigma_prime(M->act, tp[(size_t)k * R2 + o]);
            }
            for (int d = 0; d < r; ++d) {
                double acc = dz[(size_t)k * r + d];
                for (int o = 0; o < R2; ++o) {
                    acc += ld(M->W1, M->dtype, (size_t)o * r + d) * dt[o];
                    g->W1[(size_t)o * r + d] += dt[o] * cop[(size_t)k * r + d];
                }
                dc[(size_t)k * r + d] = acc;
            }
        }
        /* Mix backward (Eq. mix) */
        for (int j = 0; j < B; ++j)
            for (int d = 0; d < r; ++d) {
                double acc = dc[(size_t)j * r + d];
                for (int k = j + 1; k < B; ++k) {
                    acc += ld(M->L, M->dtype, ((size_t)d * B + k) * B + j) * dc[(size_t)k * r + d];
                    g->L[((size_t)d * B + k) * B + j] += dc[(size_t)k * r + d] * a[(size_t)j * r + d];
                }
                da[(size_t)j * r + d] = acc;
            }
        /* Fuse backward (Eq. fuse) */
        for (int k = 0; k < B; ++k)
            for (int e = 0; e < r; ++e) {
                double duh = 0.0, dug_k = 0.0, de = 0.0;
                const double xe = ld(M->W_e, M->dtype, (size_t)x[k] * r + e);
                for (int d = 0; d < r; ++d) {
                    const double dad = da[(size_t)k * r + d];
                    duh += ld(M->W_in, M->dtype, (size_t)d * 3 * r + e) * dad;
                    dug_k += ld(M->W_in, M->dtype, (size_t)d * 3 * r + r + e) * dad;
                    de += ld(M->W_in, M->dtype, (size_t)d * 3 * r + 2 * r + e) * dad;
                    g->W_in[(size_t)d * 3 * r + e] += dad * uh[(size_t)k * r + e];
                    g->W_in[(size_t)d * 3 * r + r + e] += dad * ug[e];
                    g->W_in[(size_t)d * 3 * r + 2 * r + e] += dad * xe;
                }
                dug[e] += dug_k;
                g->W_e[(size_t)x[k] * r + e] += de;
                for (int i = 0; i < H; ++i) g->W_h[(size_t)e * H + i] += duh * ld(h, M->dtype, (size_t)k * H + i);
            }
        for (int e = 0; e < r; ++e)
            for (int i = 0; i < H; ++i) g->W_g[(size_t)e * H + i] += dug[e] * gm[i];
    }
    free(uh); free(ug); free(gm); free(a); free(c); free(cop); free(tp); free(uop); free(z); free(zop);
    free(ell); free(tr); free(dl); free(p); free(q); free(dz); free(dc); free(da); free(du); free(dt); free(dug);
    return L;
}

/* One training step of Sec. 4.3 on one block, T = 1:
 *   L_total = L(p^r) + lambda L(p^b) + beta L(p^r-hat)
 * with L(p) = sum_k w_k [a_ce (-log p_k(x*_k)) + a_l1 |p_k - p^t_k|_1],
 * w_k = exp(-(k-1)/gamma), p^t_k = softmax(target_k):
 *   p^r      the refiner under teacher forcing (inputs x*_{k-1}, x*_0 = anchor);
 *   p^b      the drafter's base distribution softmax(s_k) (no refiner weight);
 *   p^r-hat  the refiner fed the drafter's argmax(s) tokens (consistency).
 * loss[4] = L(p^r), L(p^b), L(p^r-hat), L_total.  With g given, dL_total /
 * dtheta of every refiner weight is added into g. */
int xo_train_step(const xo_model *M, const void *h, const void *s, const void *tgt, const int32_t *ystar,
                  int32_t anchor, double a_ce, double a_l1, double gam, double lambda, double beta, double *loss,
                  double *gW_e, double *gW_h, double *gW_g, double *gW_in, double *gL, double *gW1, double *gW2,
                  double *gW_r)
{
    const int B = M->B, V = M->V;
    if (anchor < 0 || anchor >= V || gam <= 0.0) return -1;
    for (int k = 0; k < B; ++k)
        if (ystar[k] < 0 || ystar[k] >= V) return -1;
    xo_grads gg = {gW_e, gW_h, gW_g, gW_in, gL, gW1, gW2, gW_r};
    xo_grads *g = gW_r ? &gg : NULL;
    int32_t *x = malloc(sizeof(int32_t) * B);
    double *row = malloc(sizeof(double) * V), *tr = malloc(sizeof(double) * V);
    double *p = malloc(sizeof(double) * V), *q = malloc(sizeof(double) * V);
    x[0] = anchor;
    for (int k = 1; k < B; ++k) x[k] = ystar[k - 1];
    const double Lr = refiner_loss(M, h, s, tgt, x, ystar, a_ce, a_l1, gam, 1.0, g);
    double Lb = 0.0;
    for (int k = 0; k < B; ++k) {
        for (int v = 0; v < V; ++v) {
            row[v] = ld(s, M->dtype, (size_t)k * V + v);
            tr[v] = ld(tgt, M->dtype, (size_t)k * V + v);
        }
        Lb += exp(-(double)k / gam) * position_loss(row, tr, V, ystar[k], a_ce, a_l1, 0.0, NULL, p, q);
        if (k + 1 < B) x[k + 1] = argmax_f32(row, V, NULL);   /* the drafter's argmax(s) token */
    }
    const double Lc = refiner_loss(M, h, s, tgt, x, ystar, a_ce, a_l1, gam, beta, g);
    loss[0] = Lr;
    loss[1] = Lb;
    loss[2] = Lc;
    loss[3] = Lr + lambda * Lb + beta * Lc;
    free(x); free(row); free(tr); free(p); free(q);
    return 0;
}
/* ----------------------------------------------------- batched test helpers */

/* Refine the same block under n different seeds (statistical pins). */
int xo_jacobi_seeds(const xo_model *M, const void *h, const void *s, int32_t anchor,
                    const int32_t *draft, double T, const uint64_t *seeds, int n, uint32_t offset,
                    int K_max, int32_t *tokens, int32_t *iters)
{
    const int B = M->B, r = M->r;
    double *lse = (double *)malloc(sizeof(double) * B);
    double *sel = (double *)malloc(sizeof(double) * B);
    double *z = (double *)malloc(sizeof(double) * (size_t)B * r);
    for (int i = 0; i < n; ++i) {
        int32_t conv;
        int rc = xo_jacobi(M, h, s, anchor, draft, T, seeds[i], offset, K_max, 0, tokens + (size_t)i * B,
                           iters + i, &conv, lse, sel, z, NULL, NULL, NULL);
        if (rc) { free(lse); free(sel); free(z); return rc; }
    }
    free(lse); free(sel); free(z);
    return 0;
}

/* Refine (from the given Y^(0), or argmax s when draft is NULL) and then
 * accept, once per seed; only the refinement / acceptance seed varies. */
int xo_refine_accept_seeds(const xo_model *M, const void *h, const void *s, const void *tgt,
                           int32_t anchor, const int32_t *draft, double T, const uint64_t *seeds,
                           int n, uint32_t offset, int K_max, int32_t *accept_len, int32_t *out)
{
    const int B = M->B, r = M->r;
    int32_t *tok = (int32_t *)malloc(sizeof(int32_t) * B);
    double *lse = (double *)malloc(sizeof(double) * B);
    double *sel = (double *)malloc(sizeof(double) * B);
    double *z = (double *)malloc(sizeof(double) * (size_t)B * r);
    for (int i = 0; i < n; ++i) {
        int32_t it, conv;
        int rc = xo_jacobi(M, h, s, anchor, draft, T, seeds[i], offset, K_max, 0, tok, &it, &conv, lse,
                           sel, z, NULL, NULL, NULL);
        if (!rc)
            rc = xo_accept(M, tgt, s, tok, lse, sel, z, T, seeds[i], offset, accept_len + i,
                           out + (size_t)i * (B + 1), NULL, NULL);
        if (rc) { free(tok); free(lse); free(sel); free(z); return rc; }
    }
    free(tok); free(lse); free(sel); free(z);
    return 0;
}
