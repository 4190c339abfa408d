// refine_kernels.cu -- the CUDA-core kernels of the refinement pass.
//
//   k_init           per-call state (Algorithm 1: Y^(0) = draft; all positions live)
//   k_rowmax         Y^(0) = argmax_v s_k,v when no draft is given (Algorithm 1)
//   k_pre_gemm       h [W_h; W_g]^T (split-K)
//   k_build_ep       at refiner creation, the folded embedding
//                    E' = W_e W_in[:, 2r:3r]^T (Sec. 4.1, "Low overhead")
//   k_pre_mix        token-independent part of Fuse + Mix, hoisted out of the
//                    loop because h and g are fixed across iterations (Sec. 4.2):
//                    P_k = W_in[:, 0:r] W_h h_k + W_in[:, r:2r] W_g g,
//                    Pc = (I + L) P per channel (Eq. mix)
//   k_mix_mlp        per pass: gather E'[x_{k-1}], Mix (Eq. mix), Trans (Eq. mlp);
//                    one 8-CTA cluster per block exchanging c and sigma(W_1 c)
//                    through distributed shared memory
//   k_read_simt      Read + Correct + selection on CUDA cores (fp32 refiners)
//   k_reduce         combine the split-vocabulary partials, finish the T > 0
//                    draw inside the winning group, apply Algorithm 1's stopping
//                    rule per block, and set the device-side loop condition
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

namespace xp {

// ----------------------------------------------------------------- k_init

// The loop condition defaults to 0 at every launch of the graph and only
// this kernel opens it, so a condition that never reached the device runs
// no pass at all instead of looping.
__global__ void k_init(Params pin, Params *pdev, cudaGraphConditionalHandle handle)
{
    const Params &p = pin;
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t == 0) {
        *pdev = pin;
        p.ctl[CTL_NACT] = p.N;
        p.ctl[CTL_DONE] = 0;
        p.ctl[CTL_PASS] = 0;
        cudaGraphSetConditional(handle, 1u);
    }
    if (t < p.N) {
        p.act_tok[t] = t;
        if (p.draft) {
            int y = p.draft[t];
            if (y < 0 || y >= p.V) { set_status(p.status, ST_BOUNDS); y = 0; }
            p.tokens[t] = y;
        }
    }
    if (t < p.b) {
        SeqState s{};
        s.active = 1; s.m = -1; s.iters = 0; s.converged = 0; s.off = t * p.B; s.cnt = p.B;
        p.st[t] = s;
        if (p.anchor[t] < 0 || p.anchor[t] >= p.V) set_status(p.status, ST_BOUNDS);
        if (p.iters) p.iters[t] = 0;
        if (p.converged) p.converged[t] = 0;
    }
}

// --------------------------------------------------------------- k_rowmax

// One CTA per row: first index of the maximum of s[row, :] (fp32 compare).
__global__ void __launch_bounds__(256) k_rowmax(const Params *__restrict__ pp)
{
    const Params &p = *pp;
    const int row = blockIdx.x;
    float best = -INFINITY;
    int idx = 0x7fffffff;
    for (int v = threadIdx.x; v < p.V; v += blockDim.x) {
        const float x = ld_any(p.s, p.dtype, (size_t)row * p.V + v);
        if (x > best) { best = x; idx = v; }
    }
    __shared__ float sb[256];
    __shared__ int si[256];
    sb[threadIdx.x] = best;
    si[threadIdx.x] = idx;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (threadIdx.x < w) {
            float ob = sb[threadIdx.x + w];
            int oi = si[threadIdx.x + w];
            float b0 = sb[threadIdx.x];
            int i0 = si[threadIdx.x];
            merge_argmax(b0, i0, ob, oi);
            sb[threadIdx.x] = b0;
            si[threadIdx.x] = i0;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) p.tokens[row] = si[0];
}

// ---------------------------------------------------------------- GEMM NT

// C[m][n] = sum_{k in [kb, ke)} A[m][k] * B[n][k] for the 64x64 tile at
// (m0, n0); A, B row-major with leading dimensions lda, ldb, C with ldc.
// 16-deep K steps, 4x4 outputs per thread, 256 threads.
template <typename TA, typename TB>
__device__ __forceinline__ void gemm_nt_tile(const TA *__restrict__ A, int lda, const TB *__restrict__ Bm, int ldb,
                                             float *__restrict__ C, int ldc, int M, int N, int kb, int ke, int m0,
                                             int n0)
{
    __shared__ float As[16][64 + 4];
    __shared__ float Bs[16][64 + 4];
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
    float acc[4][4] = {};
    for (int k0 = kb; k0 < ke; k0 += 16) {
        for (int i = threadIdx.x; i < 64 * 16; i += 256) {
            const int r = i / 16, c = i % 16;
            const int kk = k0 + c;
            As[c][r] = (m0 + r < M && kk < ke) ? ldf(A, (size_t)(m0 + r) * lda + kk) : 0.0f;
            Bs[c][r] = (n0 + r < N && kk < ke) ? ldf(Bm, (size_t)(n0 + r) * ldb + kk) : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) { a[i] = As[c][ty * 4 + i]; b[i] = Bs[c][tx * 4 + i]; }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int m = m0 + ty * 4 + i, n = n0 + tx * 4 + j;
            if (m < M && n < N) C[(size_t)m * ldc + n] = acc[i][j];
        }
}

// Upart[z][t][which * r + o] = sum over K-slice z of h[t][:] . W[o][:],
// W = W_h (which = 0) or W_g (which = 1).  grid (r / 64, ceil(N / 64), ksplit).
__global__ void __launch_bounds__(256) k_pre_gemm(const Params *__restrict__ pp, int which, int kchunk)
{
    const Params &p = *pp;
    const int kb = blockIdx.z * kchunk, ke = min(p.H, kb + kchunk);
    float *C = p.Upart + (size_t)blockIdx.z * p.N * 2 * RANK + which * RANK;
    const void *W = which ? p.W_g : p.W_h;
    if (p.dtype)
        gemm_nt_tile(static_cast<const uint16_t *>(p.h), p.H, static_cast<const uint16_t *>(W), p.H, C, 2 * RANK,
                     p.N, RANK, kb, ke, blockIdx.y * 64, blockIdx.x * 64);
    else
        gemm_nt_tile(static_cast<const float *>(p.h), p.H, static_cast<const float *>(W), p.H, C, 2 * RANK, p.N,
                     RANK, kb, ke, blockIdx.y * 64, blockIdx.x * 64);
}

// Folded embedding E'[v][d] = sum_e W_in[d][2r + e] W_e[v][e] (Sec. 4.1: Fuse
// is linear, so the token slot folds into one table).  grid (r/64, ceil(V/64)).
__global__ void __launch_bounds__(256) k_build_ep(const void *W_e, const void *W_in, float *Ep, int V, int dtype)
{
    if (dtype)
        gemm_nt_tile(static_cast<const uint16_t *>(W_e), RANK, static_cast<const uint16_t *>(W_in) + 2 * RANK,
                     3 * RANK, Ep, RANK, V, RANK, 0, RANK, blockIdx.y * 64, blockIdx.x * 64);
    else
        gemm_nt_tile(static_cast<const float *>(W_e), RANK, static_cast<const float *>(W_in) + 2 * RANK, 3 * RANK,
                     Ep, RANK, V, RANK, 0, RANK, blockIdx.y * 64, blockIdx.x * 64);
}

// -------------------------------------------------------------- k_pre_mix

// grid (b, RANK / 32): block s, channels [32 y, 32 y + 32).
__global__ void __launch_bounds__(256) k_pre_mix(const Params *__restrict__ pp)
{
    const Params &p = *pp;
    extern __shared__ float sm[];
    const int B = p.B, s = blockIdx.x, d0 = blockIdx.y * 32;
    float *U = sm;                     // [B][2r]   W_h h_k | W_g h_k
    float *ug = U + B * 2 * RANK;      // [r]       W_g g
    float *P = ug + RANK;              // [B][32]   P for this channel slice
    const size_t tok0 = (size_t)s * B;
    for (int i = threadIdx.x; i < B * 2 * RANK; i += blockDim.x) {
        const int k = i / (2 * RANK), o = i % (2 * RANK);
        float acc = 0.0f;
        for (int z = 0; z < p.ksplit; ++z) acc += p.Upart[((size_t)z * p.N + tok0 + k) * 2 * RANK + o];
        U[i] = acc;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < RANK; e += blockDim.x) {
        float acc = 0.0f;
        for (int k = 0; k < B; ++k) acc += U[k * 2 * RANK + RANK + e];
        ug[e] = acc / (float)B;
    }
    __syncthreads();
    // P[k][d] = sum_e W_in[d][e] u_h,k[e] + sum_e W_in[d][r + e] u_g[e]
    for (int i = threadIdx.x; i < B * 32; i += blockDim.x) {
        const int k = i / 32, dd = i % 32, d = d0 + dd;
        float acc = 0.0f;
        const size_t wrow = (size_t)d * 3 * RANK;
        for (int e = 0; e < RANK; ++e) acc = fmaf(ld_any(p.W_in, p.dtype, wrow + e), U[k * 2 * RANK + e], acc);
        for (int e = 0; e < RANK; ++e) acc = fmaf(ld_any(p.W_in, p.dtype, wrow + RANK + e), ug[e], acc);
        P[k * 32 + dd] = acc;
    }
    __syncthreads();
    // Pc = (I + L) P, channel by channel (Eq. mix)
    for (int i = threadIdx.x; i < B * 32; i += blockDim.x) {
        const int k = i / 32, dd = i % 32, d = d0 + dd;
        float acc = P[k * 32 + dd];
        for (int j = 0; j < k; ++j) acc = fmaf(ld_any(p.L, p.dtype, ((size_t)d * B + k) * B + j), P[j * 32 + dd], acc);
        p.Pc[(tok0 + k) * RANK + d] = acc;
    }
}

// -------------------------------------------------------------- k_mix_mlp

constexpr int MLP_CLUSTER = 8;

// grid (8, b), cluster (8, 1, 1), 256 threads.  CTA `rank` of block s owns
// channels [32 rank, +32) of c and z, and rows [64 rank, +64) of W_1.
__global__ void __cluster_dims__(MLP_CLUSTER, 1, 1) __launch_bounds__(256) k_mix_mlp(const Params *__restrict__ pp)
{
    const Params &p = *pp;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int s = blockIdx.y, B = p.B;
    const SeqState st = p.st[s];
    if (!st.active) return;            // uniform over the cluster
    const int m = st.m, cnt = B - 1 - m, off = st.off;
    const int d0 = rank * 32;

    __shared__ float e[MAX_B][32];      // gathered E' rows, own channel slice
    __shared__ float cown[MAX_B][32];   // c, own channel slice (unrounded)
    __shared__ float uown[MAX_B][64];   // sigma(W_1 c), own rows, operand-rounded
    extern __shared__ float dyn[];
    float *cop = dyn;                   // [cnt][RANK]    all of c, operand-rounded
    float *uop = dyn + MAX_B * RANK;    // [cnt][2 RANK]  all of sigma(W_1 c)

    // Fuse (token part) + Mix for the own channel slice
    for (int i = threadIdx.x; i < B * 32; i += blockDim.x) {
        const int j = i / 32, dd = i % 32;
        int x = j == 0 ? p.anchor[s] : p.tokens[(size_t)s * B + j - 1];
        if (x < 0 || x >= p.V) x = 0;   // reported by k_init
        e[j][dd] = p.Ep[(size_t)x * RANK + d0 + dd];
    }
    __syncthreads();
    for (int i = threadIdx.x; i < cnt * 32; i += blockDim.x) {
        const int t = i / 32, dd = i % 32, k = m + 1 + t, d = d0 + dd;
        float acc = p.Pc[((size_t)s * B + k) * RANK + d] + e[k][dd];
        for (int j = 0; j < k; ++j) acc = fmaf(ld_any(p.L, p.dtype, ((size_t)d * B + k) * B + j), e[j][dd], acc);
        cown[t][dd] = acc;
    }
    cluster.sync();
    for (int i = threadIdx.x; i < cnt * RANK; i += blockDim.x) {
        const int t = i / RANK, d = i % RANK;
        const float *peer = cluster.map_shared_rank(&cown[0][0], d / 32);
        cop[t * RANK + d] = round_op(peer[t * 32 + (d % 32)], p.dtype);
    }
    __syncthreads();
    // t = W_1 c for rows [64 rank, +64): thread (row, token group of 4)
    {
        const int row = threadIdx.x % 64, tg = threadIdx.x / 64, o = rank * 64 + row;
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.0f;
        for (int d = 0; d < RANK; ++d) {
            const float w = ld_any(p.W1, p.dtype, (size_t)o * RANK + d);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int t = tg + 4 * q;
                if (t < cnt) acc[q] = fmaf(w, cop[t * RANK + d], acc[q]);
            }
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int t = tg + 4 * q;
            if (t < cnt) uown[t][row] = round_op(act_fn(p.act, acc[q]), p.dtype);
        }
    }
    cluster.sync();
    for (int i = threadIdx.x; i < cnt * 2 * RANK; i += blockDim.x) {
        const int t = i / (2 * RANK), f = i % (2 * RANK);
        const float *peer = cluster.map_shared_rank(&uown[0][0], f / 64);
        uop[t * 2 * RANK + f] = peer[t * 64 + (f % 64)];
    }
    __syncthreads();
    // z = c + W_2 u for channels [32 rank, +32): thread (row, token group of 8)
    {
        const int row = threadIdx.x % 32, tg = threadIdx.x / 32, d = d0 + row;
        float acc[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[q] = 0.0f;
        for (int f = 0; f < 2 * RANK; ++f) {
            const float w = ld_any(p.W2, p.dtype, (size_t)d * 2 * RANK + f);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int t = tg + 8 * q;
                if (t < cnt) acc[q] = fmaf(w, uop[t * 2 * RANK + f], acc[q]);
            }
        }
        float *zf = p.z_final ? p.z_final : p.zbuf;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int t = tg + 8 * q;
            if (t < cnt) {
                const int k = m + 1 + t;
                const float z = cown[t][row] + acc[q];
                zf[((size_t)s * B + k) * RANK + d] = z;
                const size_t zi = (size_t)(off + t) * RANK + d;
                if (p.dtype) static_cast<uint16_t *>(p.zpack)[zi] = f2bf(z);
                else static_cast<float *>(p.zpack)[zi] = z;
            }
        }
    }
    cluster.sync();                     // peers may still read our shared memory
}

// ------------------------------------------------------------ k_read_simt

// Read + Correct + selection on CUDA cores.  grid = S vocabulary ranges,
// 256 threads; tokens in tiles of 32.  Lane = vocabulary id while computing
// l = s + W_r z, then lane = token while folding a 32-id group into its state.
__global__ void __launch_bounds__(256) k_read_simt(const Params *__restrict__ pp)
{
    const Params &p = *pp;
    const int n = p.ctl[CTL_NACT];
    if (n == 0) return;
    const int G = (p.V + GROUP - 1) / GROUP;
    const int g0 = (int)((long long)G * blockIdx.x / gridDim.x);
    const int g1 = (int)((long long)G * (blockIdx.x + 1) / gridDim.x);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    extern __shared__ float simt_dyn[];
    float (*zs)[RANK + 1] = reinterpret_cast<float (*)[RANK + 1]>(simt_dyn);               // [32][r + 1]
    float (*ls)[32][33] = reinterpret_cast<float (*)[32][33]>(simt_dyn + 32 * (RANK + 1));  // [8][32][33]
    __shared__ SelState sst[8][32];
    for (int t0 = 0; t0 < n; t0 += 32) {
        const int nt = min(32, n - t0);
        for (int i = threadIdx.x; i < 32 * RANK; i += blockDim.x) {
            const int t = i / RANK, d = i % RANK;
            zs[t][d] = t < nt ? ld_any(p.zpack, p.dtype, (size_t)(t0 + t) * RANK + d) : 0.0f;
        }
        __syncthreads();
        // the token this lane stands for in the selection step
        const int ti = t0 + lane;
        int tok = 0, pos = 0, seq = 0;
        float invT = 0.0f;
        if (lane < nt) {
            tok = p.act_tok[ti];
            seq = tok / p.B;
            pos = tok % p.B;
            const float T = p.temperature[seq];
            invT = T > 0.0f ? 1.0f / T : 0.0f;
        }
        const unsigned long long seed = lane < nt ? p.seed[seq] : 0ull;
        SelState sel;
        sel.init();
        for (int g = g0 + warp; g < g1; g += 8) {
            const int v = g * GROUP + lane;
            float acc[32];
#pragma unroll
            for (int t = 0; t < 32; ++t) acc[t] = 0.0f;
            if (v < p.V) {
                for (int d = 0; d < RANK; ++d) {
                    const float w = ld_any(p.W_r, p.dtype, (size_t)v * RANK + d);
#pragma unroll
                    for (int t = 0; t < 32; ++t) acc[t] = fmaf(w, zs[t][d], acc[t]);
                }
            }
#pragma unroll
            for (int t = 0; t < 32; ++t) {
                float l = -INFINITY;
                if (t < nt && v < p.V) {
                    const int tk = p.act_tok[t0 + t];
                    l = acc[t] + ld_any(p.s, p.dtype, (size_t)tk * p.V + v);
                    if (p.logits) p.logits[(size_t)tk * p.V + v] = l;
                }
                ls[warp][t][lane] = l;
            }
            __syncwarp();
            if (lane < nt) {
                float row[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) row[j] = ls[warp][lane][j];
                select_group(sel, row, g * GROUP, min(GROUP, p.V - g * GROUP), invT, seed, pos, p.offset);
            }
            __syncwarp();
        }
        sst[warp][lane] = sel;
        __syncthreads();
        if (warp == 0 && lane < nt) {
            const bool sampling = invT > 0.0f;
            Partial a{sst[0][lane].best, sst[0][lane].idx, sst[0][lane].m, sst[0][lane].s};
            for (int w = 1; w < 8; ++w) {
                const Partial b{sst[w][lane].best, sst[w][lane].idx, sst[w][lane].m, sst[w][lane].s};
                merge_partial(a, b, sampling);
            }
            p.part[(size_t)blockIdx.x * p.N + t0 + lane] = a;
        }
        __syncthreads();
    }
}

// --------------------------------------------------------------- k_reduce

// grid b, 1024 threads (warp k = block position k).  After every block has
// been reduced, the last CTA to finish packs the positions of the next pass
// and sets the WHILE condition of the graph.
__global__ void __launch_bounds__(1024) k_reduce(const Params *__restrict__ pp, cudaGraphConditionalHandle handle)
{
    const Params &p = *pp;
    const int s = blockIdx.x, B = p.B, warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const SeqState st = p.st[s];
    __shared__ int last;
    __shared__ int ynew[MAX_B];
    const float T = p.temperature[s];
    const float invT = T > 0.0f ? 1.0f / T : 0.0f;
    const bool sampling = invT > 0.0f;
    if (st.active && warp < B && warp > st.m) {
        const int k = warp, i = st.off + (k - st.m - 1), tok = s * B + k;
        Partial a{-INFINITY, 0x7fffffff, -INFINITY, 0.0f};
        for (int r = lane; r < p.S; r += 32) merge_partial(a, p.part[(size_t)r * p.N + i], sampling);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            Partial b;
            b.best = __shfl_xor_sync(0xffffffffu, a.best, o);
            b.idx = __shfl_xor_sync(0xffffffffu, a.idx, o);
            b.m = __shfl_xor_sync(0xffffffffu, a.m, o);
            b.s = __shfl_xor_sync(0xffffffffu, a.s, o);
            merge_partial(a, b, sampling);
        }
        int y;
        float sel, lse;
        if (!sampling) {
            y = a.idx;
            sel = a.best;
            lse = __int_as_float(0x7fc00000);
        } else {
            // second stage: Gumbel-max over the members of the drawn group
            const int v = a.idx * GROUP + lane;
            float x = -INFINITY, score = -INFINITY;
            if (v < p.V) {
                float acc = 0.0f;
                for (int d = 0; d < RANK; ++d)
                    acc = fmaf(ld_any(p.W_r, p.dtype, (size_t)v * RANK + d),
                               ld_any(p.zpack, p.dtype, (size_t)i * RANK + d), acc);
                x = (acc + ld_any(p.s, p.dtype, (size_t)tok * p.V + v)) * invT;
                score = x + gumbel(p.seed[s], (uint32_t)v, (uint32_t)k, STREAM_ELEM, p.offset);
            }
            float bs = score;
            int bi = v;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float os = __shfl_xor_sync(0xffffffffu, bs, o);
                const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
                merge_argmax(bs, bi, os, oi);
            }
            y = bi;
            sel = __shfl_sync(0xffffffffu, x, (bi - a.idx * GROUP) & (GROUP - 1));
            lse = a.m + logf(a.s);
        }
        if (lane == 0) {
            ynew[k] = y;
            if (p.lse) p.lse[tok] = lse;
            if (p.logit_sel) p.logit_sel[tok] = sel;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        if (st.active) {
            int first = -1;
            for (int k = st.m + 1; k < B; ++k) {
                const int old = p.tokens[(size_t)s * B + k];
                if (ynew[k] != old && first < 0) first = k;
                p.tokens[(size_t)s * B + k] = ynew[k];
            }
            SeqState ns = st;
            ns.iters = st.iters + 1;
            ns.converged = first < 0;
            if (p.fixed_K) {
                ns.active = ns.iters < p.K_max;
                ns.m = -1;
            } else if (first < 0 || ns.iters >= p.K_max) {
                ns.active = 0;
            } else if (first == B - 1) {
                // the next pass would evaluate no position and change nothing:
                // it is Algorithm 1's final, unchanged pass
                ns.iters += 1;
                ns.converged = 1;
                ns.active = 0;
            } else {
                ns.active = 1;
                ns.m = first;
            }
            p.st[s] = ns;
            if (p.iters) p.iters[s] = ns.iters;
            if (p.converged) p.converged[s] = ns.converged;
        }
        __threadfence();
        last = atomicAdd(&p.ctl[CTL_DONE], 1) == p.b - 1;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    __shared__ int total;
    // pack the positions of the next pass (b <= 1024 blocks per call)
    if (threadIdx.x == 0) {
        int acc = 0;
        for (int q = 0; q < p.b; ++q) {
            SeqState ns;
            const volatile int *src = reinterpret_cast<const volatile int *>(&p.st[q]);
            ns.active = src[0]; ns.m = src[1]; ns.iters = src[2]; ns.converged = src[3];
            ns.pad0 = ns.pad1 = 0;
            if (ns.active) {
                ns.off = acc;
                ns.cnt = B - 1 - ns.m;
                acc += ns.cnt;
            } else {
                ns.cnt = 0;
            }
            p.st[q] = ns;
        }
        total = acc;
    }
    __syncthreads();
    for (int q = warp; q < p.b; q += 32) {
        const SeqState ns = p.st[q];
        if (ns.active)
            for (int t = lane; t < ns.cnt; t += 32) p.act_tok[ns.off + t] = q * B + ns.m + 1 + t;
    }
    if (threadIdx.x == 0) {
        const int passes = p.ctl[CTL_PASS] + 1;
        p.ctl[CTL_NACT] = total;
        p.ctl[CTL_DONE] = 0;
        p.ctl[CTL_PASS] = passes;
        // no block can take part in more than K_max passes; the cap also bounds
        // the loop should the per-block bookkeeping ever disagree
        cudaGraphSetConditional(handle, (total > 0 && passes < p.K_max) ? 1u : 0u);
    }
}

// Profiling hook: the next Read pass evaluates tokens 0..n-1.
__global__ void k_prof_prepare(int32_t *ctl, int32_t *act_tok, int n)
{
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t < n) act_tok[t] = t;
    if (t == 0) ctl[CTL_NACT] = n;
}

}  // namespace xp
