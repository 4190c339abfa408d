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
#include "mlp_common.cuh"
#include "reduce_common.cuh"

namespace cg = cooperative_groups;

namespace xp {

// ----------------------------------------------------------------- k_init

// The loop condition defaults to 0 at every launch of the graph and only
// this kernel opens it, so a condition that never reached the device runs
// no pass at all instead of looping.
__global__ void k_init(Params pin, Params *pdev, cudaGraphConditionalHandle handle)
{
    const Params &p = pin;
    const unsigned long long t_start = globaltimer_ns();
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    const int n0 = p.sequential ? p.b : p.N;   // tokens of the first pass: all positions, or position 0
    if (t == 0) {
        *pdev = pin;
        p.ctl[CTL_NACT] = n0;
        p.ctl[CTL_DONE] = 0;
        p.ctl[CTL_PASS] = 0;
        p.ctl[CTL_EVAL] = n0;
        if (p.use_graph) cudaGraphSetConditional(handle, 1u);
    }
    if (t < n0) p.act_tok[t] = p.sequential ? t * p.B : t;
    if (t < p.N) {
        if (p.draft) {
            int y = p.draft[t];
            if (y < 0 || y >= p.V) { set_status(p.status, ST_BOUNDS); y = 0; }
            p.tokens[t] = y;
        }
    }
    if (t < p.b) {
        SeqState s{};
        s.active = 1; s.m = -1; s.iters = 0; s.converged = 0;
        s.off = p.sequential ? t : t * p.B; s.cnt = p.sequential ? 1 : p.B;
        p.st[t] = s;
        if (p.anchor[t] < 0 || p.anchor[t] >= p.V) set_status(p.status, ST_BOUNDS);
        if (p.iters) p.iters[t] = 0;
        if (p.converged) p.converged[t] = 0;
    }
    if (threadIdx.x == 0) trace_mark(p.trace, 0, t_start);
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

// bf16, at most 32 tokens: Upart[z][t][o] = h[t][K-slice z] . [W_h; W_g][o][K-slice z].
// grid (2r / 8, KS), 256 threads: warp w owns output row o = 8 x + w; the
// CTA stages its K-slice of every token's h in shared memory ([N][kslice]).
__global__ void __launch_bounds__(256) k_pre_gemv(const Params *__restrict__ pp, int kslice)
{
    const unsigned long long t_start = globaltimer_ns();
    const Params &p = *pp;
    extern __shared__ __align__(16) uint16_t hs[];
    const int N = p.N, H = p.H, warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int kb = blockIdx.y * kslice, ke = min(H, kb + kslice), kl = ke - kb;
    const uint16_t *h = static_cast<const uint16_t *>(p.h);
    // this warp's weight row: 16-byte pieces k0 = 8 lane + 256 q of the K-slice,
    // the next piece requested while the current one is used
    const int o = blockIdx.x * 8 + warp;
    const uint16_t *W = static_cast<const uint16_t *>(o < RANK ? p.W_h : p.W_g) + (size_t)(o % RANK) * H + kb;
    uint4 wcur = make_uint4(0, 0, 0, 0), wnext = make_uint4(0, 0, 0, 0);
    if (8 * lane < kl) wcur = __ldg(reinterpret_cast<const uint4 *>(W + 8 * lane));
    if (8 * lane + 256 < kl) wnext = __ldg(reinterpret_cast<const uint4 *>(W + 8 * lane + 256));
    {
        // stage h[:, K-slice] in batches of 8 16-byte loads per thread
        const int per = kl / 8, total = N * per;
        for (int i0 = 0; i0 < total; i0 += 8 * 256) {
            uint4 hv[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int i = i0 + q * 256 + threadIdx.x;
                if (i < total)
                    hv[q] = __ldg(reinterpret_cast<const uint4 *>(h + (size_t)(i / per) * H + kb) + (i % per));
            }
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int i = i0 + q * 256 + threadIdx.x;
                if (i < total) reinterpret_cast<uint4 *>(hs + (size_t)(i / per) * kslice)[i % per] = hv[q];
            }
        }
    }
    __syncthreads();
    float v[32];
#pragma unroll
    for (int t = 0; t < 32; ++t) v[t] = 0.0f;
#pragma unroll 1
    for (int k0 = 8 * lane; k0 < kl; k0 += 256) {
        float w[8];
        bf16x8_to_f32(wcur, w);
        wcur = wnext;
        if (k0 + 512 < kl) wnext = __ldg(reinterpret_cast<const uint4 *>(W + k0 + 512));
#pragma unroll
        for (int t = 0; t < 32; ++t) {
            if (t < N) {
                float x[8];
                bf16x8_to_f32(*reinterpret_cast<const uint4 *>(hs + (size_t)t * kslice + k0), x);
#pragma unroll
                for (int j = 0; j < 8; ++j) v[t] = fmaf(w[j], x[j], v[t]);
            }
        }
    }
    const float sum = reduce_scatter32(v, lane);
    if (lane < N) p.Upart[((size_t)blockIdx.y * N + lane) * 2 * RANK + o] = sum;
    __syncthreads();
    if (threadIdx.x == 0) trace_mark(p.trace, 2, t_start);
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

// grid (b, RANK / 32): block s, channels [32 y, 32 y + 32).  Dynamic shared
// memory: U [B][2r], u_g [r], W_in rows [32][2r + 1], P [B][32].
__global__ void __launch_bounds__(256) k_pre_mix(const Params *__restrict__ pp)
{
    const unsigned long long t_start = globaltimer_ns();
    const Params &p = *pp;
    extern __shared__ float sm[];
    const int B = p.B, s = blockIdx.x, d0 = blockIdx.y * 32;
    const size_t tok0 = (size_t)s * B;
    float *P;                              // [B][32]   P for this channel slice
    if (p.pre_folded) {
        // the partials already are h F^T: P_k = F_h h_k + mean_j F_g h_j for
        // the 32 channels (the h slot at column d, the g slot at r + d)
        float *Uh = sm, *Ug = Uh + B * 32;
        P = Ug + B * 32;
        const int ks = p.ksplit, NN = p.N;
        for (int i = threadIdx.x; i < B * 64; i += blockDim.x) {
            const int k = i / 64, c = i % 64, slot = c / 32, dd = c % 32;
            const float *up = p.Upart + (tok0 + k) * 2 * RANK + slot * RANK + d0 + dd;
            float v = 0.0f;
            for (int z = 0; z < ks; ++z) v += __ldcg(up + (size_t)z * NN * 2 * RANK);
            (slot ? Ug : Uh)[k * 32 + dd] = v;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < B * 32; i += blockDim.x) {
            const int k = i / 32, dd = i % 32;
            float gs = 0.0f;
            for (int j = 0; j < B; ++j) gs += Ug[j * 32 + dd];
            P[k * 32 + dd] = Uh[k * 32 + dd] + gs / (float)B;
        }
        __syncthreads();
    } else {
        float *U = sm;                         // [B][2r]   W_h h_k | W_g h_k
        float *ug = U + B * 2 * RANK;          // [r]       W_g g
        float *Ws = ug + RANK;                 // [32][2r + 1]  W_in[d0 + dd][0:2r]
        P = Ws + 32 * (2 * RANK + 1);
        if (p.dtype) {
            constexpr int PER = 32 * 2 * RANK / 8 / 256;   // 8 16-byte pieces per thread
            uint4 wv[PER];
#pragma unroll
            for (int q = 0; q < PER; ++q) {
                const int i = threadIdx.x + 256 * q, dd = i / (2 * RANK / 8), c = i % (2 * RANK / 8);
                wv[q] = __ldg(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.W_in) +
                                                              (size_t)(d0 + dd) * 3 * RANK) + c);
            }
#pragma unroll
            for (int q = 0; q < PER; ++q) {
                const int i = threadIdx.x + 256 * q, dd = i / (2 * RANK / 8), c = i % (2 * RANK / 8);
                float x[8];
                bf16x8_to_f32(wv[q], x);
#pragma unroll
                for (int j = 0; j < 8; ++j) Ws[dd * (2 * RANK + 1) + 8 * c + j] = x[j];
            }
        } else {
            for (int i = threadIdx.x; i < 32 * 2 * RANK; i += blockDim.x) {
                const int dd = i / (2 * RANK), e = i % (2 * RANK);
                Ws[dd * (2 * RANK + 1) + e] = ld_any(p.W_in, p.dtype, (size_t)(d0 + dd) * 3 * RANK + e);
            }
        }
        {
            // U = sum of the K-slice partials; each thread issues its loads as one batch
            const int ks = p.ksplit, NN = p.N;
            const float *up = p.Upart + tok0 * 2 * RANK;
            for (int i0 = 0; i0 < B * 2 * RANK; i0 += 8 * 256) {
                float v[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const int i = i0 + q * 256 + threadIdx.x;
                    v[q] = i < B * 2 * RANK ? up[i] : 0.0f;
                }
                for (int z = 1; z < ks; ++z)
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const int i = i0 + q * 256 + threadIdx.x;
                        if (i < B * 2 * RANK) v[q] += up[(size_t)z * NN * 2 * RANK + i];
                    }
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const int i = i0 + q * 256 + threadIdx.x;
                    if (i < B * 2 * RANK) U[i] = v[q];
                }
            }
        }
        __syncthreads();
        for (int e = threadIdx.x; e < RANK; e += blockDim.x) {
            float acc = 0.0f;
            for (int k = 0; k < B; ++k) acc += U[k * 2 * RANK + RANK + e];
            ug[e] = acc / (float)B;
        }
        __syncthreads();
        // P[k][d] = sum_e W_in[d][e] u_h,k[e] + sum_e W_in[d][r + e] u_g[e]
        {
            const int dd = threadIdx.x % 32, kg = threadIdx.x / 32;
            const float *w = Ws + dd * (2 * RANK + 1);
            float gpart = 0.0f;
            for (int e = 0; e < RANK; ++e) gpart = fmaf(w[RANK + e], ug[e], gpart);
            for (int k = kg; k < B; k += 8) {
                float acc = gpart;
                const float *u = U + k * 2 * RANK;
                for (int e = 0; e < RANK; ++e) acc = fmaf(w[e], u[e], acc);
                P[k * 32 + dd] = acc;
            }
        }
        __syncthreads();
    }
    // Pc = (I + L) P, channel by channel (Eq. mix)
    for (int i = threadIdx.x; i < B * 32; i += blockDim.x) {
        const int k = i / 32, dd = i % 32, d = d0 + dd;
        float lrow[MAX_B];
        if (p.Lpk) {
            // packed L: a warp's 32 channels of one (k, j) are 64 contiguous bytes
            const uint16_t *lp = p.Lpk + (size_t)(k * (k - 1) / 2) * RANK + d;
#pragma unroll
            for (int j = 0; j < MAX_B; ++j) lrow[j] = j < k ? bf2f(lp[(size_t)j * RANK]) : 0.0f;
        } else {
            const size_t lb = ((size_t)d * B + k) * B;
#pragma unroll
            for (int j = 0; j < MAX_B; ++j) lrow[j] = j < k ? ld_any(p.L, p.dtype, lb + j) : 0.0f;
        }
        float acc = P[k * 32 + dd];
#pragma unroll
        for (int j = 0; j < MAX_B; ++j)
            if (j < k) acc = fmaf(lrow[j], P[j * 32 + dd], acc);
        p.Pc[(tok0 + k) * RANK + d] = acc;
    }
    __syncthreads();
    if (threadIdx.x == 0) trace_mark(p.trace, 3, t_start);
}

// -------------------------------------------------------------- k_mix_mlp

constexpr int MLP_CLUSTER = 8;
constexpr int W1S_LD = RANK + 2;        // padded row strides (in elements) so that
constexpr int W2S_LD = 2 * RANK + 2;    // 32 rows hit 32 different banks

// Trans for the cluster's tokens, one CTA's share:  u rows [64 rank, +64) of
// sigma(W_1 c) and z channels [32 rank, +32) of c + W_2 u.  The CTA's W_1 and
// W_2 rows are staged in shared memory (T = storage type of the weights).
// STAGE = false reads the rows straight from global memory (fp32 weights,
// which would not fit next to the activations).
template <typename T, bool STAGE>
__device__ __forceinline__ void mlp_share(const Params &p, cg::cluster_group &cluster, int rank, int cnt, int m,
                                          int s, int off, float (*cown)[32], float (*uown)[64], float *cop,
                                          float *uop, T *stage)
{
    const int B = p.B, d0 = rank * 32;
    const T *W1 = static_cast<const T *>(p.W1) + (size_t)rank * 64 * RANK;
    const T *W2 = static_cast<const T *>(p.W2) + (size_t)d0 * 2 * RANK;
    const T *w1s = W1, *w2s = W2;
    int ld1 = RANK, ld2 = 2 * RANK;
    if constexpr (STAGE) {
        // bf16 rows, 16-byte loads issued back to back; the padded smem rows are
        // written as 4-byte pairs
        T *s1 = stage, *s2 = stage + 64 * W1S_LD;
        constexpr int N1 = 64 * RANK / 8, N2 = 32 * 2 * RANK / 8;
        uint4 r1[N1 / 256], r2[N2 / 256];
#pragma unroll
        for (int q = 0; q < N1 / 256; ++q) r1[q] = __ldg(reinterpret_cast<const uint4 *>(W1) + threadIdx.x + 256 * q);
#pragma unroll
        for (int q = 0; q < N2 / 256; ++q) r2[q] = __ldg(reinterpret_cast<const uint4 *>(W2) + threadIdx.x + 256 * q);
#pragma unroll
        for (int q = 0; q < N1 / 256; ++q) {
            const int i = threadIdx.x + 256 * q, row = i / (RANK / 8), c = i % (RANK / 8);
            uint32_t *dst = reinterpret_cast<uint32_t *>(s1 + row * W1S_LD + 8 * c);
            dst[0] = r1[q].x; dst[1] = r1[q].y; dst[2] = r1[q].z; dst[3] = r1[q].w;
        }
#pragma unroll
        for (int q = 0; q < N2 / 256; ++q) {
            const int i = threadIdx.x + 256 * q, row = i / (2 * RANK / 8), c = i % (2 * RANK / 8);
            uint32_t *dst = reinterpret_cast<uint32_t *>(s2 + row * W2S_LD + 8 * c);
            dst[0] = r2[q].x; dst[1] = r2[q].y; dst[2] = r2[q].z; dst[3] = r2[q].w;
        }
        w1s = s1;
        w2s = s2;
        ld1 = W1S_LD;
        ld2 = W2S_LD;
    }
    // all of c from the 8 CTAs of the cluster (float4 loads of peer shared memory)
    for (int i = threadIdx.x; i < cnt * RANK / 4; i += blockDim.x) {
        const int t = i / (RANK / 4), d = 4 * (i % (RANK / 4));
        const float4 *peer = reinterpret_cast<const float4 *>(cluster.map_shared_rank(&cown[0][0], d / 32));
        const float4 c4 = peer[(t * 32 + (d % 32)) / 4];
        float *dst = cop + t * RANK + d;
        dst[0] = round_op(c4.x, p.dtype);
        dst[1] = round_op(c4.y, p.dtype);
        dst[2] = round_op(c4.z, p.dtype);
        dst[3] = round_op(c4.w, p.dtype);
    }
    __syncthreads();
    // t = W_1 c for rows [64 rank, +64): thread (row, token group of 4)
    {
        const int row = threadIdx.x % 64, tg = threadIdx.x / 64;
        const T *w = w1s + row * ld1;
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.0f;
        for (int d = 0; d < RANK; ++d) {
            const float wv = ldf(w, d);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int t = tg + 4 * q;
                if (t < cnt) acc[q] = fmaf(wv, cop[t * RANK + d], acc[q]);
            }
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int t = tg + 4 * q;
            if (t < cnt) uown[t][row] = round_op(act_fn(p.act, acc[q]), p.dtype);
        }
    }
    cluster.sync();
    for (int i = threadIdx.x; i < cnt * 2 * RANK / 4; i += blockDim.x) {
        const int t = i / (2 * RANK / 4), f = 4 * (i % (2 * RANK / 4));
        const float4 *peer = reinterpret_cast<const float4 *>(cluster.map_shared_rank(&uown[0][0], f / 64));
        reinterpret_cast<float4 *>(uop + t * 2 * RANK)[f / 4] = peer[(t * 64 + (f % 64)) / 4];
    }
    __syncthreads();
    // z = c + W_2 u for channels [32 rank, +32): thread (row, token group of 8)
    {
        const int row = threadIdx.x % 32, tg = threadIdx.x / 32, d = d0 + row;
        const T *w = w2s + row * ld2;
        float acc[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[q] = 0.0f;
        for (int f = 0; f < 2 * RANK; ++f) {
            const float wv = ldf(w, f);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int t = tg + 8 * q;
                if (t < cnt) acc[q] = fmaf(wv, uop[t * 2 * RANK + f], acc[q]);
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
}

__device__ __forceinline__ void mlp_share_mma(const Params &p, cg::cluster_group &cluster, int rank, int cnt, int m,
                                              int s, int off, float (*cown)[32], uint16_t *cop, uint16_t *uop,
                                              uint16_t *uown, const MlpFrags &fr)
{
    const int B = p.B, d0 = rank * 32, warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int g = lane >> 2, tq = lane & 3;      // fragment row group, thread in group
    const int khalf = warp >> 2;                 // W_2: K half of this warp
    // all of c from the cluster, rounded to bf16 (rows past cnt are zero)
    {
        constexpr int PER = 32 * RANK / 4 / 256;     // 8 float4 per thread
        float4 c4[PER];
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int i = threadIdx.x + 256 * q, t = i / (RANK / 4), d = 4 * (i % (RANK / 4));
            c4[q] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (t < cnt)
                c4[q] = reinterpret_cast<const float4 *>(cluster.map_shared_rank(&cown[0][0], d / 32))[
                    (t * 32 + (d % 32)) / 4];
        }
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int i = threadIdx.x + 256 * q, t = i / (RANK / 4), d = 4 * (i % (RANK / 4));
            uint32_t *dst = reinterpret_cast<uint32_t *>(cop + t * COP_LD + d);
            dst[0] = (uint32_t)f2bf(c4[q].x) | ((uint32_t)f2bf(c4[q].y) << 16);
            dst[1] = (uint32_t)f2bf(c4[q].z) | ((uint32_t)f2bf(c4[q].w) << 16);
        }
    }
    __syncthreads();
    // u = sigma(W_1 c): warp w -> 8 output rows, both token tiles
    for (int mt = 0; mt * 16 < cnt; ++mt) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        const uint16_t *arow0 = cop + (mt * 16 + g) * COP_LD, *arow1 = arow0 + 8 * COP_LD;
#pragma unroll
        for (int ks = 0; ks < RANK / 16; ++ks) {
            uint32_t a[4];
            a[0] = *reinterpret_cast<const uint32_t *>(arow0 + ks * 16 + 2 * tq);
            a[1] = *reinterpret_cast<const uint32_t *>(arow1 + ks * 16 + 2 * tq);
            a[2] = *reinterpret_cast<const uint32_t *>(arow0 + ks * 16 + 8 + 2 * tq);
            a[3] = *reinterpret_cast<const uint32_t *>(arow1 + ks * 16 + 8 + 2 * tq);
            mma_bf16_16816(acc, a, fr.b1[ks][0], fr.b1[ks][1]);
        }
        const int col = 8 * warp + 2 * tq;          // local W_1 row (0..63)
        const int t0 = mt * 16 + g, t1 = t0 + 8;
        *reinterpret_cast<uint32_t *>(uown + t0 * UOWN_LD + col) =
            (uint32_t)f2bf(act_fn(p.act, acc[0])) | ((uint32_t)f2bf(act_fn(p.act, acc[1])) << 16);
        *reinterpret_cast<uint32_t *>(uown + t1 * UOWN_LD + col) =
            (uint32_t)f2bf(act_fn(p.act, acc[2])) | ((uint32_t)f2bf(act_fn(p.act, acc[3])) << 16);
    }
    cluster.sync();
    // all of u from the cluster (16-byte pieces of the peers' rows)
    {
        constexpr int PER = 32 * (2 * RANK / 8) / 256;   // 8 uint4 per thread
        uint4 u4[PER];
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int i = threadIdx.x + 256 * q, t = i / (2 * RANK / 8), f = 8 * (i % (2 * RANK / 8));
            u4[q] = make_uint4(0, 0, 0, 0);
            if (t < cnt)
                u4[q] = *reinterpret_cast<const uint4 *>(cluster.map_shared_rank(uown, f / 64) + t * UOWN_LD +
                                                         (f % 64));
        }
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int i = threadIdx.x + 256 * q, t = i / (2 * RANK / 8), f = 8 * (i % (2 * RANK / 8));
            *reinterpret_cast<uint4 *>(uop + t * UOP_LD + f) = u4[q];
        }
    }
    __syncthreads();
    // z = c + W_2 u: warp w -> 8 channels (w % 4), half of K (w / 4); the two
    // halves meet in shared memory
    __shared__ float zhalf[2][32][32];
    for (int mt = 0; mt * 16 < cnt; ++mt) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        const uint16_t *arow0 = uop + (mt * 16 + g) * UOP_LD + khalf * RANK, *arow1 = arow0 + 8 * UOP_LD;
#pragma unroll
        for (int ks = 0; ks < RANK / 16; ++ks) {
            uint32_t a[4];
            a[0] = *reinterpret_cast<const uint32_t *>(arow0 + ks * 16 + 2 * tq);
            a[1] = *reinterpret_cast<const uint32_t *>(arow1 + ks * 16 + 2 * tq);
            a[2] = *reinterpret_cast<const uint32_t *>(arow0 + ks * 16 + 8 + 2 * tq);
            a[3] = *reinterpret_cast<const uint32_t *>(arow1 + ks * 16 + 8 + 2 * tq);
            mma_bf16_16816(acc, a, fr.b2[ks][0], fr.b2[ks][1]);
        }
        const int col = 8 * (warp & 3) + 2 * tq;
        const int t0 = mt * 16 + g;
        zhalf[khalf][t0][col] = acc[0];
        zhalf[khalf][t0][col + 1] = acc[1];
        zhalf[khalf][t0 + 8][col] = acc[2];
        zhalf[khalf][t0 + 8][col + 1] = acc[3];
    }
    __syncthreads();
    float *zf = p.z_final ? p.z_final : p.zbuf;
    for (int i = threadIdx.x; i < cnt * 32; i += blockDim.x) {
        const int t = i / 32, dd = i % 32, k = m + 1 + t, d = d0 + dd;
        const float z = cown[t][dd] + (zhalf[0][t][dd] + zhalf[1][t][dd]);
        zf[((size_t)s * B + k) * RANK + d] = z;
        static_cast<uint16_t *>(p.zpack)[(size_t)(off + t) * RANK + d] = f2bf(z);
    }
}

// grid (8, b), cluster (8, 1, 1), 256 threads.  CTA `rank` of block s owns
// channels [32 rank, +32) of c and z, and rows [64 rank, +64) of W_1; c and
// sigma(W_1 c) are exchanged through distributed shared memory.
__global__ void __cluster_dims__(MLP_CLUSTER, 1, 1) __launch_bounds__(256, 2) k_mix_mlp(const Params *__restrict__ pp)
{
    const unsigned long long t_start = globaltimer_ns();
    pdl_trigger();                     // the Read kernel may start its prologue
    const Params &p = *pp;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int s = blockIdx.y, B = p.B;
    MlpFrags fr;
    if (p.dtype) load_mlp_frags(p, rank, fr);
    pdl_wait();                        // the previous pass (or the precompute) is complete
    const int trs = (p.trace && s == 0 && rank == 0 && threadIdx.x == 0 && p.ctl[CTL_PASS] < 2)
                        ? 210 + 8 * p.ctl[CTL_PASS] : 0;
    if (trs) trace_mark(p.trace, trs, t_start);
    const SeqState st = p.st[s];
    if (!st.active) return;            // uniform over the cluster
    const int m = st.m, cnt = st.cnt, off = st.off;
    const int d0 = rank * 32;

    __shared__ float e[MAX_B][32];                     // gathered E' rows, own channel slice
    __shared__ __align__(16) float cown[MAX_B][32];    // c, own channel slice (unrounded)
    __shared__ __align__(16) float uown[MAX_B][64];    // sigma(W_1 c), own rows (fp32 path)
    extern __shared__ __align__(16) float dyn[];

    // Fuse (token part) + Mix for the own channel slice
    for (int i = threadIdx.x; i < B * 32; i += blockDim.x) {
        const int j = i / 32, dd = i % 32;
        int x = j == 0 ? p.anchor[s] : p.tokens[(size_t)s * B + j - 1];
        if (x < 0 || x >= p.V) x = 0;   // reported by k_init
        e[j][dd] = p.Ep[(size_t)x * RANK + d0 + dd];
    }
    __syncthreads();
    if (trs) trace_mark(p.trace, trs + 1, t_start);
    for (int i = threadIdx.x; i < cnt * 32; i += blockDim.x) {
        const int t = i / 32, dd = i % 32, k = m + 1 + t, d = d0 + dd;
        float lrow[MAX_B];
        if (p.Lpk) {
            const uint16_t *lp = p.Lpk + (size_t)(k * (k - 1) / 2) * RANK + d;
#pragma unroll
            for (int j = 0; j < MAX_B; ++j) lrow[j] = j < k ? bf2f(lp[(size_t)j * RANK]) : 0.0f;
        } else {
            const size_t lb = ((size_t)d * B + k) * B;
#pragma unroll
            for (int j = 0; j < MAX_B; ++j) lrow[j] = j < k ? ld_any(p.L, p.dtype, lb + j) : 0.0f;
        }
        float acc = p.Pc[((size_t)s * B + k) * RANK + d] + e[k][dd];
#pragma unroll
        for (int j = 0; j < MAX_B; ++j)
            if (j < k) acc = fmaf(lrow[j], e[j][dd], acc);
        cown[t][dd] = acc;
    }
    if (trs) trace_mark(p.trace, trs + 2, t_start);
    cluster.sync();
    if (trs) trace_mark(p.trace, trs + 3, t_start);
    if (p.dtype) {
        uint16_t *cop = reinterpret_cast<uint16_t *>(dyn);
        uint16_t *uop = cop + 32 * COP_LD;
        uint16_t *uo = uop + 32 * UOP_LD;
        mlp_share_mma(p, cluster, rank, cnt, m, s, off, cown, cop, uop, uo, fr);
    } else {
        float *cop = dyn;
        float *uop = dyn + MAX_B * RANK;
        mlp_share<float, false>(p, cluster, rank, cnt, m, s, off, cown, uown, cop, uop, nullptr);
    }
    if (trs) trace_mark(p.trace, trs + 4, t_start);
    cluster.sync();                     // peers may still read our shared memory
    if (trs) trace_mark(p.trace, trs + 5, t_start);
    if (threadIdx.x == 0 && p.trace) trace_mark(p.trace, 8 + 4 * p.ctl[CTL_PASS], t_start);
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
                select_group(sel, row, g * GROUP, min(GROUP, p.V - g * GROUP), invT,
                             invT > 0.0f ? group_noise(seed, (uint32_t)g, pos, p.offset) : 0.0f);
            }
            __syncwarp();
        }
        sst[warp][lane] = sel;
        __syncthreads();
        if (warp == 0 && lane < nt) {
            const bool sampling = invT > 0.0f;
            RPartial a = sst[0][lane].partial();
            for (int w = 1; w < 8; ++w) merge_rpartial(a, sst[w][lane].partial(), sampling);
            p.part[(size_t)(t0 + lane) * p.S + blockIdx.x] = a;
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
    const unsigned long long t_start = globaltimer_ns();
    pdl_wait();
    const Params &p = *pp;
    const int s = blockIdx.x, B = p.B, warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int pass = p.ctl[CTL_PASS];               // passes before this one (updated by the last CTA)
    const int tr_slot = 8 + 4 * pass + 2;
    const SeqState st = p.st[s];
    __shared__ int last;
    __shared__ int ynew[MAX_B], yold[MAX_B];
    __shared__ int wsum[32];
    if (st.active && warp < B && warp > st.m && warp <= st.m + st.cnt) {
        const int k = warp, i = st.off + (k - st.m - 1), tok = s * B + k;
        if (lane == 0) yold[k] = p.tokens[tok];
        const float T = p.temperature[s];
        const TokenResult res = reduce_token(p, i, tok, T > 0.0f ? 1.0f / T : 0.0f, p.seed[s]);
        if (lane == 0) {
            ynew[k] = res.y;
            if (p.lse) p.lse[tok] = res.lse;
            if (p.logit_sel) p.logit_sel[tok] = res.sel;
            p.tokens[tok] = res.y;
            record_traj(p, tok, pass, res.y);
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        if (st.active) converge_block(p, s, st, ynew, yold, 0);
        __threadfence();
        last = atomicAdd(&p.ctl[CTL_DONE], 1) == p.b - 1;
        if (!last) trace_mark(p.trace, tr_slot, t_start);
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    pack_next_pass(p, handle, wsum);
    if (threadIdx.x == 0) trace_mark(p.trace, tr_slot, t_start);
}

// Profiling hook: the next Read pass evaluates tokens 0..n-1.
__global__ void k_prof_prepare(int32_t *ctl, int32_t *act_tok, int n)
{
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t < n) act_tok[t] = t;
    if (t == 0) ctl[CTL_NACT] = n;
}

}  // namespace xp
