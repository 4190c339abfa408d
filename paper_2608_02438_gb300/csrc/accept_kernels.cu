// accept_kernels.cu -- speculative acceptance of refined blocks (Sec. 3.1).
//
//   k_acc_rows    per target row (block position k = 1..B+1) and vocabulary
//                 chunk: argmax (T <= 0) or the running max / sum of exp of
//                 target / T (T > 0)
//   k_acc_finalize per block and vocabulary chunk: the decision (greedy --
//                 longest prefix equal to the target argmax plus the target's
//                 next token; lossless -- accept y_k while u_k q_k(y_k) <
//                 p_k(y_k), q from the refinement pass (exp(l_y/T - lse)),
//                 p = softmax(target_k / T)), then for a sampling block the
//                 draw over the chunk: Gumbel-max over log max(0, p_k - q_k)
//                 at the first rejected position (q_k recomputed from z_final
//                 through W_r), with the draw from p_k alongside for an empty
//                 residual, or the bonus draw from p_{B+1} after B acceptances;
//                 the block's last chunk combines the draws and emits the token
#include "common.cuh"
#include "kernels.h"

namespace xp {

// 8 consecutive values of a row as fp32 (zeros past `n`).
__device__ __forceinline__ void load8(float (&x)[8], const void *base, int dtype, size_t i, int n)
{
    if (n >= 8) {
        if (dtype) {
            const uint4 w = __ldg(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(base) + i));
            const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                x[2 * q] = __uint_as_float(ww[q] << 16);
                x[2 * q + 1] = __uint_as_float(ww[q] & 0xFFFF0000u);
            }
        } else {
            const float4 a = __ldg(reinterpret_cast<const float4 *>(static_cast<const float *>(base) + i));
            const float4 b = __ldg(reinterpret_cast<const float4 *>(static_cast<const float *>(base) + i + 4));
            x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
        }
        return;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) x[j] = j < n ? ld_any(base, dtype, i + j) : 0.0f;
}

__device__ __forceinline__ Partial ldcg_partial16(const Partial *q)
{
    const float4 v = __ldcg(reinterpret_cast<const float4 *>(q));
    return Partial{v.x, __float_as_int(v.y), v.z, v.w};
}

// grid (b * (B + 1), chunks); chunk boundaries are multiples of 8 ids.
// The four kernels are chained with programmatic dependent launch: each lets
// the next one start early and waits (griddepcontrol.wait) for its
// predecessor's results right before reading them.  k_acc_rows reads only the
// target logits and temperatures, so it may run while the preceding kernel of
// the stream (the refinement) finishes; it waits for that kernel before it
// exits, so that the later kernels' waits cover it too.
__global__ void __launch_bounds__(256) k_acc_rows(AcceptParams p)
{
    pdl_trigger();
    if (blockIdx.x == 0 && blockIdx.y == 0) {
        if (threadIdx.x == 0) *p.status = 0;
        for (int q = threadIdx.x; q < p.b; q += blockDim.x) p.ticket[q] = 0;
    }
    const int row = blockIdx.x;                   // seq * (B + 1) + k
    const int seq = row / (p.B + 1);
    const int chunks = gridDim.y, c = blockIdx.y;
    const int V8 = (p.V + 7) / 8;
    const int v0 = 8 * (int)((long long)V8 * c / chunks), v1 = min(p.V, 8 * (int)((long long)V8 * (c + 1) / chunks));
    const float T = p.temperature[seq];
    const float invT = T > 0.0f ? 1.0f / T : 0.0f;
    Partial a{-INFINITY, 0x7fffffff, -INFINITY, 0.0f};
    const size_t base = (size_t)row * p.V;
    for (int v = v0 + 8 * threadIdx.x; v < v1; v += 8 * blockDim.x) {
        float x[8];
        const int nv = min(8, v1 - v);
        load8(x, p.target, p.dtype, base + v, nv);
        if (invT <= 0.0f) {
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (j < nv && x[j] > a.best) { a.best = x[j]; a.idx = v + j; }
        } else {
            float mx = -INFINITY;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (j < nv) mx = fmaxf(mx, x[j] * invT);
            float sum = 0.0f;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (j < nv) sum += __expf(x[j] * invT - mx);
            merge_lse(a.m, a.s, mx, sum);
        }
    }
    __shared__ Partial sp[256];
    sp[threadIdx.x] = a;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (threadIdx.x < w) {
            Partial x = sp[threadIdx.x];
            merge_partial(x, sp[threadIdx.x + w], invT > 0.0f);
            sp[threadIdx.x] = x;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) p.rowpart[(size_t)row * chunks + c] = sp[0];
    pdl_wait();
}

// grid (b, chunks2), 256 threads.  Warp 0 of every CTA takes block seq's
// decision: lane k combines the chunk partials of target row k and decides
// position k (greedy: y_k equals the target argmax; lossless: u_k q_k(y_k) <
// p_k(y_k), q from the refinement pass, p = softmax(target_k / T)); a ballot
// finds the first position not accepted.  Chunk 0 publishes the accepted
// prefix (and, greedy, the target's token after it).  For a sampling block
// every CTA then draws over its vocabulary chunk -- Gumbel-max over
// log max(0, p_k - q_k) at the first rejected position (q_k recomputed from
// z_final through W_r), with the draw from p_k alongside for an empty
// residual, or the bonus draw from p_{B+1} after B acceptances -- and the last
// CTA of the block (ticket) combines the chunks and emits the token.
//
// k_acc_finalize never triggers its dependents early (no griddepcontrol.
// launch_dependents): the next acceptance call's k_acc_rows, which may reuse
// the same scratch (always, for xpress_accept_noalloc), clears the status
// word and the tickets before its own dependency wait, so it must not start
// until every CTA of this kernel has exited.
__global__ void __launch_bounds__(256) k_acc_finalize(AcceptParams p, int chunks)
{
    pdl_wait();                                   // the row partials (and the refinement before them)
    const int seq = blockIdx.x, c = blockIdx.y, nch = gridDim.y;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int B = p.B;
    const float T = p.temperature[seq];
    const bool sampling = T > 0.0f;
    const float invT = sampling ? 1.0f / T : 0.0f;
    __shared__ Partial rows[MAX_B + 1];
    __shared__ int s_n;
    __shared__ float s_lsep;
    __shared__ int s_last;
    if (warp == 0) {
        for (int k = lane; k <= B; k += 32) {
            Partial a{-INFINITY, 0x7fffffff, -INFINITY, 0.0f};
            const size_t r = (size_t)seq * (B + 1) + k;
            // eight chunks' partials requested together per round
            for (int c0 = 0; c0 < chunks; c0 += 8) {
                Partial q[8];
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    q[u] = c0 + u < chunks ? ldcg_partial16(p.rowpart + r * chunks + c0 + u)
                                           : Partial{-INFINITY, 0x7fffffff, -INFINITY, 0.0f};
#pragma unroll
                for (int u = 0; u < 8; ++u) merge_partial(a, q[u], sampling);
            }
            rows[k] = a;
        }
        __syncwarp();
        int y = -1;
        bool ok = false;
        if (lane < B) {
            y = p.tokens[(size_t)seq * B + lane];
            if (y < 0 || y >= p.V) {
                if (c == 0) set_status(p.status, ST_BOUNDS);
                y = 0;
            }
            if (!sampling) {
                ok = y == rows[lane].idx;
            } else {
                const int row = seq * (B + 1) + lane;
                const float lse_p = rows[lane].m + logf(rows[lane].s);
                const float p_y = expf(ld_any(p.target, p.dtype, (size_t)row * p.V + y) * invT - lse_p);
                const float q_y = expf(p.logit_sel[(size_t)seq * B + lane] - p.lse[(size_t)seq * B + lane]);
                const float u = uniform01(p.seed[seq], 0u, (uint32_t)lane, STREAM_ACCEPT, p.offset);
                ok = u * q_y < p_y;
            }
        }
        const unsigned rejected = __ballot_sync(0xffffffffu, lane < B && !ok);
        const int n = rejected ? __ffs(rejected) - 1 : B;
        if (c == 0) {
            int32_t *out = p.out_tokens + (size_t)seq * (B + 1);
            for (int k = lane; k <= B; k += 32) out[k] = k < n ? p.tokens[(size_t)seq * B + k] : -1;
            __syncwarp();
            if (lane == 0) {
                if (!sampling) out[n] = rows[n].idx;
                p.accept_len[seq] = n;
            }
        }
        if (lane == 0) {
            s_n = n;
            s_lsep = (sampling && n < B) ? rows[n].m + logf(rows[n].s) : 0.0f;
        }
    }
    __syncthreads();
    if (!sampling) return;
    const int k = s_n;
    const int v0 = (int)((long long)p.V * c / nch), v1 = (int)((long long)p.V * (c + 1) / nch);
    __shared__ float zop[RANK];
    const bool resid = k < B;
    if (resid)
        for (int d = threadIdx.x; d < RANK; d += blockDim.x)
            zop[d] = round_op(p.z_final[((size_t)seq * B + k) * RANK + d], p.dtype);
    __syncthreads();
    const unsigned long long seed = p.seed[seq];
    const size_t trow = (size_t)seq * (B + 1) + k;
    const float lse_p = s_lsep;
    const float lse_q = resid ? p.lse[(size_t)seq * B + k] : 0.0f;
    float rb = -INFINITY, pb = -INFINITY;
    int ri = 0x7fffffff, pi = 0x7fffffff;
    if (resid && p.dtype) {
        // bf16: a warp takes 32 rows of W_r at a time, one coalesced 512-byte
        // row per load (lane l holds z[8l .. 8l + 7] and the same slice of the
        // row), the partial products meet through shuffles, and lane u keeps
        // row u's sum for the draw
        const int lane = threadIdx.x % 32, nw = blockDim.x / 32;
        float z8[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) z8[j] = zop[8 * lane + j];
        const uint16_t *wr = static_cast<const uint16_t *>(p.W_r);
        for (int gb = v0 + (threadIdx.x / 32) * 32; gb < v1; gb += nw * 32) {
            float myacc = 0.0f;
#pragma unroll 1
            for (int u0 = 0; u0 < 32; u0 += 8) {
                uint4 w[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int row = gb + u0 + u;
                    w[u] = row < v1 ? __ldg(reinterpret_cast<const uint4 *>(wr + (size_t)row * RANK) + lane)
                                    : make_uint4(0, 0, 0, 0);
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const uint32_t ww[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
                    float part = 0.0f;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        part = fmaf(__uint_as_float(ww[q] << 16), z8[2 * q], part);
                        part = fmaf(__uint_as_float(ww[q] & 0xFFFF0000u), z8[2 * q + 1], part);
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
                    if (lane == u0 + u) myacc = part;
                }
            }
            const int v = gb + lane;
            if (v < v1) {
                const float tx = ld_any(p.target, p.dtype, trow * p.V + v) * invT;
                const float g = gumbel(seed, (uint32_t)v, (uint32_t)k, STREAM_RESID, p.offset);
                merge_argmax(pb, pi, tx + g, v);
                const float lx = (myacc + ld_any(p.s, p.dtype, ((size_t)seq * B + k) * p.V + v)) * invT;
                const float res = expf(tx - lse_p) - expf(lx - lse_q);
                if (res > 0.0f) merge_argmax(rb, ri, logf(res) + g, v);
            }
        }
    } else
    for (int v = v0 + threadIdx.x; v < v1; v += blockDim.x) {
        const float tx = ld_any(p.target, p.dtype, trow * p.V + v) * invT;
        const float g = gumbel(seed, (uint32_t)v, (uint32_t)k, STREAM_RESID, p.offset);
        merge_argmax(pb, pi, tx + g, v);
        if (resid) {
            float acc = 0.0f;
            for (int d = 0; d < RANK; ++d) acc = fmaf(ld_any(p.W_r, p.dtype, (size_t)v * RANK + d), zop[d], acc);
            const float lx = (acc + ld_any(p.s, p.dtype, ((size_t)seq * B + k) * p.V + v)) * invT;
            const float res = expf(tx - lse_p) - expf(lx - lse_q);
            if (res > 0.0f) merge_argmax(rb, ri, logf(res) + g, v);
        }
    }
    __shared__ float sb[2][256];
    __shared__ int si[2][256];
    sb[0][threadIdx.x] = rb; si[0][threadIdx.x] = ri;
    sb[1][threadIdx.x] = pb; si[1][threadIdx.x] = pi;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (threadIdx.x < w)
            for (int h = 0; h < 2; ++h) {
                float b0 = sb[h][threadIdx.x];
                int i0 = si[h][threadIdx.x];
                merge_argmax(b0, i0, sb[h][threadIdx.x + w], si[h][threadIdx.x + w]);
                sb[h][threadIdx.x] = b0;
                si[h][threadIdx.x] = i0;
            }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        p.spart[(size_t)seq * nch + c] = Partial{sb[0][0], si[0][0], sb[1][0], __int_as_float(si[1][0])};
        __threadfence();
        s_last = atomicAdd(p.ticket + seq, 1) == nch - 1;
    }
    __syncthreads();
    if (!s_last) return;
    // every chunk of this block has drawn: the last CTA combines the chunks'
    // results (each thread a share, then the tree above) and emits the token
    __threadfence();
    float cb = -INFINITY, cp = -INFINITY;
    int ci = 0x7fffffff, cpi = 0x7fffffff;
    for (int cc = threadIdx.x; cc < nch; cc += blockDim.x) {
        const Partial a = ldcg_partial16(p.spart + (size_t)seq * nch + cc);
        merge_argmax(cb, ci, a.best, a.idx);
        merge_argmax(cp, cpi, a.m, __float_as_int(a.s));
    }
    sb[0][threadIdx.x] = cb; si[0][threadIdx.x] = ci;
    sb[1][threadIdx.x] = cp; si[1][threadIdx.x] = cpi;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (threadIdx.x < w)
            for (int h = 0; h < 2; ++h) {
                float b0 = sb[h][threadIdx.x];
                int i0 = si[h][threadIdx.x];
                merge_argmax(b0, i0, sb[h][threadIdx.x + w], si[h][threadIdx.x + w]);
                sb[h][threadIdx.x] = b0;
                si[h][threadIdx.x] = i0;
            }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        const bool use_resid = k < B && sb[0][0] > -INFINITY;
        p.out_tokens[(size_t)seq * (B + 1) + k] = use_resid ? si[0][0] : si[1][0];
    }
}

}  // namespace xp
