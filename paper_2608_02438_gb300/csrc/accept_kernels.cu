// accept_kernels.cu -- speculative acceptance of refined blocks (Sec. 3.1).
//
//   k_acc_rows    per target row (block position k = 1..B+1) and vocabulary
//                 chunk: argmax (T <= 0) or the running max / sum of exp of
//                 target / T (T > 0)
//   k_acc_decide  per block: the decision (greedy -- longest prefix equal to
//                 the target argmax plus the target's next token; lossless --
//                 accept y_k while u_k q_k(y_k) < p_k(y_k), q from the
//                 refinement pass (exp(l_y/T - lse)), p = softmax(target_k / T))
//                 and, for a sampling block, its draw descriptor
//                 (batches of at most ACCEPT_FUSED_MAX_B blocks skip this
//                 kernel: every CTA of k_acc_draw takes the decisions itself,
//                 which saves a dependent launch on the latency-bound path)
//   k_acc_draw    every draw of the batch over every vocabulary range:
//                 Gumbel-max over log max(0, p_k - q_k) at the first rejected
//                 position (q_k recomputed from z_final through W_r, read once
//                 per 16 draws), with the draw from p_k alongside for an empty
//                 residual, or the bonus draw from p_{B+1} after B acceptances;
//                 the last CTA emits the drawn tokens
#include "common.cuh"
#include "kernels.h"
#include "mlp_common.cuh"

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

// Persistent grid; work item i = (target row i / chunks, vocabulary chunk
// i % chunks), dealt round-robin so that the CTAs stay evenly loaded (a large
// batch has many more items than resident CTAs); chunk boundaries are
// multiples of 8 ids.  The three kernels are chained with programmatic dependent launch: each of
// the first two lets the next one start early and every kernel waits
// (griddepcontrol.wait) for its predecessor's results right before reading
// them.  k_acc_rows reads only the target logits and temperatures, so it may
// run while the preceding kernel of the stream (the refinement) finishes; it
// waits for that kernel before it exits, so that the later kernels' waits
// cover it too.  It clears the status word and the draw counters.
__global__ void __launch_bounds__(256) k_acc_rows(AcceptParams p, int chunks)
{
    pdl_trigger();
    if (blockIdx.x == 0) {
        if (threadIdx.x == 0) {
            *p.status = 0;
            p.ticket[0] = 0;                      // draws listed by k_acc_decide
            p.ticket[1] = 0;                      // CTAs of k_acc_draw done
        }
        for (int i = threadIdx.x; i < 2 * p.b; i += blockDim.x) p.keys[i] = 0ull;   // draw keys
    }
    __shared__ Partial sp[256];
    const int items = p.b * (p.B + 1) * chunks;
    for (int item = blockIdx.x; item < items; item += gridDim.x) {
        const int row = item / chunks;            // seq * (B + 1) + k
        const int seq = row / (p.B + 1);
        const int c = item % chunks;
        const int V8 = (p.V + 7) / 8;
        const int v0 = 8 * (int)((long long)V8 * c / chunks);
        const int v1 = min(p.V, 8 * (int)((long long)V8 * (c + 1) / chunks));
        const float T = p.temperature[seq];
        const float invT = T > 0.0f ? 1.0f / T : 0.0f;
        Partial a{-INFINITY, 0x7fffffff, -INFINITY, 0.0f};
        const size_t base = (size_t)row * p.V;
        // four 8-value pieces per thread in flight (the stream is latency-bound
        // with one); pieces are visited in increasing id order per thread.
        // Sampling rows keep the running max in log2 units (y = x log2(e) / T)
        // and rescale the running sum once per piece, so that each value costs
        // one multiply, one max, one subtract, one ex2 and one add.
        constexpr int U = 4;
        const int step = 8 * blockDim.x;
        const float c2 = invT * 1.4426950408889634f;
        float m2 = -INFINITY, s2 = 0.0f;
        for (int vv = v0 + 8 * threadIdx.x; vv < v1; vv += U * step) {
            float x[U][8];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int v = vv + u * step;
                if (v < v1) load8(x[u], p.target, p.dtype, base + v, min(8, v1 - v));
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int v = vv + u * step;
                if (v >= v1) break;
                const int nv = min(8, v1 - v);
                if (nv < 8)                               // the chunk's ragged end: past V reads as -inf
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        if (j >= nv) x[u][j] = -INFINITY;
                if (invT <= 0.0f) {
                    const float m8 = fmaxf(fmaxf(fmaxf(x[u][0], x[u][1]), fmaxf(x[u][2], x[u][3])),
                                           fmaxf(fmaxf(x[u][4], x[u][5]), fmaxf(x[u][6], x[u][7])));
                    if (m8 > a.best) {                    // the first id of the piece that holds it
                        int jj = 7;
#pragma unroll
                        for (int j = 6; j >= 0; --j)
                            if (x[u][j] == m8) jj = j;
                        a.best = m8;
                        a.idx = v + jj;
                    }
                } else {
                    float y[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) y[j] = x[u][j] * c2;
                    const float m8 = fmaxf(fmaxf(fmaxf(y[0], y[1]), fmaxf(y[2], y[3])),
                                           fmaxf(fmaxf(y[4], y[5]), fmaxf(y[6], y[7])));
                    const float mn = fmaxf(m2, m8);
                    float t = 0.0f;
#pragma unroll
                    for (int j = 0; j < 8; ++j) t += ex2_approx(y[j] - mn);
                    s2 = s2 * ex2_approx(m2 - mn) + t;
                    m2 = mn;
                }
            }
        }
        if (invT > 0.0f && m2 > -INFINITY) {              // back to natural units: sum e^(x / T - m)
            a.m = m2 * 0.6931471805599453f;
            a.s = s2;
        }
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
        __syncthreads();                          // sp is reused by the next item
    }
    pdl_wait();
}

// One warp: the decision of block `seq`.  Lane k combines the chunk partials
// of target row k and decides position k (greedy: y_k equals the target
// argmax; lossless: u_k q_k(y_k) < p_k(y_k), q from the refinement pass,
// p = softmax(target_k / T)); a ballot finds the first position not
// accepted.  With `write`, the warp writes the accepted prefix, -1 past it
// and the accept length; a greedy block also the target's token after the
// prefix (a sampling block's token there is the draw's).  Returns whether the
// block samples and, for a sampling block, fills its draw descriptor (its
// rejected position, or B for the bonus draw).
__device__ __forceinline__ bool decide_block(const AcceptParams &p, int seq, int lane, Partial *rows, bool write,
                                             DrawDesc &dd)
{
    const int B = p.B, chunks = p.chunks;
    const float T = p.temperature[seq];
    const bool sampling = T > 0.0f;
    const float invT = sampling ? 1.0f / T : 0.0f;
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
            set_status(p.status, ST_BOUNDS);
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
    if (write) {
        int32_t *out = p.out_tokens + (size_t)seq * (B + 1);
        for (int k = lane; k <= B; k += 32)
            if (k != n) out[k] = k < n ? p.tokens[(size_t)seq * B + k] : -1;
        if (lane == 0) {
            p.accept_len[seq] = n;
            if (!sampling) out[n] = rows[n].idx;
        }
    }
    if (sampling) {
        dd.seq = seq;
        dd.k = n;
        dd.invT = invT;
        dd.lse_p = rows[n].m + logf(rows[n].s);
        dd.lse_q = n < B ? p.lse[(size_t)seq * B + n] : 0.0f;
    }
    __syncwarp();                                 // rows is reused by the warp's next block
    return sampling;
}

// grid b, 32 threads (one warp per block): the block's decision
// (decide_block); a sampling block appends its draw descriptor for
// k_acc_draw.
__global__ void __launch_bounds__(32) k_acc_decide(AcceptParams p)
{
    pdl_trigger();                                // k_acc_draw may start its prologue
    pdl_wait();                                   // the row partials (and the refinement before them)
    __shared__ Partial rows[MAX_B + 1];
    DrawDesc dd{};
    if (decide_block(p, blockIdx.x, threadIdx.x, rows, true, dd) && threadIdx.x == 0) p.draws[atomicAdd(p.ticket, 1)] = dd;
}

// Small batches (fused): every CTA of the draw kernel takes all the
// decisions itself (warp w: blocks w, w + 8, ...), CTA 0 writes the accepted
// prefixes, and the sampling blocks' draw descriptors are listed in block
// order in shared memory (the same list in every CTA).  Returns their count.
__device__ __forceinline__ int decide_all(const AcceptParams &p, DrawDesc *list, Partial (*rows)[MAX_B + 1],
                                          int *sflag)
{
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32, nwarps = blockDim.x / 32;
    for (int seq = warp; seq < p.b; seq += nwarps) {
        DrawDesc dd{};
        const bool s = decide_block(p, seq, lane, rows[warp], blockIdx.x == 0, dd);
        if (lane == 0) {
            sflag[seq] = s;
            if (s) list[seq] = dd;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int nd = 0;
        for (int seq = 0; seq < p.b; ++seq)
            if (sflag[seq]) list[nd++] = list[seq];
        sflag[ACCEPT_FUSED_MAX_B] = nd;
    }
    __syncthreads();
    return sflag[ACCEPT_FUSED_MAX_B];
}

namespace {
constexpr int DRAW_NZ = 16;         // draws per sweep of the vocabulary (accumulators per lane)
constexpr int DRAW_THREADS = 256;

// 32 consecutive elements of row v of W_r (bf16 or fp32) as floats.
__device__ __forceinline__ void load_row32(float (&w)[32], const void *W_r, int dtype, int v, int k0)
{
    if (dtype) {
        const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(W_r) + (size_t)v * RANK + k0);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint4 x = __ldg(src + c);
            const uint32_t ww[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                w[8 * c + 2 * q] = __uint_as_float(ww[q] << 16);
                w[8 * c + 2 * q + 1] = __uint_as_float(ww[q] & 0xFFFF0000u);
            }
        }
    } else {
        const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(W_r) + (size_t)v * RANK + k0);
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const float4 x = __ldg(src + c);
            w[4 * c] = x.x; w[4 * c + 1] = x.y; w[4 * c + 2] = x.z; w[4 * c + 3] = x.w;
        }
    }
}
}  // namespace

// The end of the draw kernel, every thread of every CTA: the CTA counts
// itself done; the last one emits each drawn token (the residual's draw, or
// the draw from p when the residual is empty or after B acceptances).
__device__ __forceinline__ void draw_finish(const AcceptParams &p, const DrawDesc *list, int nd, int G, int *s_last)
{
    if (threadIdx.x == 0) {
        __threadfence();
        *s_last = atomicAdd(p.ticket + 1, 1) == G - 1;
    }
    __syncthreads();
    if (!*s_last) return;
    __threadfence();
    for (int j = threadIdx.x; j < nd; j += blockDim.x) {
        const DrawDesc dd = list[j];
        const unsigned long long kr = __ldcg(p.keys + 2 * dd.seq), kp = __ldcg(p.keys + 2 * dd.seq + 1);
        float best;
        int idx;
        argmax_unkey(dd.k < p.B && kr ? kr : kp, best, idx);
        p.out_tokens[(size_t)dd.seq * (p.B + 1) + dd.k] = idx;
    }
}

// The Gumbel noise of ids v and v + 1 (v even: one Philox call gives both).
__device__ __forceinline__ void gumbel_pair(unsigned long long seed, uint32_t v, uint32_t pos, uint32_t stream,
                                            uint32_t offset, float &g0, float &g1)
{
    const uint4 o = philox10(make_uint4(v >> 2, pos, stream, offset), (uint32_t)seed, (uint32_t)(seed >> 32));
    const uint32_t w0 = (v & 2u) ? o.z : o.x, w1 = (v & 2u) ? o.w : o.y;
    g0 = -logf(-logf(((float)(w0 >> 9) + 0.5f) * (1.0f / 8388608.0f)));
    g1 = -logf(-logf(((float)(w1 >> 9) + 0.5f) * (1.0f / 8388608.0f)));
}

// Scores of one (draw, vocabulary id) pair, merged into the lane's running
// bests: the p draw tx + g, and for a residual draw log(max(0, p - q)) + g
// with l = acc + s recomputed (acc = (W_r z)_v).
__device__ __forceinline__ void draw_element(const AcceptParams &p, const DrawDesc &dd, unsigned long long seed, int v,
                                             float acc, float g, float &rb, int &ri, float &pb, int &pi)
{
    const size_t trow = (size_t)dd.seq * (p.B + 1) + dd.k;
    const float tx = ld_any(p.target, p.dtype, trow * p.V + v) * dd.invT;
    merge_argmax(pb, pi, tx + g, v);
    if (dd.k < p.B) {
        const float lx = (acc + ld_any(p.s, p.dtype, ((size_t)dd.seq * p.B + dd.k) * p.V + v)) * dd.invT;
        const float res = expf(tx - dd.lse_p) - expf(lx - dd.lse_q);
        if (res > 0.0f) merge_argmax(rb, ri, logf(res) + g, v);
    }
}

// grid G, 256 threads; CTA r owns the vocabulary range [V r / G, V (r+1) / G).
// Every draw of the batch (one per sampling block, listed by k_acc_decide) is
// taken over every range: Gumbel-max over log max(0, p_k - q_k) at the first
// rejected position k (q_k recomputed from z_final through W_r: each lane owns
// one vocabulary row and takes its dot products with the z of up to 16 draws
// held in shared memory, so W_r is read once per 16 draws), with the draw from
// p_k alongside for an empty residual, or the bonus draw from p_{B+1} after B
// acceptances.  Each range's best keys meet through 64-bit atomicMax (the
// fp32 score made order-preserving, then the inverted id: ties go to the
// smallest id); the last CTA to finish emits every drawn token.
//
// This is the last kernel of an acceptance call and it never triggers its
// dependents early (no griddepcontrol.launch_dependents): the next call's
// k_acc_rows, which may reuse the same scratch (always, for
// xpress_accept_noalloc), clears the counters before its own dependency wait,
// so it must not start until every CTA of this kernel has exited.
__global__ void __launch_bounds__(DRAW_THREADS) k_acc_draw_simt(AcceptParams p)
{
    pdl_wait();                                   // the draw list of k_acc_decide (or the row partials)
    __shared__ DrawDesc flist[ACCEPT_FUSED_MAX_B];
    __shared__ Partial frows[DRAW_THREADS / 32][MAX_B + 1];
    __shared__ int fflag[ACCEPT_FUSED_MAX_B + 1];
    const int nd = p.fused ? decide_all(p, flist, frows, fflag) : __ldcg(p.ticket);
    const DrawDesc *list = p.fused ? flist : p.draws;
    if (nd == 0) return;
    const int G = gridDim.x, r = blockIdx.x, warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int nwarps = DRAW_THREADS / 32, B = p.B;
    const int v0 = (int)((long long)p.V * r / G), v1 = (int)((long long)p.V * (r + 1) / G);
    __shared__ float zs[DRAW_NZ][RANK];
    __shared__ DrawDesc dsc[DRAW_NZ];
    __shared__ unsigned long long wkey[DRAW_THREADS / 32][DRAW_NZ][2];
    __shared__ int s_any_resid, s_last;
    for (int g0 = 0; g0 < nd; g0 += DRAW_NZ) {
        const int nz = min(DRAW_NZ, nd - g0);
        if (threadIdx.x < nz) dsc[threadIdx.x] = list[g0 + threadIdx.x];
        if (threadIdx.x == 0) s_any_resid = 0;
        __syncthreads();
        for (int i = threadIdx.x; i < nz * RANK; i += DRAW_THREADS) {
            const int j = i / RANK, d = i % RANK;
            const DrawDesc dd = dsc[j];
            const bool resid = dd.k < B;
            zs[j][d] = resid ? round_op(p.z_final[((size_t)dd.seq * B + dd.k) * RANK + d], p.dtype) : 0.0f;
            if (resid && d == 0) s_any_resid = 1;
        }
        __syncthreads();
        const bool any_resid = s_any_resid != 0;
        float rb[DRAW_NZ], pb[DRAW_NZ];
        int ri[DRAW_NZ], pi[DRAW_NZ];
#pragma unroll
        for (int j = 0; j < DRAW_NZ; ++j) { rb[j] = pb[j] = -INFINITY; ri[j] = pi[j] = 0x7fffffff; }
        for (int vb = v0 + warp * 32; vb < v1; vb += nwarps * 32) {
            const int v = vb + lane;
            const bool valid = v < v1;
            float acc[DRAW_NZ];
#pragma unroll
            for (int j = 0; j < DRAW_NZ; ++j) acc[j] = 0.0f;
            if (any_resid && valid) {
#pragma unroll 1
                for (int k0 = 0; k0 < RANK; k0 += 32) {
                    float w[32];
                    load_row32(w, p.W_r, p.dtype, v, k0);
#pragma unroll
                    for (int j = 0; j < DRAW_NZ; ++j) {
                        if (j < nz) {
                            const float4 *zz = reinterpret_cast<const float4 *>(&zs[j][k0]);
                            float a = acc[j];
#pragma unroll
                            for (int c = 0; c < 8; ++c) {
                                const float4 z4 = zz[c];
                                a = fmaf(w[4 * c], z4.x, a);
                                a = fmaf(w[4 * c + 1], z4.y, a);
                                a = fmaf(w[4 * c + 2], z4.z, a);
                                a = fmaf(w[4 * c + 3], z4.w, a);
                            }
                            acc[j] = a;
                        }
                    }
                }
            }
            if (valid) {
#pragma unroll
                for (int j = 0; j < DRAW_NZ; ++j) {
                    if (j < nz) {
                        const DrawDesc dd = dsc[j];
                        const unsigned long long seed = p.seed[dd.seq];
                        const float g = gumbel(seed, (uint32_t)v, (uint32_t)dd.k, STREAM_RESID, p.offset);
                        draw_element(p, dd, seed, v, acc[j], g, rb[j], ri[j], pb[j], pi[j]);
                    }
                }
            }
        }
        // warp, then CTA, then grid (atomicMax of the 64-bit keys)
#pragma unroll
        for (int j = 0; j < DRAW_NZ; ++j) {
            if (j < nz) {
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    merge_argmax(rb[j], ri[j], __shfl_xor_sync(0xffffffffu, rb[j], o),
                                 __shfl_xor_sync(0xffffffffu, ri[j], o));
                    merge_argmax(pb[j], pi[j], __shfl_xor_sync(0xffffffffu, pb[j], o),
                                 __shfl_xor_sync(0xffffffffu, pi[j], o));
                }
                if (lane == 0) {
                    wkey[warp][j][0] = ri[j] != 0x7fffffff ? argmax_key(rb[j], ri[j]) : 0ull;
                    wkey[warp][j][1] = pi[j] != 0x7fffffff ? argmax_key(pb[j], pi[j]) : 0ull;
                }
            }
        }
        __syncthreads();
        if (threadIdx.x < 2 * nz) {
            const int j = threadIdx.x >> 1, h = threadIdx.x & 1;
            unsigned long long k = 0ull;
            for (int w = 0; w < nwarps; ++w) k = wkey[w][j][h] > k ? wkey[w][j][h] : k;
            if (k) atomicMax(p.keys + 2 * dsc[j].seq + h, k);
        }
        __syncthreads();
    }
    draw_finish(p, list, nd, G, &s_last);
}


// bf16 refiners: the same draws with the residual's products W_r z on tensor
// cores (warp-level m16n8k16): the <= 16 draws of a sweep are the M rows
// (their bf16 z operands held as A fragments for the whole sweep), 8
// vocabulary rows the N columns, K = r.  Any permutation of K applied to
// both operands leaves the products unchanged; lane (g, t) takes, for each
// 32-wide K slab, the 16-byte piece [8t, 8t + 8) of vocabulary row g (one
// coalesced load) as the B fragments of two k-steps, and the A fragments
// follow the same order.  Lane (g, t) then owns draws g and g + 8 at rows
// 2t and 2t + 1 of the 8, whose Gumbel noise comes from one Philox call.
// CTA ranges start at multiples of 8 ids.
__global__ void __launch_bounds__(DRAW_THREADS, 2) k_acc_draw(AcceptParams p)
{
    pdl_wait();                                   // the draw list of k_acc_decide (or the row partials)
    __shared__ DrawDesc flist[ACCEPT_FUSED_MAX_B];
    __shared__ Partial frows[DRAW_THREADS / 32][MAX_B + 1];
    __shared__ int fflag[ACCEPT_FUSED_MAX_B + 1];
    const int nd = p.fused ? decide_all(p, flist, frows, fflag) : __ldcg(p.ticket);
    const DrawDesc *list = p.fused ? flist : p.draws;
    if (nd == 0) return;
    const int G = gridDim.x, r = blockIdx.x, warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int nwarps = DRAW_THREADS / 32, B = p.B;
    const int g = lane >> 2, tq = lane & 3;
    const int V8 = (p.V + 7) / 8;
    const int v0 = 8 * (int)((long long)V8 * r / G), v1 = min(p.V, 8 * (int)((long long)V8 * (r + 1) / G));
    constexpr int ZP = RANK + 8;                  // bf16 row pitch of the z operands (conflict-free fragment loads)
    __shared__ __align__(16) uint16_t zb[DRAW_NZ][ZP];
    __shared__ DrawDesc dsc[DRAW_NZ];
    __shared__ unsigned long long dseed[DRAW_NZ];
    __shared__ unsigned long long wkey[DRAW_THREADS / 32][DRAW_NZ][2];
    __shared__ int s_last;
    const uint16_t *wr = static_cast<const uint16_t *>(p.W_r);
    for (int g0 = 0; g0 < nd; g0 += DRAW_NZ) {
        const int nz = min(DRAW_NZ, nd - g0);
        if (threadIdx.x < DRAW_NZ) {
            DrawDesc dd{};
            dd.k = B;                                 // padding draws: no residual, never read
            if (threadIdx.x < nz) dd = list[g0 + threadIdx.x];
            dsc[threadIdx.x] = dd;
            dseed[threadIdx.x] = threadIdx.x < nz ? p.seed[dd.seq] : 0ull;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < DRAW_NZ * RANK; i += DRAW_THREADS) {
            const int j = i / RANK, d = i % RANK;
            const DrawDesc dd = dsc[j];
            const bool resid = j < nz && dd.k < B;
            zb[j][d] = resid ? f2bf(p.z_final[((size_t)dd.seq * B + dd.k) * RANK + d]) : (uint16_t)0;
        }
        __syncthreads();
        // A fragments of the sweep: k-step 2s + h of slab s takes physical
        // columns 32 s + 8 t + 4 h + {0, 1} (logical 2t, 2t + 1) and
        // + {2, 3} (logical 2t + 8, 2t + 9)
        uint32_t af[2 * RANK / 32][4];
#pragma unroll
        for (int s = 0; s < RANK / 32; ++s)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int c = 32 * s + 8 * tq + 4 * h;
                af[2 * s + h][0] = *reinterpret_cast<const uint32_t *>(&zb[g][c]);
                af[2 * s + h][1] = *reinterpret_cast<const uint32_t *>(&zb[g + 8][c]);
                af[2 * s + h][2] = *reinterpret_cast<const uint32_t *>(&zb[g][c + 2]);
                af[2 * s + h][3] = *reinterpret_cast<const uint32_t *>(&zb[g + 8][c + 2]);
            }
        const DrawDesc d0 = dsc[g], d1 = dsc[g + 8];
        const unsigned long long seed0 = dseed[g], seed1 = dseed[g + 8];
        const bool on0 = g < nz, on1 = g + 8 < nz;
        float rb[2] = {-INFINITY, -INFINITY}, pb[2] = {-INFINITY, -INFINITY};
        int ri[2] = {0x7fffffff, 0x7fffffff}, pi[2] = {0x7fffffff, 0x7fffffff};
        for (int vb = v0 + warp * 8; vb < v1; vb += nwarps * 8) {
            const int vrow = vb + g;                  // the row this lane loads
            uint4 w[RANK / 32];
#pragma unroll
            for (int s = 0; s < RANK / 32; ++s)
                w[s] = vrow < v1 ? __ldg(reinterpret_cast<const uint4 *>(wr + (size_t)vrow * RANK + 32 * s + 8 * tq))
                                 : make_uint4(0, 0, 0, 0);
            float c[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int s = 0; s < RANK / 32; ++s) {
                mma_bf16_16816(c, af[2 * s], w[s].x, w[s].y);
                mma_bf16_16816(c, af[2 * s + 1], w[s].z, w[s].w);
            }
            // this lane: draws g (c[0], c[1]) and g + 8 (c[2], c[3]) at ids
            // vb + 2t and vb + 2t + 1
            const int v = vb + 2 * tq;
            if (v < v1) {
                const bool two = v + 1 < v1;
                if (on0) {
                    float g0v, g1v;
                    gumbel_pair(seed0, (uint32_t)v, (uint32_t)d0.k, STREAM_RESID, p.offset, g0v, g1v);
                    draw_element(p, d0, seed0, v, c[0], g0v, rb[0], ri[0], pb[0], pi[0]);
                    if (two) draw_element(p, d0, seed0, v + 1, c[1], g1v, rb[0], ri[0], pb[0], pi[0]);
                }
                if (on1) {
                    float g0v, g1v;
                    gumbel_pair(seed1, (uint32_t)v, (uint32_t)d1.k, STREAM_RESID, p.offset, g0v, g1v);
                    draw_element(p, d1, seed1, v, c[2], g0v, rb[1], ri[1], pb[1], pi[1]);
                    if (two) draw_element(p, d1, seed1, v + 1, c[3], g1v, rb[1], ri[1], pb[1], pi[1]);
                }
            }
        }
        // the four lanes of a row group share their two draws: reduce over t
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int o = 1; o <= 2; o <<= 1) {
                merge_argmax(rb[h], ri[h], __shfl_xor_sync(0xffffffffu, rb[h], o), __shfl_xor_sync(0xffffffffu, ri[h], o));
                merge_argmax(pb[h], pi[h], __shfl_xor_sync(0xffffffffu, pb[h], o), __shfl_xor_sync(0xffffffffu, pi[h], o));
            }
        if (tq == 0)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                wkey[warp][g + 8 * h][0] = ri[h] != 0x7fffffff ? argmax_key(rb[h], ri[h]) : 0ull;
                wkey[warp][g + 8 * h][1] = pi[h] != 0x7fffffff ? argmax_key(pb[h], pi[h]) : 0ull;
            }
        __syncthreads();
        if (threadIdx.x < 2 * nz) {
            const int j = threadIdx.x >> 1, hh = threadIdx.x & 1;
            unsigned long long k = 0ull;
            for (int w2 = 0; w2 < nwarps; ++w2) k = wkey[w2][j][hh] > k ? wkey[w2][j][hh] : k;
            if (k) atomicMax(p.keys + 2 * dsc[j].seq + hh, k);
        }
        __syncthreads();
    }
    draw_finish(p, list, nd, G, &s_last);
}

}  // namespace xp
