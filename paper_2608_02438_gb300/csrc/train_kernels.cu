// train_kernels.cu -- the memory-bound and per-block steps of the refiner
// training step (Sec. 4.3) around the tensor-core products.  Every kernel of
// the step is launched with programmatic dependent launch: it signals its
// successor at once and waits for its predecessor before touching memory.
//
//   k_train_rows / _fin   one pass over s and the target logits t of every
//                         position: log-sum-exp of both (log2 domain), s at
//                         y*, and the first argmax of s (the consistency
//                         forward's inputs, argmax p^b)
//   k_train_fuse          the Fuse operand [u_h | u_g | W_e[x]] of both
//                         forwards (Eq. fuse; u_g = W_g g with g the block
//                         mean of h, taken as the mean of W_g h_j), u_h and
//                         u_g as bf16 hi + lo pairs so that W_in sees them to
//                         about 16 bits
//   k_train_mix           c_k = a_k + sum_{j<k} L_kj a_j per channel (Eq. mix),
//                         L staged in shared memory per 32 channels
//   k_train_stats_fin     lse of every row's logits from the split partials
//   k_train_tv_fin        per block the three losses and L_total; per row the
//                         coefficients of dL/dl
//   k_train_dz, _dact     dL/dz from the vocabulary splits and its bf16 copy;
//                         dL/dt = dL/du sigma'(t)
//   k_train_mix_bwd       dL/da_j = dc_j + sum_{k>j} L_kj dc_k and dL/dL_kj
//   k_train_fuse_bwd      dL/du_h per position (both forwards), dL/du_g / B
//                         per block, dL/dW_e rows (atomic, both forwards)
#include "train_common.cuh"
#include "kernels.h"

namespace xp {

namespace {

constexpr float L2E = 1.4426950408889634f;
constexpr float LN2 = 0.69314718055994531f;

__device__ __forceinline__ int pair_row(int i, int f) { return (i >> 6) * 128 + f * 64 + (i & 63); }

__device__ __forceinline__ void lse2_merge(float &m, float &s, float om, float os)
{
    const float M = fmaxf(m, om);
    if (M == -INFINITY) return;
    s = s * ex2_approx(m - M) + os * ex2_approx(om - M);
    m = M;
}

__device__ __forceinline__ float sigma_prime(int act, float t)
{
    if (act == 2) return t > 0.0f ? 1.0f : 0.0f;
    if (act == 1)
        return 0.5f * (1.0f + erff(t * 0.70710678118654752f)) + t * 0.39894228040143268f * expf(-0.5f * t * t);
    const float sg = 1.0f / (1.0f + expf(-t));
    return sg + t * sg * (1.0f - sg);
}

}  // namespace

namespace {

constexpr int ROWS_STAGES = 3;
constexpr uint32_t ROWS_SEG = TRAIN_ROW_CHUNK * 2;          // bytes of one s (or t) segment
constexpr int ROWS_THREADS = 32 * 9;                         // a copy warp, 8 reducing warps

struct RowsShared {
    uint64_t full[ROWS_STAGES], empty[ROWS_STAGES];
    float4 wp[2][8];                                          // per item parity and warp: max / sum of s and t
    float wb[2][8];
    int wi[2][8];
    int abort;
};

constexpr size_t ROWS_SMEM = 128 + ROWS_STAGES * 2 * ROWS_SEG + sizeof(RowsShared);

// OR of `pred` over the 256 reducing threads (named barrier 1): every one of
// them takes the same decision.
__device__ __forceinline__ bool rows_bar_or(bool pred)
{
    uint32_t res;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, 256, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(res)
        : "r"((uint32_t)pred)
        : "memory");
    return res != 0;
}

}  // namespace

const size_t kTrainRowsSmemBytes = ROWS_SMEM;
const int kTrainRowsThreads = ROWS_THREADS;

// grid min(SMs, P nch), ROWS_THREADS threads, ROWS_SMEM bytes: persistent
// over the (position, chunk of TRAIN_ROW_CHUNK ids) items, position-major.
// Warp 0 streams each item's s and t segments into a ROWS_STAGES-deep ring by
// bulk copies; reducing warp w takes the 8-id pieces 32 w + lane + 256 c
// (c < 8), so each of its shared-memory reads is one 512-byte run, and
// releases the stage as soon as its pieces are in registers.  The warp's
// maxima are reduced first, so every exponential is taken against the warp
// maximum and the sums need no rescale.
__global__ void __launch_bounds__(ROWS_THREADS, 1) k_train_rows(TrainMisc m)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
    RowsShared &sh = *reinterpret_cast<RowsShared *>(base + ROWS_STAGES * 2 * ROWS_SEG);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int items = m.P * m.nch;
    if (threadIdx.x == 0) {
        for (int i = 0; i < ROWS_STAGES; ++i) {
            mbar_init(&sh.full[i], 1);
            mbar_init(&sh.empty[i], 8);
        }
        sh.abort = 0;
        fence_barrier_init();
    }
    __syncthreads();
    pdl_trigger();
    pdl_wait();
    volatile int *abort = &sh.abort;
    if (warp == 0) {
        if (lane == 0) {
            uint32_t pending = 0, pend_par = 0;
            int k = 0;
            for (int it = blockIdx.x; it < items; it += gridDim.x, ++k) {
                const int st = k % ROWS_STAGES;
                const uint32_t ph = (uint32_t)((k / ROWS_STAGES) & 1);
                if (!mbar_wait(&sh.empty[st], ph ^ 1, abort)) break;
                const int i = it / m.nch, v0 = (it % m.nch) * TRAIN_ROW_CHUNK;
                // V % 8 == 0: the segment's bytes are a multiple of 16
                const uint32_t bytes = (uint32_t)min(TRAIN_ROW_CHUNK, m.V - v0) * 2u;
                uint8_t *dst = base + st * 2 * ROWS_SEG;
                mbar_expect_tx(&sh.full[st], 2 * bytes);
                bulk_load_1d(dst, static_cast<const uint16_t *>(m.s) + (size_t)i * m.V + v0, bytes, &sh.full[st]);
                bulk_load_1d(dst + ROWS_SEG, static_cast<const uint16_t *>(m.t) + (size_t)i * m.V + v0, bytes,
                             &sh.full[st]);
                pending |= 1u << st;
                pend_par = (pend_par & ~(1u << st)) | (ph << st);
            }
            if (*abort) {
                // no copy may still be landing when the CTA leaves
                int dummy = 0;
                for (int st = 0; st < ROWS_STAGES; ++st)
                    if (pending & (1u << st)) mbar_wait(&sh.full[st], (pend_par >> st) & 1, &dummy, 100000000ull);
            }
        }
    } else {
        const int w = warp - 1;
        constexpr uint32_t NEG2 = 0xFF80FF80u;   // two bf16 -inf
        int k = 0;
        for (int it = blockIdx.x; it < items; it += gridDim.x, ++k) {
            const int st = k % ROWS_STAGES;
            const bool got = mbar_wait(&sh.full[st], (uint32_t)((k / ROWS_STAGES) & 1), abort);
            if (rows_bar_or(!got)) break;
            const int i = it / m.nch, ch = it % m.nch;
            const int v0 = ch * TRAIN_ROW_CHUNK, n = min(TRAIN_ROW_CHUNK, m.V - v0);
            const uint4 *ss = reinterpret_cast<const uint4 *>(base + st * 2 * ROWS_SEG);
            const uint4 *tt = ss + ROWS_SEG / 16;
            uint4 ps[8], pt[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const int pc = 32 * w + lane + 256 * c;
                if (8 * pc < n) {
                    ps[c] = ss[pc];
                    pt[c] = tt[pc];
                } else {
                    ps[c] = pt[c] = make_uint4(NEG2, NEG2, NEG2, NEG2);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.empty[st]);
            // the thread's ids increase along (c, word, half): a strict > keeps the first
            const int vt = v0 + 8 * (32 * w + lane);
            float best = -INFINITY, mt = -INFINITY;
            int idx = 0x7fffffff;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint32_t ws[4] = {ps[c].x, ps[c].y, ps[c].z, ps[c].w};
                const uint32_t wt[4] = {pt[c].x, pt[c].y, pt[c].z, pt[c].w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float s0 = __uint_as_float(ws[q] << 16), s1 = __uint_as_float(ws[q] & 0xFFFF0000u);
                    const int v = vt + 2048 * c + 2 * q;
                    if (s0 > best) { best = s0; idx = v; }
                    if (s1 > best) { best = s1; idx = v + 1; }
                    mt = fmaxf(mt, fmaxf(__uint_as_float(wt[q] << 16), __uint_as_float(wt[q] & 0xFFFF0000u)));
                }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float ob = __shfl_xor_sync(0xffffffffu, best, o);
                const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
                mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, o));
                merge_argmax(best, idx, ob, oi);
            }
            // best is now the warp's maximum of s (log2 domain below)
            const float ms2 = best * L2E, mt2 = mt * L2E;
            const bool has_s = best != -INFINITY, has_t = mt != -INFINITY;
            float sa[2] = {0.f, 0.f}, ta[2] = {0.f, 0.f};
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint32_t ws[4] = {ps[c].x, ps[c].y, ps[c].z, ps[c].w};
                const uint32_t wt[4] = {pt[c].x, pt[c].y, pt[c].z, pt[c].w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    if (has_s) {
                        sa[q & 1] += ex2_approx(fmaf(__uint_as_float(ws[q] << 16), L2E, -ms2));
                        sa[q & 1] += ex2_approx(fmaf(__uint_as_float(ws[q] & 0xFFFF0000u), L2E, -ms2));
                    }
                    if (has_t) {
                        ta[q & 1] += ex2_approx(fmaf(__uint_as_float(wt[q] << 16), L2E, -mt2));
                        ta[q & 1] += ex2_approx(fmaf(__uint_as_float(wt[q] & 0xFFFF0000u), L2E, -mt2));
                    }
                }
            }
            float sum_s = sa[0] + sa[1], sum_t = ta[0] + ta[1];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                sum_s += __shfl_xor_sync(0xffffffffu, sum_s, o);
                sum_t += __shfl_xor_sync(0xffffffffu, sum_t, o);
            }
            // the 8 warps' partials (double-buffered by item parity: the
            // merge of item k reads buffer k & 1 before the barrier of
            // item k + 1, the writes of item k + 2 come after it)
            const int pb = k & 1;
            if (lane == 0) {
                sh.wp[pb][w] = make_float4(has_s ? ms2 : -INFINITY, sum_s, has_t ? mt2 : -INFINITY, sum_t);
                sh.wb[pb][w] = best;
                sh.wi[pb][w] = idx;
            }
            asm volatile("bar.sync 1, 256;" ::: "memory");
            if (w == 0 && lane == 0) {
                float4 a = sh.wp[pb][0];
                float b = sh.wb[pb][0];
                int bi = sh.wi[pb][0];
                for (int k2 = 1; k2 < 8; ++k2) {
                    lse2_merge(a.x, a.y, sh.wp[pb][k2].x, sh.wp[pb][k2].y);
                    lse2_merge(a.z, a.w, sh.wp[pb][k2].z, sh.wp[pb][k2].w);
                    merge_argmax(b, bi, sh.wb[pb][k2], sh.wi[pb][k2]);
                }
                m.rpart[(size_t)i * m.nch + ch] = a;
                m.rkey[(size_t)i * m.nch + ch] = argmax_key(b, bi);
            }
        }
    }
    __syncthreads();
    if (threadIdx.x == 0 && sh.abort) set_status(m.status, ST_TIMEOUT);
}

// grid ceil(P / 8), 256 threads: one warp per position.
__global__ void __launch_bounds__(256) k_train_rows_fin(TrainMisc m)
{
    pdl_trigger();
    pdl_wait();
    const int i = blockIdx.x * 8 + threadIdx.x / 32, lane = threadIdx.x % 32;
    if (i >= m.P) return;
    float ms = -INFINITY, ss = 0.f, mt = -INFINITY, st = 0.f;
    unsigned long long key = 0;
    for (int c = lane; c < m.nch; c += 32) {
        const float4 a = m.rpart[(size_t)i * m.nch + c];
        lse2_merge(ms, ss, a.x, a.y);
        lse2_merge(mt, st, a.z, a.w);
        key = max(key, m.rkey[(size_t)i * m.nch + c]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lse2_merge(ms, ss, __shfl_xor_sync(0xffffffffu, ms, o), __shfl_xor_sync(0xffffffffu, ss, o));
        lse2_merge(mt, st, __shfl_xor_sync(0xffffffffu, mt, o), __shfl_xor_sync(0xffffffffu, st, o));
        key = max(key, __shfl_xor_sync(0xffffffffu, key, o));
    }
    if (lane == 0) {
        m.lse_s2[i] = ms + log2f(ss);
        m.lse_q2[i] = mt + log2f(st);
        int y = m.ystar[i];
        if (y < 0 || y >= m.V) {
            set_status(m.status, ST_BOUNDS);
            y = 0;
        }
        m.s_y[i] = bf2f(static_cast<const uint16_t *>(m.s)[(size_t)i * m.V + y]);
        if (m.xhat_in) {
            m.xhat[i] = m.xhat_in[i];
        } else {
            float b;
            int bi;
            argmax_unkey(key, b, bi);
            m.xhat[i] = bi;
        }
    }
}

// grid b * 4 + (NR / 2 - P), r threads: CTA 4 blk + k4 (< 4 b) builds the
// rows of positions k4, k4 + 4, ... of block blk (u_g of the block summed by
// each of its four CTAs), the others zero one padding position each.
__global__ void __launch_bounds__(RANK) k_train_fuse(TrainMisc m)
{
    pdl_trigger();
    pdl_wait();
    const int d = threadIdx.x, r3 = 3 * RANK;
    if ((int)blockIdx.x >= 4 * m.b) {
        // padding rows: zero operands and activations so that every product
        // over them vanishes
        const int i = m.P + (int)blockIdx.x - 4 * m.b;
        for (int f = 0; f < 2; ++f) {
            const int row = pair_row(i, f);
            m.X[(size_t)row * r3 + d] = 0;
            m.X[(size_t)row * r3 + RANK + d] = 0;
            m.X[(size_t)row * r3 + 2 * RANK + d] = 0;
            m.Xlo[(size_t)row * 2 * RANK + d] = 0;
            m.Xlo[(size_t)row * 2 * RANK + RANK + d] = 0;
            m.c[(size_t)row * RANK + d] = 0.f;
            m.cop[(size_t)row * RANK + d] = 0;
            m.dab[(size_t)row * RANK + d] = 0;
            if (d == 0) m.xrow[row] = -1;
        }
        return;
    }
    const int blk = blockIdx.x >> 2, k4 = blockIdx.x & 3, B = m.B;
    // the K-split slices of W_h h and W_g h, summed in a fixed order
    const size_t slice = (size_t)m.P * RANK;
    float ug = 0.f;
    for (int j = 0; j < B; ++j) {
        float uj = 0.f;
#pragma unroll 8
        for (int sp = 0; sp < m.usplits; ++sp) uj += m.Ug[sp * slice + (size_t)(blk * B + j) * RANK + d];
        ug += uj;
    }
    ug /= (float)B;
    const uint16_t ugb = f2bf(ug), ugl = f2bf(ug - bf2f(ugb));
    for (int k = k4; k < B; k += 4) {
        const int i = blk * B + k;
        float uhv = 0.f;
#pragma unroll 8
        for (int sp = 0; sp < m.usplits; ++sp) uhv += m.Uh[sp * slice + (size_t)i * RANK + d];
        const uint16_t uh = f2bf(uhv), uhl = f2bf(uhv - bf2f(uh));
        for (int f = 0; f < 2; ++f) {
            const int row = pair_row(i, f);
            int x = k == 0 ? m.anchor[blk] : (f == 0 ? m.ystar[i - 1] : m.xhat[i - 1]);
            if (x < 0 || x >= m.V) {
                if (d == 0) set_status(m.status, ST_BOUNDS);
                x = 0;
            }
            m.X[(size_t)row * r3 + d] = uh;
            m.X[(size_t)row * r3 + RANK + d] = ugb;
            m.X[(size_t)row * r3 + 2 * RANK + d] = m.W_e[(size_t)x * RANK + d];
            m.Xlo[(size_t)row * 2 * RANK + d] = uhl;
            m.Xlo[(size_t)row * 2 * RANK + RANK + d] = ugl;
            if (d == 0) m.xrow[row] = x;
        }
    }
}

namespace {

// The causal mixer of 32 channels, staged as Ls[(k B + j) 32 + d] (fp32,
// channel innermost); only j < k is read.
__device__ __forceinline__ void stage_L(const TrainMisc &m, float *Ls, int d0)
{
    const int B = m.B, n = 32 * B * B;
    for (int e = threadIdx.y * 32 + threadIdx.x; e < n; e += 32 * B) {
        const int dl = e / (B * B), kj = e % (B * B);
        Ls[kj * 32 + dl] = bf2f(m.L[(size_t)(d0 + dl) * B * B + kj]);
    }
}

constexpr int MIX_SEQ = 2;        // sequences (block, forward) per CTA

inline size_t mix_smem(int B) { return (size_t)(32 * B * B + 2 * B * 32) * 4; }

}  // namespace

size_t train_mix_smem(int B) { return mix_smem(B); }

// grid (r / 32, ceil(2 b / MIX_SEQ)), block (32, B): channel d0 + x, position y
// of the sequences 2 blk + f of the CTA's group: c_k = a_k + sum_{j<k} L_kj a_j.
__global__ void __launch_bounds__(1024) k_train_mix(TrainMisc m)
{
    pdl_trigger();
    extern __shared__ float smf[];
    const int B = m.B, dl = threadIdx.x, k = threadIdx.y, d0 = blockIdx.x * 32, d = d0 + dl;
    float *Ls = smf, *sa = smf + 32 * B * B;
    stage_L(m, Ls, d0);
    pdl_wait();
    for (int q = 0; q < MIX_SEQ; ++q) {
        const int sq = blockIdx.y * MIX_SEQ + q;
        if (sq >= 2 * m.b) break;
        const int blk = sq >> 1, f = sq & 1;
        const int row = pair_row(blk * B + k, f);
        const float ak = m.a[(size_t)row * RANK + d];
        __syncthreads();                           // Ls staged; the previous sequence's sa read
        sa[k * 32 + dl] = ak;
        __syncthreads();
        float acc = ak;
        for (int j = 0; j < k; ++j) acc = fmaf(Ls[(k * B + j) * 32 + dl], sa[j * 32 + dl], acc);
        m.c[(size_t)row * RANK + d] = acc;
        m.cop[(size_t)row * RANK + d] = f2bf(acc);
    }
}

// Same grid: dL/da_j = dc_j + sum_{k>j} L_kj dc_k, and this group's share of
// dL/dL_kj = sum over sequences of dc_k a_j (added atomically into gL).
__global__ void __launch_bounds__(1024) k_train_mix_bwd(TrainMisc m)
{
    pdl_trigger();
    extern __shared__ float smf[];
    const int B = m.B, dl = threadIdx.x, j = threadIdx.y, d0 = blockIdx.x * 32, d = d0 + dl;
    float *Ls = smf, *sdc = smf + 32 * B * B, *sa = sdc + B * 32;
    stage_L(m, Ls, d0);
    pdl_wait();
    float gl[MAX_B];                               // thread (d, k = j) holds dL/dL_kj' for j' < k
    for (int jj = 0; jj < MAX_B; ++jj) gl[jj] = 0.f;
    for (int q = 0; q < MIX_SEQ; ++q) {
        const int sq = blockIdx.y * MIX_SEQ + q;
        if (sq >= 2 * m.b) break;
        const int blk = sq >> 1, f = sq & 1;
        const int row = pair_row(blk * B + j, f);
        const float dcj = m.dc[(size_t)row * RANK + d];
        const float aj = m.a[(size_t)row * RANK + d];
        __syncthreads();
        sdc[j * 32 + dl] = dcj;
        sa[j * 32 + dl] = aj;
        __syncthreads();
        float acc = dcj;
        for (int k = j + 1; k < B; ++k) acc = fmaf(Ls[(k * B + j) * 32 + dl], sdc[k * 32 + dl], acc);
        m.dab[(size_t)row * RANK + d] = f2bf(acc);
#pragma unroll
        for (int jj = 0; jj < MAX_B; ++jj)
            if (jj < j) gl[jj] = fmaf(dcj, sa[jj * 32 + dl], gl[jj]);
    }
#pragma unroll
    for (int jj = 0; jj < MAX_B; ++jj)
        if (jj < j) atomicAdd(m.gL + ((size_t)d * B + j) * B + jj, gl[jj]);
}

// grid NR / 8, 256 threads: one warp per row.  The row's log-sum-exp from the
// split partials, and its logit at y*: s_y* + W_r[y*] . z (the bf16 operands
// of the Read, fp32 accumulation).
__global__ void __launch_bounds__(256) k_train_stats_fin(TrainMisc m)
{
    pdl_trigger();
    pdl_wait();
    const int row = blockIdx.x * 8 + threadIdx.x / 32, lane = threadIdx.x % 32;
    if (row >= m.NR) return;
    const int i = (row >> 7) * 64 + (row & 63);
    if (i >= m.P) {
        if (lane == 0) {
            m.lse_p2[row] = 0.f;
            m.ly[row] = 0.f;
        }
        return;
    }
    float mx = -INFINITY, s = 0.f;
    for (int sv = lane; sv < m.splits; sv += 32) {
        const float4 a = m.part[(size_t)sv * m.NR + row];
        lse2_merge(mx, s, a.x, a.y);
    }
    int y = m.ystar[i];
    if (y < 0 || y >= m.V) y = 0;                 // reported by k_train_rows_fin
    // lane: 8 consecutive elements of the 256
    const uint4 a = reinterpret_cast<const uint4 *>(m.W_r + (size_t)y * RANK)[lane];
    const uint4 b = reinterpret_cast<const uint4 *>(m.zop + (size_t)row * RANK)[lane];
    const uint32_t wa[4] = {a.x, a.y, a.z, a.w}, wb[4] = {b.x, b.y, b.z, b.w};
    float acc = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        acc = fmaf(__uint_as_float(wa[q] << 16), __uint_as_float(wb[q] << 16), acc);
        acc = fmaf(__uint_as_float(wa[q] & 0xFFFF0000u), __uint_as_float(wb[q] & 0xFFFF0000u), acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        acc += __shfl_xor_sync(0xffffffffu, acc, o);
        lse2_merge(mx, s, __shfl_xor_sync(0xffffffffu, mx, o), __shfl_xor_sync(0xffffffffu, s, o));
    }
    if (lane == 0) {
        m.lse_p2[row] = mx + log2f(s);
        m.ly[row] = m.s_y[i] + acc;
    }
}

// grid b, 32 threads: lane k = position k of block blockIdx.x.
__global__ void __launch_bounds__(32) k_train_tv_fin(TrainMisc m)
{
    pdl_trigger();
    pdl_wait();
    const int blk = blockIdx.x, k = threadIdx.x;
    float lr = 0.f, lb = 0.f, lc = 0.f;
    if (k < m.B) {
        const int i = blk * m.B + k;
        const float w = expf(-(float)k / m.gamma);
        float anc = 0.f;
        float lf[2];
        for (int f = 0; f < 2; ++f) {
            const int row = pair_row(i, f);
            float sm = 0.f, lt = 0.f, eq = 0.f;
            for (int sv = 0; sv < m.splits; ++sv) {
                const float4 a = m.part[(size_t)sv * m.NR + row];
                sm += a.x;
                lt += a.y;
                eq += a.z;
                anc += a.w;
            }
            // lt: sum of p where p < q plus half of it where p = q (k_train_tok)
            const float l1 = 2.0f * (1.0f - sm);
            const float S = 1.0f - 2.0f * lt - eq;          // sum_v sgn(p_v - q_v) p_v
            const float ce = m.lse_p2[row] * LN2 - m.ly[row];
            lf[f] = w * (m.a_ce * ce + m.a_l1 * l1);
            // dL/dl_v = cf [a_ce (p_v - [v = y*]) + a_l1 p_v (sgn(p_v - q_v) - S)]
            const float cf = w * (f == 0 ? 1.0f : m.beta);
            RowCoef rc;
            rc.lse_p2 = m.lse_p2[row];
            rc.lse_q2 = m.lse_q2[i];
            rc.Apos = cf * (m.a_ce + m.a_l1 * (1.0f - S));
            rc.Aneg = cf * (m.a_ce - m.a_l1 * (1.0f + S));
            m.coef[row] = rc;
            m.A2[row] = cf * m.a_ce;
        }
        lr = lf[0];
        lc = lf[1];
        const float ceb = m.lse_s2[i] * LN2 - m.s_y[i];
        lb = w * (m.a_ce * ceb + m.a_l1 * 2.0f * (1.0f - anc));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lr += __shfl_xor_sync(0xffffffffu, lr, o);
        lb += __shfl_xor_sync(0xffffffffu, lb, o);
        lc += __shfl_xor_sync(0xffffffffu, lc, o);
    }
    if (k == 0) {
        m.loss[blk * 4 + 0] = lr;
        m.loss[blk * 4 + 1] = lb;
        m.loss[blk * 4 + 2] = lc;
        m.loss[blk * 4 + 3] = lr + m.lambda * lb + m.beta * lc;
    }
}

// grid ceil(NR r / 1024), 256 threads, 4 elements each: dL/dz as the sum of
// the vocabulary splits' slices in a fixed order plus the -A2 [v = y*] term of
// dL/dl (-A2 W_r[y*]), and its bf16 copy; the same term of dL/dW_r,
// -A2 z at row y*, is added into gW_r (atomic: positions share ids).
__global__ void __launch_bounds__(256) k_train_dz(TrainMisc m)
{
    pdl_trigger();
    pdl_wait();
    const size_t e = ((size_t)blockIdx.x * 256 + threadIdx.x) * 4;
    const size_t n = (size_t)m.NR * RANK;
    if (e >= n) return;
    float4 v = *reinterpret_cast<const float4 *>(m.dzp + e);
    for (int sp = 1; sp < m.splits; ++sp) {
        const float4 o = *reinterpret_cast<const float4 *>(m.dzp + sp * n + e);
        v.x += o.x;
        v.y += o.y;
        v.z += o.z;
        v.w += o.w;
    }
    const int row = (int)(e / RANK), d = (int)(e % RANK);
    const float a2 = m.A2[row];
    if (a2 != 0.0f) {
        int y = m.ystar[(row >> 7) * 64 + (row & 63)];
        if (y < 0 || y >= m.V) y = 0;             // reported by k_train_rows_fin
        const uint2 wv = *reinterpret_cast<const uint2 *>(m.W_r + (size_t)y * RANK + d);
        v.x -= a2 * __uint_as_float(wv.x << 16);
        v.y -= a2 * __uint_as_float(wv.x & 0xFFFF0000u);
        v.z -= a2 * __uint_as_float(wv.y << 16);
        v.w -= a2 * __uint_as_float(wv.y & 0xFFFF0000u);
        const uint2 zv = *reinterpret_cast<const uint2 *>(m.zop + (size_t)row * RANK + d);
        float *g = m.gW_r + (size_t)y * RANK + d;
        atomicAdd(g + 0, -a2 * __uint_as_float(zv.x << 16));
        atomicAdd(g + 1, -a2 * __uint_as_float(zv.x & 0xFFFF0000u));
        atomicAdd(g + 2, -a2 * __uint_as_float(zv.y << 16));
        atomicAdd(g + 3, -a2 * __uint_as_float(zv.y & 0xFFFF0000u));
    }
    *reinterpret_cast<float4 *>(m.dz + e) = v;
    *reinterpret_cast<uint2 *>(m.dzb + e) = make_uint2(pack_bf16x2(v.x, v.y), pack_bf16x2(v.z, v.w));
}

// grid ceil(NR 2r / 1024), 256 threads: dL/dt = dL/du sigma'(t), 4 elements each.
__global__ void __launch_bounds__(256) k_train_dact(TrainMisc m)
{
    pdl_trigger();
    pdl_wait();
    const size_t e = ((size_t)blockIdx.x * 256 + threadIdx.x) * 4;
    if (e >= (size_t)m.NR * 2 * RANK) return;
    const float4 du = *reinterpret_cast<const float4 *>(m.du + e);
    const float4 t = *reinterpret_cast<const float4 *>(m.tpre + e);
    *reinterpret_cast<uint2 *>(m.dtb + e) =
        make_uint2(pack_bf16x2(du.x * sigma_prime(m.act, t.x), du.y * sigma_prime(m.act, t.y)),
                   pack_bf16x2(du.z * sigma_prime(m.act, t.z), du.w * sigma_prime(m.act, t.w)));
}

// grid P, r threads.
__global__ void __launch_bounds__(RANK) k_train_fuse_bwd(TrainMisc m)
{
    pdl_trigger();
    pdl_wait();
    const int i = blockIdx.x, d = threadIdx.x, r3 = 3 * RANK;
    const int blk = i / m.B;
    const int rt = pair_row(i, 0), rc = pair_row(i, 1);
    m.D[(size_t)i * 2 * RANK + d] = f2bf(m.dX[(size_t)rt * r3 + d] + m.dX[(size_t)rc * r3 + d]);
    float dug = 0.f;
    for (int jj = 0; jj < m.B; ++jj) {
        const int p = blk * m.B + jj;
        dug += m.dX[(size_t)pair_row(p, 0) * r3 + RANK + d] + m.dX[(size_t)pair_row(p, 1) * r3 + RANK + d];
    }
    m.D[(size_t)i * 2 * RANK + RANK + d] = f2bf(dug / (float)m.B);
    atomicAdd(m.gW_e + (size_t)m.xrow[rt] * RANK + d, m.dX[(size_t)rt * r3 + 2 * RANK + d]);
    atomicAdd(m.gW_e + (size_t)m.xrow[rc] * RANK + d, m.dX[(size_t)rc * r3 + 2 * RANK + d]);
}

}  // namespace xp
