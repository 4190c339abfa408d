// reduce_common.cuh -- the end-of-pass step shared by k_reduce and the fused
// reduce of k_read_tcv: combine the split-vocabulary partials of a token,
// finish the T > 0 draw inside the winning group, apply Algorithm 1's
// stopping rule to a block, and pack the positions of the next pass.
#pragma once

#include "common.cuh"

namespace xp {

__device__ __forceinline__ void bf16x8_to_float(const uint4 &w, float (&x)[8])
{
    const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        x[2 * q] = __uint_as_float(ww[q] << 16);
        x[2 * q + 1] = __uint_as_float(ww[q] & 0xFFFF0000u);
    }
}

struct TokenResult {
    int y;
    float sel, lse;
    int grp;                     // T > 0: the drawn group
};

// Warp-collective: the re-selected token of packed token i (global token id
// tok = seq * B + k).  Combines the S partials in a fixed tree (deterministic);
// T > 0 recomputes l = s + W_r z over the 32 members of the drawn group and
// draws one by Gumbel-max (the second level of the hierarchical draw).
__device__ __forceinline__ Partial ldcg_partial(const Partial *q)
{
    const float4 v = __ldcg(reinterpret_cast<const float4 *>(q));
    return Partial{v.x, __float_as_int(v.y), v.z, v.w};
}

// A Read partial through L2 (a CTA of the persistent kernel may combine
// several passes, so L1 could hold an older copy).
__device__ __forceinline__ RPartial ldcg_rpartial(const RPartial *q)
{
    const float4 a = __ldcg(reinterpret_cast<const float4 *>(q));
    const float4 b = __ldcg(reinterpret_cast<const float4 *>(q) + 1);
    return RPartial{a.x, __float_as_int(a.y), a.z, a.w, __float_as_int(b.x), b.y, 0, 0};
}

// Second half of reduce_token: combines the lane partials `a` of one evaluated
// token across the warp.  T <= 0: the argmax and its logit.  T > 0: the drawn
// group's member draw (taken by the Read when the group became its range's
// best), l_y / T, and log sum exp(l / T).  Warp-collective.
__device__ __forceinline__ TokenResult finish_token(RPartial a, bool sampling)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        RPartial b;
        b.best = __shfl_xor_sync(0xffffffffu, a.best, o);
        b.idx = __shfl_xor_sync(0xffffffffu, a.idx, o);
        b.m = __shfl_xor_sync(0xffffffffu, a.m, o);
        b.s = __shfl_xor_sync(0xffffffffu, a.s, o);
        b.y = __shfl_xor_sync(0xffffffffu, a.y, o);
        b.sel = __shfl_xor_sync(0xffffffffu, a.sel, o);
        merge_rpartial(a, b, sampling);
    }
    TokenResult res;
    if (!sampling) {
        res.y = a.idx;
        res.sel = a.best;
        res.lse = __int_as_float(0x7fc00000);
    } else {
        res.y = a.y;
        res.sel = a.sel;
        res.lse = a.m + logf(a.s);
    }
    res.grp = a.idx;
    return res;
}

// T > 0 member draw of a token whose Read partials carry none (the graph
// path's epilogues leave it out): recompute the 32 logits of the drawn group
// g, l_v = s_v + W_r[v] . z_i, and take the Gumbel-max over its members.
// Warp-collective (lane = member).
__device__ __forceinline__ void draw_in_group(const Params &p, int i, int tok, int g, float invT,
                                              unsigned long long seed, TokenResult &res)
{
    const int lane = threadIdx.x % 32, k = tok % p.B;
    const int v = g * GROUP + lane;
    float x = -INFINITY, score = -INFINITY;
    float acc_bf = 0.0f;
    if (p.dtype) {
        // the warp takes the group's rows one at a time: lane l holds z[8l ..
        // 8l + 7] and the same slice of the row (one coalesced 512-byte row
        // per load), the partial products meet through shuffles
        float z8[8];
        bf16x8_to_float(__ldcg(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.zpack) +
                                                               (size_t)i * RANK) + lane), z8);
        const uint16_t *wr0 = static_cast<const uint16_t *>(p.W_r);
#pragma unroll 1
        for (int r0 = 0; r0 < GROUP; r0 += 8) {
            uint4 w[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int row = g * GROUP + r0 + u;
                w[u] = row < p.V ? __ldg(reinterpret_cast<const uint4 *>(wr0 + (size_t)row * RANK) + lane)
                                 : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                float w8[8];
                bf16x8_to_float(w[u], w8);
                float part = 0.0f;
#pragma unroll
                for (int j = 0; j < 8; ++j) part = fmaf(w8[j], z8[j], part);
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
                if (lane == r0 + u) acc_bf = part;
            }
        }
    }
    if (v < p.V) {
        float acc = acc_bf;
        if (!p.dtype) {
            for (int d = 0; d < RANK; ++d)
                acc = fmaf(ld_any(p.W_r, 0, (size_t)v * RANK + d), ld_any(p.zpack, 0, (size_t)i * RANK + d), acc);
        }
        x = (acc + ld_any(p.s, p.dtype, (size_t)tok * p.V + v)) * invT;
        score = x + gumbel(seed, (uint32_t)v, (uint32_t)k, STREAM_ELEM, p.offset);
    }
    float bs = score;
    int bi = v;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float os = __shfl_xor_sync(0xffffffffu, bs, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        merge_argmax(bs, bi, os, oi);
    }
    res.y = bi;
    res.sel = __shfl_sync(0xffffffffu, x, (bi - g * GROUP) & (GROUP - 1));
}

// Combines the S Read partials of evaluated token i (global id tok).  For
// T > 0 the member of the drawn group comes with the partials when the Read
// drew it, else it is drawn here.  Warp-collective.
__device__ __forceinline__ TokenResult reduce_token(const Params &p, int i, int tok, float invT,
                                                    unsigned long long seed)
{
    const int lane = threadIdx.x % 32;
    const bool sampling = invT > 0.0f;
    RPartial a = rpartial_identity();
    // the lane's partials (ranges lane, lane + 32, ...) requested together
    // (one round for up to 160 ranges)
    constexpr int PER = 5;
    for (int r0 = 0; r0 < p.S; r0 += 32 * PER) {
        RPartial pv[PER];
#pragma unroll
        for (int j = 0; j < PER; ++j) {
            const int r = r0 + lane + 32 * j;
            pv[j] = r < p.S ? ldcg_rpartial(p.part + (size_t)i * p.S + r) : rpartial_identity();
        }
#pragma unroll
        for (int j = 0; j < PER; ++j) merge_rpartial(a, pv[j], sampling);
    }
    TokenResult res = finish_token(a, sampling);
    if (sampling && res.y == 0x7fffffff) draw_in_group(p, i, tok, res.grp, invT, seed, res);
    return res;
}

// Algorithm 1's stopping rule for block s after a pass that evaluated
// positions m+1..B-1: ynew[base + k] / yold[base + k] hold the new and the
// previous token of evaluated position k.  Single thread.
__device__ __forceinline__ SeqState converge_state(const Params &p, const SeqState &st, const int *ynew,
                                                   const int *yold, int base)
{
    const int B = p.B;
    SeqState ns = st;
    ns.iters = st.iters + 1;
    if (p.sequential) {
        // sequential decode: the pass decided position m + 1 from the
        // decided prefix; the block is complete after position B - 1
        ns.m = st.m + 1;
        ns.active = ns.m + 1 < B;
        ns.converged = !ns.active;
        return ns;
    }
    int first = -1;
    for (int k = st.m + 1; k < B; ++k)
        if (ynew[base + k] != yold[base + k]) { first = k; break; }
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
    return ns;
}

// Positions the next pass evaluates for a block in state ns: all after the
// first one the last pass changed (Algorithm 1 with Theorem 1's frontier), or
// the next one of the sequential decode.
__device__ __forceinline__ int eval_count(const Params &p, const SeqState &ns)
{
    return ns.active ? (p.sequential ? 1 : p.B - 1 - ns.m) : 0;
}

__device__ __forceinline__ void converge_block(const Params &p, int s, const SeqState &st, const int *ynew,
                                               const int *yold, int base)
{
    const SeqState ns = converge_state(p, st, ynew, yold, base);
    p.st[s] = ns;
    if (p.iters) p.iters[s] = ns.iters;
    if (p.converged) p.converged[s] = ns.converged;
}

// Warp-collective version of converge + pack for at most 32 blocks whose
// states sit in shared memory (lane q: block q): applies the stopping rule,
// scans the counts, writes the states, the packed token list and the control
// words, and sets the loop condition.  Returns (in every lane) whether another
// pass follows.
__device__ __forceinline__ bool converge_pack_small(const Params &p, const SeqState *st_in, const int *ynew,
                                                    const int *yold, int passes_before,
                                                    cudaGraphConditionalHandle handle)
{
    const int q = threadIdx.x % 32, B = p.B;
    SeqState ns{};
    int c = 0;
    if (q < p.b) {
        const SeqState st = st_in[q];
        ns = st.active ? converge_state(p, st, ynew, yold, st.off - st.m - 1) : st;
        if (st.active) {
            if (p.iters) p.iters[q] = ns.iters;
            if (p.converged) p.converged[q] = ns.converged;
        }
        c = eval_count(p, ns);
    }
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (q >= o) incl += v;
    }
    const int total = __shfl_sync(0xffffffffu, incl, 31);
    if (q < p.b) {
        ns.off = incl - c;
        ns.cnt = c;
        p.st[q] = ns;
        for (int t = 0; t < c; ++t) p.act_tok[ns.off + t] = q * B + ns.m + 1 + t;
    }
    const int passes = passes_before + 1;
    const bool more = total > 0 && passes < p.K_max;
    if (q == 0) {
        p.ctl[CTL_NACT] = total;
        p.ctl[CTL_DONE] = 0;
        p.ctl[CTL_PASS] = passes;
        if (more) p.ctl[CTL_EVAL] += total;
        if (p.use_graph) cudaGraphSetConditional(handle, more ? 1u : 0u);
    }
    return more;
}

// Block-collective (any multiple of 32 threads): packs the positions of the
// next pass (exclusive scan of the per-block counts), updates the control
// words and sets the graph's loop condition.  Call after every block state of
// this pass is final and visible.
__device__ __forceinline__ void pack_next_pass(const Params &p, cudaGraphConditionalHandle handle, int *wsum)
{
    const int B = p.B, warp = threadIdx.x / 32, lane = threadIdx.x % 32, nwarps = blockDim.x / 32;
    int carry = 0;
    // greedy blocks first, then sampling ones: the Read's warps then mostly
    // see one kind of selection
    for (int cls = 0; cls < 2; ++cls)
    for (int q0 = 0; q0 < p.b; q0 += blockDim.x) {
        const int q = q0 + threadIdx.x;
        SeqState ns{};
        int c = 0;
        bool mine = false;
        if (q < p.b) {
            const volatile int *src = reinterpret_cast<const volatile int *>(&p.st[q]);
            ns.active = src[0]; ns.m = src[1]; ns.iters = src[2]; ns.converged = src[3];
            mine = (p.temperature[q] > 0.0f) == (cls == 1);
            c = mine ? eval_count(p, ns) : 0;
        }
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            int w = lane < nwarps ? wsum[lane] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += v;
            }
            wsum[lane] = w;
        }
        __syncthreads();
        const int off = carry + (warp ? wsum[warp - 1] : 0) + incl - c;
        if (q < p.b && mine) {
            ns.off = off;
            ns.cnt = c;
            p.st[q] = ns;
            for (int t = 0; t < c; ++t) p.act_tok[off + t] = q * B + ns.m + 1 + t;
        }
        carry += wsum[nwarps - 1];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        const int passes = p.ctl[CTL_PASS] + 1;
        p.ctl[CTL_NACT] = carry;
        p.ctl[CTL_DONE] = 0;
        p.ctl[CTL_PASS] = passes;
        if (carry > 0 && passes < p.K_max) p.ctl[CTL_EVAL] += carry;
        // no block can take part in more than K_max passes; the cap also bounds
        // the loop should the per-block bookkeeping ever disagree
        if (p.use_graph) cudaGraphSetConditional(handle, (carry > 0 && passes < p.K_max) ? 1u : 0u);
    }
}

}  // namespace xp
