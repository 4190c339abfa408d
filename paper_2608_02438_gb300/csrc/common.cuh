// common.cuh -- device helpers shared by the xPress kernels (sm_103a).
//
// Contents: problem constants, the device parameter block, bf16 conversion,
// Philox4x32-10 (Salmon et al., SC'11) with the counter layout the library
// uses, and thin inline-PTX wrappers for mbarrier, TMA and tcgen05.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace xp {

constexpr int RANK = 256;        // refiner rank r (Sec. 4.1 fixes r = 256)
constexpr int GROUP = 32;        // vocabulary group of the hierarchical Gumbel-max
constexpr int MAX_B = 32;        // largest block the kernels support
constexpr int STREAM_GROUP = 0;  // Philox counter word 2: which draw
constexpr int STREAM_ELEM = 1;
constexpr int STREAM_ACCEPT = 2;
constexpr int STREAM_RESID = 3;

// device status word bits (xpress_get_device_status maps them to xpress_status)
constexpr int ST_TIMEOUT = 1;
constexpr int ST_BOUNDS = 2;

// control block slots (int32, in the workspace)
constexpr int CTL_NACT = 0;     // tokens evaluated by the next pass
constexpr int CTL_DONE = 1;     // last-block-done ticket of the reduce kernel
constexpr int CTL_PASS = 2;     // passes executed so far
constexpr int CTL_ACC_DONE = 3; // ticket of the accept kernels
constexpr int CTL_EVAL = 4;     // tokens evaluated by all passes so far (sum over passes)
constexpr int CTL_WORDS = 8;
constexpr int RMAX_SEG = 32;    // vocabulary segments of the argmax-s scan

struct SeqState {
    int active;     // takes part in the next pass
    int m;          // the next pass evaluates positions k > m (0-based; -1 = all)
    int iters;      // passes executed
    int converged;  // the last pass left the block unchanged
    int off;        // packed index of the first evaluated position in the next pass
    int cnt;        // number of evaluated positions in the next pass
    int pad0, pad1;
};

// One split-vocabulary partial per (vocab range, evaluated token).
// T <= 0: best = max logit, idx = its token id (smallest on ties).
// T  > 0: best = max group score (lse_g + Gumbel), idx = that group,
//         (m, s) = running max and sum of exp(x - m) of x = l / T.
struct Partial {
    float best;
    int idx;
    float m;
    float s;
};

// One split-vocabulary partial of the Read (per vocabulary range and evaluated
// token): Partial's fields plus, for T > 0, the member draw of the range's
// best group -- y (token id) and sel = l_y / T -- taken when that group became
// the range's best, so that combining the ranges needs no second pass over the
// winning group.
struct alignas(16) RPartial {
    float best;
    int idx;
    float m;
    float s;
    int y;
    float sel;
    int pad0, pad1;
};

// Counters through which the CTAs of the persistent small-batch kernel hand
// work to one another (one 128-byte line each).  They only grow during a
// call; STOP_BIT set in a counter tells its waiters to leave.  A call uses one
// of two blocks (named by the area's parity word) and clears the other, which
// the next call uses.
constexpr unsigned STOP_BIT = 1u << 30;
struct alignas(128) CtlLine {
    unsigned v;
    unsigned pad[31];
};
struct SmallCtl {
    CtlLine pre_done;    // Read CTAs done with the precompute (Pc and the first c)
    CtlLine c_ready;     // Trans CTAs that published their slice of c (8 per pass)
    CtlLine u_ready;     // ... of sigma(W_1 c)
    CtlLine z_ready;     // ... of z
    CtlLine read_done;   // Read CTAs done with their partials (S per pass)
    CtlLine exit_cnt;    // CTAs that left (ticket)
    CtlLine status;      // device status bits of the call
};
struct SmallCtlArea {
    CtlLine parity;      // which block the next call uses (flipped by each call's last CTA)
    SmallCtl blk[2];
};

// Everything a call needs on the device; written by the init kernel from the
// by-value copy the host places in the graph's first node.
struct Params {
    int b, B, H, V, N;           // N = b * B
    int dtype, act;              // 0 f32, 1 bf16;  0 SiLU, 1 GELU, 2 ReLU
    int K_max, fixed_K;
    int sequential;              // 1: Theorem 1's sequential decode (pass j evaluates position j only)
    uint32_t offset;
    int S;                       // vocabulary ranges of the Read kernel
    int use_graph;               // 1: the pass loop is a graph WHILE node
    unsigned long long wait_ns;  // persistent kernel: bound on each wait for another CTA (2 s by default)
    unsigned long long *trace;   // optional kernel timeline (profiling), else NULL
    int ksplit;                  // split-K factor of the hidden projection
    // inputs (caller-owned)
    const void *h, *s;
    const int32_t *draft, *anchor;
    const float *temperature;
    const unsigned long long *seed;
    // weights (caller-owned) and derived tensors (refiner-owned)
    const void *W_h, *W_g, *W_in, *L, *W1, *W2, *W_r;
    const float *Ep;             // E' = W_in[:, 2r:3r] W_e, fp32 [V, r]
    // outputs (caller-owned; NULL allowed except tokens)
    int32_t *tokens, *iters, *converged;
    float *lse, *logit_sel, *z_final, *logits;
    int32_t *traj;               // [b, K_max, B] optional: token selected at each evaluated (pass, position)
    // workspace
    int32_t *status;
    int32_t *ctl;
    SeqState *st;
    float *Upart;                // [ksplit, N, 2r] partial sums of h [W_h; W_g]^T (pre_folded: of h F^T,
                                 // F = [W_in[:, 0:r] W_h ; W_in[:, r:2r] W_g])
    int pre_folded;              // Upart holds the folded projection (k_pre_tc)
    float *Pc;                   // [N, r] token-independent part of c after Mix
    int32_t *Ynew;               // [N]
    int32_t *act_tok;            // [N] packed evaluated tokens (global token ids)
    void *zpack;                 // [N, r] W_r operand of the evaluated tokens
    float *zbuf;                 // [N, r] fp32 z when the caller passes no z_final
    float *cbuf;                 // [N, r] fp32 c of the evaluated tokens (graph path, bf16, > 32 tokens)
    uint16_t *ubuf;              // [N, 2r] bf16 sigma(W_1 c) of the evaluated tokens (same)
    RPartial *part;              // [N, S] token-major (a token's ranges are contiguous)
    // persistent small-batch kernel only
    const uint16_t *Fhl;         // [2][2r, H] bf16: hi then lo term of the fp32 rows W_in[:, 0:r] W_h,
                                 // then W_in[:, r:2r] W_g (hi + lo carries about 16 significant bits)
    float *c0x;                  // [32, r] c of the first pass (with a draft), fp32
    uint16_t *cx, *ux;           // [32, r] c and [32, 2r] sigma(W_1 c), bf16, exchanged by the Trans CTAs
    float *pcx;                  // [32, r] Pc = (I + L) P, fp32
    const uint16_t *Lpk;         // [B(B-1)/2, r] bf16: L's strictly lower part, row q = k(k-1)/2 + j
    Partial *rmax;               // [N, RMAX_SEG] argmax-s partials (calls without a draft)
    SmallCtlArea *sctl;          // control blocks of the persistent kernel
    unsigned long long *best64;  // [2][32] per pass parity: max over ranges of argmax_key (greedy tokens)
};

// ------------------------------------------------------------------ numbers

__device__ __forceinline__ float bf2f(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }
__device__ __forceinline__ float round_op(float x, int dtype) { return dtype ? bf2f(f2bf(x)) : x; }

template <typename T> __device__ __forceinline__ float ldf(const T *p, size_t i);
template <> __device__ __forceinline__ float ldf<float>(const float *p, size_t i) { return p[i]; }
template <> __device__ __forceinline__ float ldf<uint16_t>(const uint16_t *p, size_t i) { return bf2f(p[i]); }

__device__ __forceinline__ float ld_any(const void *p, int dtype, size_t i)
{
    return dtype ? bf2f(static_cast<const uint16_t *>(p)[i]) : static_cast<const float *>(p)[i];
}

// Optional trajectory output: the token pass `pass` (0-based) selected for
// global token `tok` (block tok / B, position tok % B).
__device__ __forceinline__ void record_traj(const Params &p, int tok, int pass, int y)
{
    if (p.traj && pass >= 0 && pass < p.K_max) p.traj[((size_t)(tok / p.B) * p.K_max + pass) * p.B + tok % p.B] = y;
}

__device__ __forceinline__ float act_fn(int act, float t)
{
    if (act == 2) return fmaxf(t, 0.0f);
    if (act == 1) return 0.5f * t * (1.0f + erff(t * 0.70710678118654752f));
    return t / (1.0f + expf(-t));
}

// Philox4x32-10, written from its published definition (10 rounds of two
// 32x32->64 multiplies and Weyl key bumps).
__device__ __forceinline__ uint4 philox10(uint4 c, uint32_t k0, uint32_t k1)
{
#pragma unroll
    for (int i = 0; i < 10; ++i) {
        const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
        const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

// Counter layout shared with the CPU oracle: (index >> 2, position, stream,
// offset), output word index & 3; u = ((x >> 9) + 0.5) 2^-23 in (0, 1).
__device__ __forceinline__ float uniform01(unsigned long long seed, uint32_t index, uint32_t pos,
                                           uint32_t stream, uint32_t offset)
{
    const uint4 o = philox10(make_uint4(index >> 2, pos, stream, offset), (uint32_t)seed,
                             (uint32_t)(seed >> 32));
    const uint32_t w = (index & 3u) == 0 ? o.x : (index & 3u) == 1 ? o.y : (index & 3u) == 2 ? o.z : o.w;
    return ((float)(w >> 9) + 0.5f) * (1.0f / 8388608.0f);
}

__device__ __forceinline__ float gumbel(unsigned long long seed, uint32_t index, uint32_t pos, uint32_t stream,
                                        uint32_t offset)
{
    return -logf(-logf(uniform01(seed, index, pos, stream, offset)));
}

__device__ __forceinline__ void set_status(int32_t *status, int bit)
{
    if (status) atomicOr(status, bit);
}

// ---------------------------------------------------- split-vocab combining

// T <= 0 argmax merge: larger value wins, equal values keep the smaller id.
__device__ __forceinline__ void merge_argmax(float &best, int &idx, float ob, int oi)
{
    if (ob > best || (ob == best && oi < idx)) { best = ob; idx = oi; }
}

// log-sum-exp merge of (m, s) pairs, s = sum exp(x - m).
__device__ __forceinline__ void merge_lse(float &m, float &s, float om, float os)
{
    if (om == -INFINITY) return;
    if (m == -INFINITY) { m = om; s = os; return; }
    if (om > m) { s = s * __expf(m - om) + os; m = om; }
    else { s += os * __expf(om - m); }
}

__device__ __forceinline__ void merge_partial(Partial &a, const Partial &b, bool sampling)
{
    merge_argmax(a.best, a.idx, b.best, b.idx);
    if (sampling) merge_lse(a.m, a.s, b.m, b.s);
}

// Greedy selection as one 64-bit key whose unsigned maximum is the argmax with
// the smallest id among equal values: the fp32 value mapped to an
// order-preserving unsigned word (high half), the inverted id (low half).
__device__ __forceinline__ unsigned long long argmax_key(float best, int idx)
{
    const uint32_t b = __float_as_uint(best);
    const uint32_t u = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
    return ((unsigned long long)u << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)idx);
}
__device__ __forceinline__ void argmax_unkey(unsigned long long key, float &best, int &idx)
{
    const uint32_t u = (uint32_t)(key >> 32);
    best = __uint_as_float((u & 0x80000000u) ? (u & 0x7FFFFFFFu) : ~u);
    idx = (int)(0xFFFFFFFFu - (uint32_t)key);
}

// Combining two Read partials: the argmax side carries its member draw.
__device__ __forceinline__ void merge_rpartial(RPartial &a, const RPartial &b, bool sampling)
{
    if (b.best > a.best || (b.best == a.best && b.idx < a.idx)) {
        a.best = b.best; a.idx = b.idx; a.y = b.y; a.sel = b.sel;
    }
    if (sampling) merge_lse(a.m, a.s, b.m, b.s);
}

// Per-token selection state over a run of 32-wide vocabulary groups.
struct SelState {
    float best; int idx; float m; float s;
    int y; float sel;                         // T > 0: member draw of the best group
    __device__ __forceinline__ void init()
    {
        best = -INFINITY; idx = 0x7fffffff; m = -INFINITY; s = 0.0f; y = 0x7fffffff; sel = -INFINITY;
    }
    __device__ __forceinline__ RPartial partial() const { return RPartial{best, idx, m, s, y, sel, 0, 0}; }
};
__device__ __forceinline__ RPartial rpartial_identity()
{
    return RPartial{-INFINITY, 0x7fffffff, -INFINITY, 0.0f, 0x7fffffff, -INFINITY, 0, 0};
}

// The member draw of the hierarchical Gumbel-max inside group [v0, v0 + 32):
// argmax over the members j < valid of x_j + Gumbel(seed, v0 + j, pos,
// STREAM_ELEM, offset), smallest id on ties; one Philox call per 4 ids.  x is
// read as x[XS * j] (XS = 1: a register array; 32: a lane's column in shared
// memory).
template <int XS = 1>
__device__ __forceinline__ void member_draw(const float *x, int valid, int v0, unsigned long long seed, uint32_t pos,
                                            uint32_t offset, int &y, float &sel)
{
    float bsc = -INFINITY, bx = x[0];
    int bj = 0;
#pragma unroll
    for (int c = 0; c < GROUP / 4; ++c) {
        const uint4 o = philox10(make_uint4(((uint32_t)v0 >> 2) + c, pos, STREAM_ELEM, offset), (uint32_t)seed,
                                 (uint32_t)(seed >> 32));
        const uint32_t w4[4] = {o.x, o.y, o.z, o.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int j = 4 * c + q;
            if (j < valid) {
                const float u = ((float)(w4[q] >> 9) + 0.5f) * (1.0f / 8388608.0f);
                const float xj = x[XS * j];
                const float sc = xj - logf(-logf(u));
                if (sc > bsc) { bsc = sc; bj = j; bx = xj; }
            }
        }
    }
    y = v0 + bj;
    sel = bx;
}

// Gumbel noise of the 4 consecutive vocabulary groups 4 g4 .. 4 g4 + 3 of one
// position (stream STREAM_GROUP): one Philox call, word q for group 4 g4 + q
// (the counter layout of uniform01), -log(-log u) with the fast logarithm.
__device__ __forceinline__ void group_noise4(unsigned long long seed, uint32_t g4, uint32_t pos, uint32_t offset,
                                             float (&gn)[4])
{
    const uint4 o = philox10(make_uint4(g4, pos, STREAM_GROUP, offset), (uint32_t)seed, (uint32_t)(seed >> 32));
    const uint32_t w[4] = {o.x, o.y, o.z, o.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) gn[q] = -__logf(-__logf(((float)(w[q] >> 9) + 0.5f) * (1.0f / 8388608.0f)));
}
__device__ __forceinline__ float group_noise(unsigned long long seed, uint32_t g, uint32_t pos, uint32_t offset)
{
    float gn[4];
    group_noise4(seed, g >> 2, pos, offset, gn);
    return gn[g & 3];
}

// 2^x with the hardware approximation (as exp's own fast path uses).
__device__ __forceinline__ float ex2_approx(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <bool FULL>
__device__ __forceinline__ void select_group_impl(SelState &st, const float *l, int v0, int valid, float invT,
                                                  float gnoise, float *xsave)
{
    // four independent chains for the max and the sum, so that few warps
    // still keep the pipes busy
    if (invT <= 0.0f) {
        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int j = 0; j < GROUP; ++j)
            if (FULL || j < valid) m4[j & 3] = fmaxf(m4[j & 3], l[j]);
        const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
        if (mx > st.best) {
            int at = 0;
#pragma unroll
            for (int j = GROUP - 1; j >= 0; --j)
                if ((FULL || j < valid) && l[j] == mx) at = j;
            st.best = mx;
            st.idx = v0 + at;
        }
        return;
    }
    // x = l / T: the max is taken on l (1/T > 0 keeps the order) and
    // exp(x - max x) = 2^(l c - max l c) with c = log2(e) / T, one FMA each
    float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
    for (int j = 0; j < GROUP; ++j)
        if (FULL || j < valid) m4[j & 3] = fmaxf(m4[j & 3], l[j]);
    const float ml = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
    const float cl = invT * 1.4426950408889634f, off2 = -ml * cl;
    float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j = 0; j < GROUP; ++j)
        if (FULL || j < valid) s4[j & 3] += ex2_approx(fmaf(l[j], cl, off2));
    const float sum = (s4[0] + s4[1]) + (s4[2] + s4[3]);
    const float mx = ml * invT;
    const float score = mx + __logf(sum) + gnoise;
    if (score > st.best) {
        st.best = score;
        st.idx = v0 / GROUP;
        if (xsave) {
            // keep the group's x for one member draw at the end of the range
#pragma unroll
            for (int j = 0; j < GROUP; ++j) xsave[32 * j] = l[j] * invT;
        }
    }
    merge_lse(st.m, st.s, mx, sum);
}

// Fold one group of 32 corrected logits l[v0 .. v0+31] (entries j >= valid
// are ignored) into the state.  T <= 0: argmax.  T > 0: x = l * invT, the
// group's log-sum-exp plus its Gumbel noise `gnoise` (group_noise) competes for
// the group draw, and (m, s) accumulate the full log-sum-exp.  xsave (T > 0
// only): when given, the x of the best group so far are stored at xsave[32 j],
// so that the caller can draw the member of the group that ends up best once
// (member_draw).  Without it the partial carries no member and the end of the
// pass draws it (draw_in_group).
__device__ __forceinline__ void select_group(SelState &st, const float *l, int v0, int valid, float invT,
                                             float gnoise, float *xsave = nullptr)
{
    if (valid >= GROUP) select_group_impl<true>(st, l, v0, GROUP, invT, gnoise, xsave);
    else if (valid > 0) select_group_impl<false>(st, l, v0, valid, invT, gnoise, xsave);
}

// ------------------------------------------------------------- PTX wrappers

__device__ __forceinline__ unsigned long long globaltimer_ns()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Optional timeline of a refinement call (enabled by the host for profiling):
// trace[slot] = earliest start, trace[TRACE_SLOTS + slot] = latest end over
// the kernel's blocks (globaltimer, ns).  Slots: 0 init, 1 argmax seed,
// 2 precompute GEMM, 3 precompute Fuse/Mix, 8 + 4 j + {0 Trans, 1 Read,
// 2 reduce} for pass j.
constexpr int TRACE_SLOTS = 256;
__device__ __forceinline__ void trace_mark(unsigned long long *tr, int slot, unsigned long long t0)
{
    if (tr && slot < TRACE_SLOTS) {
        atomicMin(tr + slot, t0);
        atomicMax(tr + TRACE_SLOTS + slot, globaltimer_ns());
    }
}

// Inter-CTA signalling in global memory at GPU scope.
__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned *p)
{
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ unsigned ld_relaxed_gpu(const unsigned *p)
{
    unsigned v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_add_release_gpu(unsigned *p, unsigned v)
{
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned atom_add_acq_rel_gpu(unsigned *p, unsigned v)
{
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}
// Makes a preceding relaxed read an acquire (and later writes ordered after it).
__device__ __forceinline__ void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }
// Orders this thread's generic-proxy global accesses with its later
// async-proxy (TMA) accesses.
__device__ __forceinline__ void fence_proxy_async_global()
{
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Programmatic dependent launch: wait for the preceding kernel of the stream
// (no-op when launched without the attribute) / let the next one start.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// try_wait with a suspend-time hint: the thread sleeps until the phase
// completes or about `hint_ns` pass, instead of spinning on issue slots that
// the other warps of its sub-partition need.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t parity, uint32_t hint_ns)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}

// Bounded wait: gives up after `limit_ns` of wall time or as soon as another
// role raised *abort; returns false then (the caller unwinds).
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort,
                                          unsigned long long limit_ns = 2000000000ull)
{
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
        if ((it & 7u) == 0) {
            if (*abort) return false;
            if (globaltimer() - t0 > limit_ns) { *abort = 1; return false; }
        }
    }
}

__device__ __forceinline__ void fence_barrier_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// Untiled bulk copy global -> shared memory, completing on `bar` (both
// addresses 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_load_1d(void *smem_dst, const void *src, uint32_t bytes, uint64_t *bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_u32(smem_dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tma_load_2d(void *smem_dst, const CUtensorMap *map, uint64_t *bar, int x, int y)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_u32(smem_dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

// Same, with an L2 cache policy (e.g. keep the readout weights resident
// across the passes of one call).
__device__ __forceinline__ void tma_load_2d_hint(void *smem_dst, const CUtensorMap *map, uint64_t *bar, int x, int y,
                                                 uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
        "%3}], [%4], %5;" ::"r"(smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}

// Bulk prefetch of [addr, addr + bytes) into L2 (16-byte aligned, multiple of 16).
__device__ __forceinline__ void prefetch_l2_bulk(const void *addr, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(addr), "r"(bytes) : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_first()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

// Same as prefetch_l2_bulk, with an L2 cache policy.
__device__ __forceinline__ void prefetch_l2_bulk_hint(const void *addr, uint32_t bytes, uint64_t policy)
{
    asm volatile("cp.async.bulk.prefetch.L2.global.L2::cache_hint [%0], %1, %2;" ::"l"(addr), "r"(bytes), "l"(policy)
                 : "memory");
}

// 16-byte asynchronous copy global -> shared (L2 only; bytes < 16 zero-fill
// the rest) with an L2 cache policy, and its commit / wait groups.
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gsrc, uint32_t bytes, uint64_t policy)
{
    asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2, %3;" ::"r"(smem_u32(smem_dst)),
                 "l"(gsrc), "r"(bytes), "l"(policy)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N> __device__ __forceinline__ void cp_async_wait()
{
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_last()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap *map)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// tcgen05 (5th-generation tensor core, accumulators in tensor memory)
__device__ __forceinline__ void tmem_alloc(uint32_t *dst_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulate)
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive on `bar` once every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void tc_commit(uint64_t *bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_u32(bar))
                 : "memory");
}

// 32 lanes x 32 consecutive fp32 columns; thread t gets lane (base + t).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]),
          "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),
          "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor for a K-major operand stored with the
// 128-byte swizzle (rows of 64 bf16 at a 128-byte pitch, 8-row groups 1024
// bytes apart): start address, leading offset 16 B, stride offset 1024 B,
// descriptor version 1, layout type 2 (SWIZZLE_128B).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr)
{
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, N >> 3 at bit 17, M >> 4 at bit 24.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

}  // namespace xp
