// refine_small.cu -- Algorithm 1 for small batches as one persistent kernel.
//
// Calls that evaluate at most 32 tokens (b * B <= 32) with a bf16 refiner run
// the whole refinement -- the token-independent part of Fuse and Mix (Sec. 4.1,
// hoisted out of the loop because h and g do not change between passes), every
// Jacobi pass of Algorithm 1 and its stopping rule -- in one cooperative launch
// of S + 8 CTAs, at most one per SM, so that no pass pays a kernel launch, a
// graph-node switch or a cold start.
//
//   Read CTAs (blockIdx < S).  Before the first pass they compute, per pair of
//     channels, Pc = (I + L) P with P_k = F_h h_k + F_g g over all of K on
//     tensor cores, F = [W_in[:, 0:r] W_h ; W_in[:, r:2r] W_g] folded once per
//     refiner (Fuse is linear, and F_g g is the block mean of F_g h_k) and
//     stored as bf16 hi + lo terms; with a draft also the first pass's c.
//     For a call without a draft they compute partial argmaxes of s
//     (Algorithm 1's Y^(0)).  In every pass they run Read + Correct +
//     selection (Eq. read / correct, the argmax or the fixed-noise group
//     draw) over a fixed range of vocabulary rows (128-row blocks): W_r rows
//     are the tcgen05 M dimension, the <= 32 tokens N, and a TMA ring of two
//     64 KB blocks (one copy per block) streams W_r, running ahead into the
//     next pass while the Trans CTAs work.
//     Each range leaves one result per token (greedy: an argmax key; T > 0: a
//     partial with the member draw of its best group already taken).
//   Trans CTAs (S .. S + 7).  CTA j owns channels [32 j, 32 j + 32).  In every
//     pass they gather E' rows for the current tokens, mix (Eq. fuse / mix;
//     with blocks of at most 16 positions every Trans CTA forms all of c) and
//     run Trans z = c + W_2 sigma(W_1 c) (Eq. mlp) on tensor cores,
//     exchanging sigma(W_1 c) through L2.  Then each of them combines the Read
//     results, applies Algorithm 1's stopping rule and packs the next pass
//     (the same result in all eight; the first one publishes it), so the next
//     pass starts without another hand-off.
//
// The roles hand work to one another through monotone counters (SmallCtl,
// release / acquire at GPU scope).  Every wait is bounded: a wait that runs
// out records ST_TIMEOUT and sets the stop bit in every counter, so that all
// CTAs leave, each after draining its own copies in flight.
#include "common.cuh"
#include "kernels.h"
#include "mlp_common.cuh"
#include "reduce_common.cuh"
#include "tcv_common.cuh"

namespace xp {

namespace {

// ------------------------------------------------------------- shared memory

constexpr int PC_BUFS_MAX = 5;                 // precompute ring buffers (at most)

struct RsShared {                              // Read CTA, after the W_r stages and z
    uint64_t full[RS_BSTAGES], empty[RS_BSTAGES];   // W_r blocks (64 KB stages)
    uint64_t z_full, z_empty, go;
    uint64_t tfull[TV_NBUF], tempty[TV_NBUF];
    uint64_t drain;
    uint64_t pfull[PC_BUFS_MAX], pempty[PC_BUFS_MAX];   // precompute ring (h and F chunks)
    uint32_t tmem_base;
    int abort;
    int pc_end;                                // the epilogue warps are done with the precompute
    uint32_t pf_early;                         // bytes of the W_r range prefetched during the precompute
    int pass_n, pass_stop;                     // published by the producer with `go`
    int tok[TV_BN], pos[TV_BN];
    float invT[TV_BN];
    unsigned long long seed[TV_BN];
    SelState sel[TV_EPI_WARPS][32];
    float tile[TV_EPI_WARPS][TV_BN][33];       // per-warp transpose: [token][vocabulary row]
    float bestx[TV_EPI_WARPS][GROUP][32];      // T > 0: x of each (warp, token)'s best group, [j][token]
};

// Trans CTA.  With blocks of at most 16 positions every Trans CTA keeps all
// r channels of E' rows, Pc and L (so it forms c itself: no exchange of c);
// with larger blocks only its own 32 channels (c is exchanged).  Dynamic
// shared memory after the head: cop [32][COP_LD] and uop [32][UOP_LD] bf16,
// e [32][CH] and pc [32][CH] fp32, Lp [B(B-1)/2][CH] bf16 (L's strictly
// lower part, channel innermost).
constexpr int FULL_C_MAX_B = 16;
struct TsShared {
    float cown[MAX_B][32];                     // c of the evaluated tokens, own channels (fp32)
    float zhalf[2][MAX_B][32];                 // W_2 u, the two K halves
    int tok[MAX_B];                            // evaluated tokens of the pass (global ids)
    int x[MAX_B];                              // current tokens Y
    int ynew[MAX_B], yold[MAX_B];              // per evaluated token: new / previous token
    int tok2[MAX_B];                           // evaluated tokens of the next pass
    int tpos[MAX_B], tseq[MAX_B];              // per global token id: position k, block s
    SeqState st[MAX_B];                        // per block: Algorithm 1 state
    int anch[MAX_B];                           // per block: anchor token (bounds-checked)
    float invT[MAX_B];                         // per block: 1 / T (0 for greedy)
    int n, n2, go, more;
};

constexpr size_t RS_BYTES = 1024 + TV_STAGES * TV_A_STAGE + TV_Z_BYTES + sizeof(RsShared);
constexpr size_t TS_HEAD = (sizeof(TsShared) + 127) / 128 * 128;
constexpr size_t TS_TAIL_FULL = 2 * 32 * RANK * 4 + RANK * (FULL_C_MAX_B * (FULL_C_MAX_B - 1) / 2) * 2;
constexpr size_t TS_TAIL_OWN = 2 * 32 * 32 * 4 + 32 * (MAX_B * (MAX_B - 1) / 2) * 2;
constexpr size_t TS_BYTES = 1024 + TS_HEAD + 32 * COP_LD * 2 + 32 * UOP_LD * 2 +
                            (TS_TAIL_FULL > TS_TAIL_OWN ? TS_TAIL_FULL : TS_TAIL_OWN);
constexpr size_t SMALL_SMEM = RS_BYTES > TS_BYTES ? RS_BYTES : TS_BYTES;

// ------------------------------------------------------------- signalling

// Records `bits` (if any) and sets the stop bit of every counter.
__device__ __forceinline__ void raise_stop(SmallCtl *c, int bits)
{
    if (bits) atomicOr(reinterpret_cast<int *>(&c->status.v), bits);
    __threadfence();
    atomicOr(&c->pre_done.v, STOP_BIT);
    atomicOr(&c->c_ready.v, STOP_BIT);
    atomicOr(&c->u_ready.v, STOP_BIT);
    atomicOr(&c->z_ready.v, STOP_BIT);
    atomicOr(&c->read_done.v, STOP_BIT);
}

// One thread: waits until *ctr >= target (true).  false once the stop bit is
// set, or after limit_ns of wall time (the caller's bound on waits for other
// CTAs, 2 s by default: the timeout is recorded and every role stops).
// Relaxed polls with a short sleep keep ~150 pollers from crowding the line's
// L2 slice; the fence after the last poll makes it an acquire.
__device__ __forceinline__ bool wait_count(SmallCtl *c, const unsigned *ctr, unsigned target,
                                           unsigned long long limit_ns)
{
    const unsigned long long t0 = globaltimer();
    for (uint32_t it = 0; it < (1u << 26); ++it) {
        const unsigned v = ld_relaxed_gpu(ctr);
        if (v & STOP_BIT) { fence_acq_rel_gpu(); return false; }
        if (v >= target) { fence_acq_rel_gpu(); return true; }
        if (it >= 2) __nanosleep(32);
        if (globaltimer() - t0 > limit_ns) break;
    }
    raise_stop(c, ST_TIMEOUT);
    return false;
}

// wait_count that, while it waits, streams [pf, pf + bytes) into L2 one
// slice every gap_ns: DRAM stays busy without queues deep enough to stall the
// latency-bound accesses of the other role (its first-pass code and operands).
__device__ __forceinline__ bool wait_count_prefetch(SmallCtl *c, const unsigned *ctr, unsigned target, const char *pf,
                                                    uint32_t bytes, uint32_t slice, unsigned gap_ns,
                                                    unsigned long long limit_ns)
{
    const unsigned long long t0 = globaltimer();
    unsigned long long t_next = t0;
    uint32_t done = 0;
    for (uint32_t it = 0; it < (1u << 26); ++it) {
        const unsigned v = ld_relaxed_gpu(ctr);
        if (v & STOP_BIT) { fence_acq_rel_gpu(); return false; }
        if (v >= target) { fence_acq_rel_gpu(); return true; }
        if (done < bytes) {
            const unsigned long long now = globaltimer();
            if (now >= t_next) {
                prefetch_l2_bulk(pf + done, min(slice, bytes - done));
                done += slice;
                t_next = now + gap_ns;
            }
        }
        if (it >= 2) __nanosleep(32);
        if (globaltimer() - t0 > limit_ns) break;
    }
    raise_stop(c, ST_TIMEOUT);
    return false;
}

// One thread per CTA, last action on the control area: the CTA that leaves
// last publishes the call's status and hands the other block to the next call.
__device__ __forceinline__ void leave(const Params &p, SmallCtlArea *a, SmallCtl *c, int par)
{
    __threadfence();
    if (atomicAdd(&c->exit_cnt.v, 1u) == gridDim.x - 1) {
        __threadfence();
        *p.status = (int32_t)__ldcg(reinterpret_cast<const int *>(&c->status.v));
        a->parity.v = (unsigned)(par ^ 1);
    }
}

// ------------------------------------------------------------- precompute
//
// Read CTAs, before the first pass: the token-independent part of Fuse and
// Mix for pairs of channels, unit u -> channels d0 = 2u, d0 + 1 (128 units).
//   U[t][o] = sum_k h[t][k] F[o][k] over all of K for the unit's four rows o
//   (the h slot W_in[:, 0:r] W_h and the g slot W_in[:, r:2r] W_g of both
//   channels), on tensor cores: F as two bf16 terms (hi + lo, so that the
//   products with the bf16 h are exact and only the fp32 sums round);
//   P_k = U_h,k + (1/B) sum_j U_g,j (the g slot is the block mean), and
//   Pc_k = P_k + sum_{j<k} L_kj P_j (Eq. mix, per channel), written to pcx;
//   with a draft also the first pass's c_k = Pc_k + e_k + sum_{j<k} L_kj e_j
//   (e_k = E'[x_{k-1}], Eq. fuse / mix), written to c0x.
// K is streamed through a ring of TMA copies (warp 0 issues them), two per
// chunk of PC_KT 64-wide K tiles: the unit's 8 F rows ([lo][slot h / g]
// [channel], one 5D box of the folded projection) and the NT rows of h (one 3D
// box; rows past N and tiles past H are zero-filled).  Both land as
// [K tile][row][128 bytes] with the 128-byte swizzle: the 16-byte piece j of
// row i of a tile sits at piece j ^ (i & 7).
constexpr int PC_ROWS = 8;
constexpr int PC_KT = SMALL_PC_KT;                            // 64-wide K tiles per chunk
constexpr int PC_KC = 64 * PC_KT;                             // K per chunk (a multiple of 8 warps x 32)
template <int NT>
struct PcShape {
    static constexpr int F_BYTES = PC_KT * PC_ROWS * 128;        // 8 KB
    static constexpr int H_BYTES = PC_KT * NT * 128;             // 16 or 32 KB
    static constexpr int BUF = F_BYTES + H_BYTES;
    static constexpr int BUFS = NT <= 16 ? 5 : 3;
};
static_assert(PcShape<16>::BUFS * PcShape<16>::BUF <= (int)(TV_STAGES * TV_A_STAGE + TV_Z_BYTES), "precompute ring");
static_assert(PcShape<32>::BUFS * PcShape<32>::BUF <= (int)(TV_STAGES * TV_A_STAGE + TV_Z_BYTES), "precompute ring");
static_assert(PcShape<16>::BUFS <= PC_BUFS_MAX && PcShape<32>::BUFS <= PC_BUFS_MAX, "precompute barriers");

__device__ __forceinline__ void tma_load_5d(void *smem_dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1, int c2,
                                            int c3, int c4)
{
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5, %6}], "
        "[%7];" ::"r"(smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(smem_u32(bar))
        : "memory");
}

// Warp 0, one lane: the chunk copies of every unit of this CTA.  tmap_f: the
// folded projection as (64 columns, 2r rows of a slot, slot, term, K tile);
// tmap_h: h as (64 columns, N rows, K tile).
template <int NT>
__device__ __forceinline__ void pc_produce(const Params &p, const CUtensorMap *tmap_f, const CUtensorMap *tmap_h,
                                           uint8_t *ring, RsShared &sh, int r, int S, volatile int *abort)
{
    using Sh = PcShape<NT>;
    const int nchk = (p.H + PC_KC - 1) / PC_KC;
    uint32_t pending = 0, pend_par = 0;
    int ci = 0;
    bool ok = true;
    for (int unit = r; unit < RANK / 2 && ok; unit += S)
        for (int kc = 0; kc < nchk; ++kc, ++ci) {
            const int buf = ci % Sh::BUFS;
            const uint32_t ph = (uint32_t)((ci / Sh::BUFS) & 1);
            if (!mbar_wait(&sh.pempty[buf], ph ^ 1, abort)) { ok = false; break; }
            uint8_t *dst = ring + buf * Sh::BUF;
            mbar_expect_tx(&sh.pfull[buf], (uint32_t)Sh::BUF);
            tma_load_5d(dst, tmap_f, &sh.pfull[buf], 0, 2 * unit, 0, 0, kc * PC_KT);
            tma_load_3d(dst + Sh::F_BYTES, tmap_h, &sh.pfull[buf], 0, 0, kc * PC_KT);
            pending |= 1u << buf;
            pend_par = (pend_par & ~(1u << buf)) | (ph << buf);
        }
    // no copy may still be landing when the ring is reused
    int dummy = 0;
    for (int b2 = 0; b2 < Sh::BUFS; ++b2)
        if (pending & (1u << b2)) mbar_wait(&sh.pfull[b2], (pend_par >> b2) & 1, &dummy, 100000000ull);
}

// The 8 epilogue warps (w = 0..7): per unit, warp w takes the 32-wide K steps
// w, w + 8, ... of every chunk (m16n8k16: A = the unit's F rows, hi in rows
// 0-7 and lo in rows 8-15, B = h, tokens in 8-column tiles).  The 16 K values
// of one product are taken from 32 consecutive ones, the same for A and B, so
// each operand is one 16-byte load per lane (one swizzled piece of a row).
template <int NT>
__device__ __forceinline__ void pc_consume(const Params &p, uint8_t *ring, RsShared &sh, int r, int S, int w,
                                           int lane, volatile int *abort, bool tm, unsigned long long t_start)
{
    using Sh = PcShape<NT>;
    const int H = p.H, N = p.N, B = p.B, V = p.V, nchk = (H + PC_KC - 1) / PC_KC;
    const int g = lane >> 2, tq = lane & 3, et = w * 32 + lane;
    const int TRI = B * (B - 1) / 2;
    float *us = &sh.bestx[0][0][0];                               // U [4][32]: rows (slot, channel)
    float2 *es = reinterpret_cast<float2 *>(us + 4 * 32);         // E' entries of the first pass [32]
    uint32_t *ls = reinterpret_cast<uint32_t *>(es + 32);         // L pairs [B(B-1)/2] (both channels)
    int ci = 0;
    bool ok = true;
    for (int unit = r; unit < RANK / 2; unit += S) {
        const int d0 = 2 * unit;
        // L of the two channels and the first pass's E' entries (latency
        // overlapped with the first chunk's copies)
        for (int q = et; q < TRI; q += 256) ls[q] = __ldg(reinterpret_cast<const uint32_t *>(p.Lpk + (size_t)q * RANK + d0));
        if (p.draft && et < N) {
            const int s = et / B, k = et % B;
            int tk = k == 0 ? p.anchor[s] : p.draft[et - 1];
            if (tk < 0 || tk >= V) tk = 0;                        // reported by the Trans CTAs
            es[et] = __ldg(reinterpret_cast<const float2 *>(p.Ep + (size_t)tk * RANK + d0));
        }
        float acc[NT / 8][4];
#pragma unroll
        for (int nt = 0; nt < NT / 8; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.0f;
        for (int kc = 0; kc < nchk; ++kc, ++ci) {
            const int buf = ci % Sh::BUFS;
            if (ok && !mbar_wait(&sh.pfull[buf], (uint32_t)((ci / Sh::BUFS) & 1), abort)) ok = false;
            if (ok) {
                if (tm && kc == 0) trace_mark(p.trace, 5, t_start);
                const int kl = min(PC_KC, H - kc * PC_KC);
                const uint8_t *fb = ring + buf * Sh::BUF, *hb = fb + Sh::F_BYTES;
                const int mh = g & 3, ml = 4 + (g & 3);             // F rows of the hi and lo terms
#pragma unroll 1
                for (int ks = w; ks * 32 < kl; ks += 8) {
                    const int ko = ks * 32 + 8 * tq;
                    const bool v = ko < kl;
                    const int tile = ko >> 6, pc = (ko >> 3) & 7;
                    const uint4 z4 = make_uint4(0u, 0u, 0u, 0u);
                    const uint8_t *ft = fb + tile * (PC_ROWS * 128);
                    const uint4 ah = v ? *reinterpret_cast<const uint4 *>(ft + mh * 128 + ((pc ^ mh) << 4)) : z4;
                    const uint4 al = v ? *reinterpret_cast<const uint4 *>(ft + ml * 128 + ((pc ^ ml) << 4)) : z4;
                    const uint32_t a0[4] = {ah.x, al.x, ah.y, al.y}, a1[4] = {ah.z, al.z, ah.w, al.w};
                    const uint8_t *ht = hb + tile * (NT * 128) + g * 128 + ((pc ^ g) << 4);
#pragma unroll
                    for (int nt = 0; nt < NT / 8; ++nt) {
                        const uint4 bb = (v && nt * 8 + g < N)
                                             ? *reinterpret_cast<const uint4 *>(ht + nt * 8 * 128)
                                             : z4;
                        mma_bf16_16816(acc[nt], a0, bb.x, bb.y);
                        mma_bf16_16816(acc[nt], a1, bb.z, bb.w);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.pempty[buf]);
        }
        if (tm && unit == r) trace_mark(p.trace, 6, t_start);
        // the 8 warps' sums (row g < 4: hi + lo of row (slot g / 2, channel g % 2))
        if (g < 4)
#pragma unroll
            for (int nt = 0; nt < NT / 8; ++nt) {
                const int t0 = nt * 8 + 2 * tq;
                sh.tile[w][t0][g] = acc[nt][0] + acc[nt][2];
                sh.tile[w][t0 + 1][g] = acc[nt][1] + acc[nt][3];
            }
        tv_epi_bar();
        if (et < 4 * N) {
            const int t = et >> 2, row = et & 3;
            float u = 0.0f;
#pragma unroll
            for (int w2 = 0; w2 < TV_EPI_WARPS; ++w2) u += sh.tile[w2][t][row];
            us[row * 32 + t] = u;
        }
        tv_epi_bar();
        if (ok && et < 2 * N) {
            const int t = et >> 1, ch = et & 1, s = t / B, k = t % B;
            const float *uh = us + ch * 32 + s * B, *ug = us + (2 + ch) * 32 + s * B;
            float gs = 0.0f;
            for (int j = 0; j < B; ++j) gs += ug[j];
            const float gm = gs / (float)B;
            const int lrow = k * (k - 1) / 2;
            float a = uh[k] + gm;
            for (int j = 0; j < k; ++j) {
                const uint32_t lw = ls[lrow + j];
                a = fmaf(__uint_as_float(ch ? (lw & 0xFFFF0000u) : (lw << 16)), uh[j] + gm, a);
            }
            p.pcx[(size_t)t * RANK + d0 + ch] = a;
            if (p.draft) {
                const float2 *eb = es + s * B;
                float m = ch ? eb[k].y : eb[k].x;
                for (int j = 0; j < k; ++j) {
                    const uint32_t lw = ls[lrow + j];
                    m = fmaf(__uint_as_float(ch ? (lw & 0xFFFF0000u) : (lw << 16)), ch ? eb[j].y : eb[j].x, m);
                }
                p.c0x[(size_t)t * RANK + d0 + ch] = a + m;
            }
        }
        tv_epi_bar();                                             // tile, us, es and ls are reused
    }
}

// Partial argmax of s[t, segment] (fp32 compare of the bf16 values, smallest
// id among equal maxima).  One warp.
__device__ __forceinline__ void rowmax_item(const Params &p, int item, int lane)
{
    const int t = item / RMAX_SEG, seg = item % RMAX_SEG, V = p.V;
    const int v0 = (int)((long long)V * seg / RMAX_SEG), v1 = (int)((long long)V * (seg + 1) / RMAX_SEG);
    const uint16_t *row = static_cast<const uint16_t *>(p.s) + (size_t)t * V;
    float best = -INFINITY;
    int idx = 0x7fffffff;
#pragma unroll 4
    for (int v = v0 + lane; v < v1; v += 32) {
        const float x = bf2f(__ldg(row + v));
        if (x > best || (x == best && v < idx)) { best = x; idx = v; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ob = __shfl_xor_sync(0xffffffffu, best, o);
        const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
        if (ob > best || (ob == best && oi < idx)) { best = ob; idx = oi; }
    }
    if (lane == 0) p.rmax[item] = Partial{best, idx, 0.0f, 0.0f};
}

// ------------------------------------------------------------- Read role

__device__ __forceinline__ void read_role(const Params &p, const CUtensorMap *tmap_wrb, const CUtensorMap *tmap_wr32,
                                          const CUtensorMap *tmap_z, const CUtensorMap *tmap_f, const CUtensorMap *tmap_h,
                                          SmallCtl *c,
                          uint8_t *base, unsigned long long t_start)
{
    uint8_t *sA = base;                                    // W_r stages (h slices before the first pass)
    uint8_t *sZ = base + TV_STAGES * TV_A_STAGE;           // z, 4 K-chunks
    RsShared &sh = *reinterpret_cast<RsShared *>(sZ + TV_Z_BYTES);
    const int V = p.V, S = p.S, r = blockIdx.x, N = p.N, B = p.B;
    // vocabulary rows [R0, R1), cut at 32-row granularity so that the ranges
    // differ by at most 32 rows; 128-row blocks, the last one possibly partial
    // (its quarters come by 32-row boxes)
    const int NQ = (V + 31) / 32;
    const int R0 = 32 * (int)((long long)NQ * r / S);
    const int R1 = min(32 * (int)((long long)NQ * (r + 1) / S), V);
    const int nblk = (R1 - R0 + TV_BM - 1) / TV_BM;        // >= 1: S <= V / 128
    const int last_q = (R1 - R0 - (nblk - 1) * TV_BM + 31) / 32;   // quarters of the last block (1..4)
    const int ahead = min(RS_BSTAGES, nblk);               // W_r blocks issued ahead of the pass
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const bool tr = p.trace && r == 0;

    if (threadIdx.x == 0) {
        for (int i = 0; i < RS_BSTAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        mbar_init(&sh.z_full, 1);
        mbar_init(&sh.z_empty, 1);
        mbar_init(&sh.go, 1);
        for (int i = 0; i < TV_NBUF; ++i) { mbar_init(&sh.tfull[i], 1); mbar_init(&sh.tempty[i], 4); }
        mbar_init(&sh.drain, 1);
        for (int i = 0; i < PC_BUFS_MAX; ++i) { mbar_init(&sh.pfull[i], 1); mbar_init(&sh.pempty[i], TV_EPI_WARPS); }
        sh.abort = 0;
        sh.pc_end = 0;
        sh.pf_early = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, TV_TMEM_COLS); tmem_relinquish(); }
    const uint64_t keep = policy_evict_last();
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(tmap_f);
        tma_prefetch_desc(tmap_h);
        tma_prefetch_desc(tmap_wrb);
        tma_prefetch_desc(tmap_z);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;

    // ---- precompute: Pc (and the first pass's c) for this CTA's channel
    // pairs, through a ring in the W_r stages; without a draft also partial
    // argmaxes of s
    if (warp == 0) {
        if (lane == 0) {
            if (N <= 16) pc_produce<16>(p, tmap_f, tmap_h, sA, sh, r, S, abort);
            else pc_produce<32>(p, tmap_f, tmap_h, sA, sh, r, S, abort);
        }
    } else if (warp == 1) {
        // meanwhile the idle MMA thread streams the start of this CTA's W_r
        // range into L2 at a gentle pace (the first pass reads it cold), until
        // the precompute ends
        if (lane == 0) {
            const char *wr = static_cast<const char *>(p.W_r) + (size_t)R0 * RANK * 2;
            const uint32_t total = (uint32_t)(R1 - R0) * RANK * 2, slice = 64 * RANK * 2;
            const unsigned long long t0 = globaltimer();
            unsigned long long t_next = t0;
            uint32_t done = 0;
            while (!*reinterpret_cast<volatile int *>(&sh.pc_end) && done < total) {
                const unsigned long long now = globaltimer();
                if (now >= t_next) {
                    prefetch_l2_bulk(wr + done, min(slice, total - done));
                    done += min(slice, total - done);
                    t_next = now + 1500u;
                }
                if (now - t0 > 100000000ull) break;          // a bound; the precompute takes microseconds
                __nanosleep(200);
            }
            sh.pf_early = done;
        }
    } else if (warp >= 2) {
        const int w = warp - 2;
        const bool tm = tr && w == 0 && lane == 0;
        if (tm) trace_mark(p.trace, 4, t_start);
        if (N <= 16) pc_consume<16>(p, sA, sh, r, S, w, lane, abort, tm, t_start);
        else pc_consume<32>(p, sA, sh, r, S, w, lane, abort, tm, t_start);
        if (w == 0 && lane == 0) *reinterpret_cast<volatile int *>(&sh.pc_end) = 1;
        if (!p.draft)
            for (int item = r * TV_EPI_WARPS + w; item < N * RMAX_SEG; item += S * TV_EPI_WARPS)
                rowmax_item(p, item, lane);
        if (tm) trace_mark(p.trace, 7, t_start);
    }
    __syncthreads();
    // (release: the other threads' writes precede it through the barrier)
    if (threadIdx.x == 0) {
        if (sh.abort) raise_stop(c, ST_TIMEOUT);
        else red_add_release_gpu(&c->pre_done.v, 1u);
        if (tr) trace_mark(p.trace, 2, t_start);
    }

    if (warp == 0) {
        // ------------------------------------------------------- producer
        if (lane == 0) {
            uint32_t pending = 0, pend_par = 0;            // last issue per stage (for the drain)
            bool z_issued = false;
            uint32_t z_par = 0;
            // ci counts W_r blocks over the passes: block ci % nblk of the range
            auto issue = [&](long long ci) -> bool {
                const int stage = (int)(ci % RS_BSTAGES);
                const uint32_t ph = (uint32_t)((ci / RS_BSTAGES) & 1);
                if (!mbar_wait(&sh.empty[stage], ph ^ 1, abort)) return false;
                const int blk = (int)(ci % nblk);
                uint8_t *dst = sA + stage * RS_B_STAGE;
                if (blk == nblk - 1 && last_q < 4) {
                    // partial last block: its quarters only, per K chunk (the
                    // MMA's other rows are stale and the epilogue leaves them out)
                    mbar_expect_tx(&sh.full[stage], (uint32_t)(last_q * TV_KCH) * (TV_A_STAGE / 4));
                    for (int kc = 0; kc < TV_KCH; ++kc)
                        for (int qq = 0; qq < last_q; ++qq)
                            tma_load_2d_hint(dst + kc * TV_A_STAGE + qq * (TV_A_STAGE / 4), tmap_wr32, &sh.full[stage],
                                             kc * TV_BK, R0 + blk * TV_BM + 32 * qq, keep);
                } else {
                    mbar_expect_tx(&sh.full[stage], RS_B_STAGE);
                    tma_load_3d_hint(dst, tmap_wrb, &sh.full[stage], 0, R0 + blk * TV_BM, 0, keep);
                }
                pending |= 1u << stage;
                pend_par = (pend_par & ~(1u << stage)) | (ph << stage);
                return true;
            };
            long long next = 0;
            bool ok = true;
            for (; next < ahead && ok; ++next) ok = issue(next);
            // while the first Trans runs, the rest of this CTA's W_r range
            // (past the chunks the ring holds) goes into L2 a slice at a time
            const int pf_row0 = max(R0 + ahead * TV_BM, R0 + (int)(sh.pf_early / (RANK * 2)));
            const int pf_rows = max(0, R1 - pf_row0);
            const uint32_t pf_bytes = (uint32_t)pf_rows * RANK * 2;
            for (int pass = 0; ok; ++pass) {
                const bool go = pass == 0
                                    ? wait_count_prefetch(c, &c->z_ready.v, 8u, static_cast<const char *>(p.W_r) +
                                                                                   (size_t)pf_row0 * RANK * 2,
                                                          pf_bytes, 64 * RANK * 2, 1000u, p.wait_ns)
                                    : wait_count(c, &c->z_ready.v, (unsigned)(8 * (pass + 1)), p.wait_ns);
                if (go) {
                    fence_proxy_async_global();
                    sh.pass_n = min(__ldcg(p.ctl + CTL_NACT), TV_BN);
                }
                sh.pass_stop = go ? 0 : 1;
                if (p.trace && pass < 2) { const unsigned long long tn = globaltimer_ns(); trace_mark(p.trace, pass ? 201 : 231, tn); }
                mbar_arrive(&sh.go);
                if (!go) break;
                // z of this pass, once the previous pass's MMAs are done with it
                if (pass > 0 && !mbar_wait(&sh.z_empty, (uint32_t)((pass - 1) & 1), abort)) { ok = false; break; }
                mbar_expect_tx(&sh.z_full, TV_Z_BYTES);
                for (int kc = 0; kc < TV_KCH; ++kc) tma_load_2d(sZ + kc * TV_Z_CHUNK, tmap_z, &sh.z_full, kc * TV_BK, 0);
                z_issued = true;
                z_par = (uint32_t)(pass & 1);
                // the rest of this pass, then the first chunks of the next one
                const long long end = (long long)(pass + 1) * nblk + ahead;
                for (; next < end; ++next)
                    if (!issue(next)) { ok = false; break; }
            }
            // no copy may still be landing when the CTA leaves
            int dummy = 0;
            for (int st = 0; st < RS_BSTAGES; ++st)
                if (pending & (1u << st)) mbar_wait(&sh.full[st], (pend_par >> st) & 1, &dummy, 100000000ull);
            if (z_issued) mbar_wait(&sh.z_full, z_par, &dummy, 100000000ull);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            // descriptors formed once, advanced per MMA
            const uint64_t zdesc0 = smem_desc_sw128(smem_u32(sZ));
            const uint64_t adesc0 = smem_desc_sw128(smem_u32(sA));
            for (int pass = 0;; ++pass) {
                if (!mbar_wait(&sh.go, (uint32_t)(pass & 1), abort)) break;
                if (*reinterpret_cast<volatile int *>(&sh.pass_stop)) break;
                if (!mbar_wait(&sh.z_full, (uint32_t)(pass & 1), abort)) break;
                tc_fence_after();
                if (p.trace && pass < 2) { const unsigned long long tn = globaltimer_ns(); trace_mark(p.trace, pass ? 202 : 232, tn); }
                bool ok = true;
                for (int i = 0; i < nblk && ok; ++i) {
                    const int ib = pass * nblk + i, buf = ib % TV_NBUF;
                    if (!mbar_wait(&sh.tempty[buf], (uint32_t)(((ib / TV_NBUF) & 1) ^ 1), abort)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t d = tmem + buf * TV_BN;
                    const long long ci = (long long)pass * nblk + i;
                    const int stage = (int)(ci % RS_BSTAGES);
                    if (!mbar_wait(&sh.full[stage], (uint32_t)((ci / RS_BSTAGES) & 1), abort)) { ok = false; break; }
                    tc_fence_after();
                    const uint64_t ad = smem_desc_advance(adesc0, stage * RS_B_STAGE);
#pragma unroll
                    for (int kc = 0; kc < TV_KCH; ++kc)
#pragma unroll
                        for (int kk = 0; kk < TV_BK / 16; ++kk)
                            tc_mma_bf16(d, smem_desc_advance(ad, kc * TV_A_STAGE + kk * 32),
                                        smem_desc_advance(zdesc0, kc * TV_Z_CHUNK + kk * 32), TV_IDESC, (kc | kk) != 0);
                    tc_commit(&sh.empty[stage]);
                    tc_commit(&sh.tfull[buf]);
                }
                if (!ok) break;
                tc_commit(&sh.z_empty);
                if (p.trace && pass < 2) { const unsigned long long tn = globaltimer_ns(); trace_mark(p.trace, pass ? 203 : 233, tn); }
            }
            tc_commit(&sh.drain);
            int dummy = 0;
            mbar_wait(&sh.drain, 0, &dummy, 100000000ull);
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int ew = warp - 2, q = warp & 3, half = ew >> 2;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        float (*tile)[33] = sh.tile[ew];
        for (int pass = 0;; ++pass) {
            // every epilogue thread takes the same decision (the named
            // barriers below need all 256)
            const bool got = mbar_wait(&sh.go, (uint32_t)(pass & 1), abort);
            if (tv_epi_bar_or(!got || *abort || *reinterpret_cast<volatile int *>(&sh.pass_stop))) break;
            const unsigned long long t_go = globaltimer_ns();
            const int n = *reinterpret_cast<volatile int *>(&sh.pass_n);
            if (ew == 0) {
                const int t = lane;
                int tok = 0, pos = 0;
                float invT = 0.0f;
                unsigned long long seed = 0;
                if (t < n) {
                    tok = __ldcg(p.act_tok + t);
                    const int s = tok / B;
                    pos = tok % B;
                    const float T = p.temperature[s];
                    invT = T > 0.0f ? 1.0f / T : 0.0f;
                    seed = p.seed[s];
                }
                sh.tok[t] = tok;
                sh.pos[t] = pos;
                sh.invT[t] = invT;
                sh.seed[t] = seed;
            }
            tv_epi_bar();
            const int my_tok = sh.tok[lane], my_pos = sh.pos[lane];
            const float my_invT = sh.invT[lane];
            const unsigned long long my_seed = sh.seed[lane];
            const bool tvalid = lane < n;
            const uint16_t *srow = static_cast<const uint16_t *>(p.s) + (size_t)my_tok * V;
            SelState sel;
            sel.init();
            bool ok = true;
            uint4 cur[4], nxt[4];
            if (half < nblk) load_s_group(cur, srow, R0 + half * TV_BM + q * 32, V, tvalid);
            for (int i = half; i < nblk; i += 2) {
                const int ib = pass * nblk + i, buf = ib % TV_NBUF;
                const int v0 = R0 + i * TV_BM + q * 32;
                if (i + 2 < nblk) load_s_group(nxt, srow, R0 + (i + 2) * TV_BM + q * 32, V, tvalid);
                if (!mbar_wait(&sh.tfull[buf], (uint32_t)((ib / TV_NBUF) & 1), abort)) { ok = false; break; }
                tc_fence_after();
                float acc[TV_BN];
                tmem_ld32(tmem + lane_base + buf * TV_BN, acc);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sh.tempty[buf]);
#pragma unroll
                for (int t2 = 0; t2 < TV_BN; ++t2) tile[t2][lane] = acc[t2];
                __syncwarp();
                const int nv = min(GROUP, R1 - v0);                // rows of this CTA's range
                if (tvalid && nv > 0) {
                    float l[GROUP];
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc) {
                        const uint32_t ww[4] = {cur[cc].x, cur[cc].y, cur[cc].z, cur[cc].w};
#pragma unroll
                        for (int e2 = 0; e2 < 4; ++e2) {
                            l[cc * 8 + 2 * e2] = tile[lane][cc * 8 + 2 * e2] + __uint_as_float(ww[e2] << 16);
                            l[cc * 8 + 2 * e2 + 1] =
                                tile[lane][cc * 8 + 2 * e2 + 1] + __uint_as_float(ww[e2] & 0xFFFF0000u);
                        }
                    }
                    if (p.logits) {
                        float *dst = p.logits + (size_t)my_tok * V + v0;
#pragma unroll
                        for (int jj = 0; jj < GROUP; ++jj)
                            if (jj < nv) dst[jj] = l[jj];
                    }
                    const float gz =
                        my_invT > 0.0f ? group_noise(my_seed, (uint32_t)(v0 / GROUP), (uint32_t)my_pos, p.offset) : 0.0f;
                    select_group(sel, l, v0, nv, my_invT, gz, &sh.bestx[ew][0][lane]);
                }
                __syncwarp();
#pragma unroll
                for (int cc = 0; cc < 4; ++cc) cur[cc] = nxt[cc];
            }
            sh.sel[ew][lane] = sel;
            if (p.trace && pass < 2 && lane == 0) { const unsigned long long tn = globaltimer_ns(); trace_mark(p.trace, pass ? 204 : 234, tn); }
            if (tv_epi_bar_or(!ok || *abort)) break;
            // T > 0: the member draw of this range's best group, once per
            // token, its 32 members split over the 8 warps (warp w: members
            // 4w .. 4w + 3, one Philox call); every warp merges the partials
            // of the 8 warps to find that group (the same result in each)
            RPartial a{};
            int wbest = 0;
            const bool draw = tv_epi_bar_or(lane < n && my_invT > 0.0f);
            if (draw && lane < n) {
                a = sh.sel[0][lane].partial();
                for (int w2 = 1; w2 < TV_EPI_WARPS; ++w2) {
                    const RPartial b2 = sh.sel[w2][lane].partial();
                    if (b2.best > a.best || (b2.best == a.best && b2.idx < a.idx)) wbest = w2;
                    merge_rpartial(a, b2, my_invT > 0.0f);
                }
                float bsc = -INFINITY, bx = 0.0f;
                int bj = 0x7fffffff;
                if (my_invT > 0.0f && a.idx != 0x7fffffff) {
                    const int v0 = a.idx * GROUP, valid = min(GROUP, V - v0);
                    const uint4 o = philox10(make_uint4(((uint32_t)v0 >> 2) + ew, (uint32_t)my_pos, STREAM_ELEM, p.offset),
                                             (uint32_t)my_seed, (uint32_t)(my_seed >> 32));
                    const uint32_t w4[4] = {o.x, o.y, o.z, o.w};
#pragma unroll
                    for (int q2 = 0; q2 < 4; ++q2) {
                        const int j = 4 * ew + q2;
                        if (j < valid) {
                            const float u = ((float)(w4[q2] >> 9) + 0.5f) * (1.0f / 8388608.0f);
                            const float xj = sh.bestx[wbest][j][lane];
                            const float sc = xj - logf(-logf(u));
                            if (sc > bsc) { bsc = sc; bj = j; bx = xj; }
                        }
                    }
                }
                tile[0][lane] = bsc;
                tile[1][lane] = __int_as_float(bj);
                tile[2][lane] = bx;
            }
            if (draw) tv_epi_bar();
            if (ew == 0 && lane < n) {
                if (my_invT > 0.0f) {
                    if (a.idx != 0x7fffffff) {
                        // members in order, the first of equal scores
                        float bsc = -INFINITY, bx = 0.0f;
                        int bj = 0;
                        for (int w2 = 0; w2 < TV_EPI_WARPS; ++w2)
                            if (sh.tile[w2][0][lane] > bsc) {
                                bsc = sh.tile[w2][0][lane];
                                bj = __float_as_int(sh.tile[w2][1][lane]);
                                bx = sh.tile[w2][2][lane];
                            }
                        if (bsc == -INFINITY) bx = sh.bestx[wbest][0][lane];
                        a.y = a.idx * GROUP + bj;
                        a.sel = bx;
                    }
                } else {
                    a = sh.sel[0][lane].partial();
                    for (int w2 = 1; w2 < TV_EPI_WARPS; ++w2) merge_rpartial(a, sh.sel[w2][lane].partial(), false);
                }
                if (my_invT > 0.0f) p.part[(size_t)lane * S + r] = a;
                else atomicMax(p.best64 + 32 * (pass & 1) + lane, argmax_key(a.best, a.idx));   // greedy: one key
                // this range's candidate for the token: its E' row into L2 for
                // the next pass's gather (the winner is one of the candidates)
                const int cand = my_invT > 0.0f ? a.y : a.idx;
                if (cand >= 0 && cand < V) prefetch_l2_bulk(p.Ep + (size_t)cand * RANK, RANK * 4);
            }
            tv_epi_bar();
            // partials of this range are written: the Trans CTAs end the pass
            if (ew == 0 && lane == 0) {
                red_add_release_gpu(&c->read_done.v, 1u);
                if (p.trace && pass < 2) { const unsigned long long tn = globaltimer_ns(); trace_mark(p.trace, 205 + pass, tn); }
                if (tr) trace_mark(p.trace, 8 + 4 * pass + 1, t_go);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TV_TMEM_COLS);
    }
    if (threadIdx.x == 0 && sh.abort) raise_stop(c, ST_TIMEOUT);
}

// ------------------------------------------------------------- Trans role

// Fuse, token part: e_j = E'[x_{j-1}] (x_{-1} = the anchor) for every position
// j of every block, channels [cb, cb + CH) (16-byte pieces).
__device__ __forceinline__ void gather_e(const Params &p, const int *x, const int *anch, float *e, int CH, int cb,
                                         int tid, int nth)
{
    const int N = p.N, B = p.B, V = p.V, total = N * CH / 4;
    constexpr int GU = 4;                                      // loads in flight per thread
    for (int i0 = tid; i0 < total; i0 += GU * nth) {
        float4 v[GU];
#pragma unroll
        for (int u = 0; u < GU; ++u) {
            const int i = i0 + u * nth;
            if (i < total) {
                const int j = i / (CH / 4), q = i % (CH / 4), k = j % B, s = j / B;
                int tk = k == 0 ? anch[s] : x[j - 1];
                if (tk < 0 || tk >= V) tk = 0;                 // reported at the start
                v[u] = __ldg(reinterpret_cast<const float4 *>(p.Ep + (size_t)tk * RANK + cb) + q);
            }
        }
#pragma unroll
        for (int u = 0; u < GU; ++u)
            if (i0 + u * nth < total) reinterpret_cast<float4 *>(e)[i0 + u * nth] = v[u];
    }
}

// Mix of one block of B = 16 positions for the channel pair d, d + 1 (full-c
// mode): c_k = Pc_k + e_k + sum_{j<k} L_kj e_j (Eq. fuse / mix) for the
// positions k > m of half KH (dealt ABBA from the last position, so that both
// halves get 60 of the 120 L terms).  Every (k, j) term is a compile-time
// slot: no per-term predicate or index arithmetic.  e and pc point at the
// block's first row; c goes to cop (bf16, row t = off + k - m - 1) and, for
// the CTA's own channels, to cown (fp32).
//
// Not inlined: the Trans CTAs run it once on scratch operands while they wait
// for the precompute, so that its code (about 600 instructions, a cold fetch
// from DRAM after the caches have been flushed) is cached before the first
// pass that mixes.
template <int KH>
__device__ __noinline__ void mix_block16(const float *e, const uint16_t *Lp, const float *pc, uint16_t *cop,
                                         float (*cown)[32], int d, int m, int mlast, int off, int rank)
{
    constexpr int BB = FULL_C_MAX_B;
    float2 er[BB];
#pragma unroll
    for (int j = 0; j < BB; ++j) er[j] = *reinterpret_cast<const float2 *>(e + j * RANK + d);
#pragma unroll
    for (int q = 0; q < BB / 2; ++q) {
        const int k = BB - 1 - ((q >> 1) * 4 + (KH ? 1 + (q & 1) : (q & 1) * 3));
        if (k <= m || k > mlast) continue;
        float2 a0 = er[k], a1 = make_float2(0.0f, 0.0f);
        const uint32_t *lrow = reinterpret_cast<const uint32_t *>(Lp + (k * (k - 1) / 2) * RANK + d);
#pragma unroll
        for (int j = 0; j < k; ++j) {
            const uint32_t lw = lrow[j * (RANK / 2)];
            float2 &a = (j & 1) ? a1 : a0;
            a.x = fmaf(__uint_as_float(lw << 16), er[j].x, a.x);
            a.y = fmaf(__uint_as_float(lw & 0xFFFF0000u), er[j].y, a.y);
        }
        const int t = off + k - m - 1;
        const float2 pcv = *reinterpret_cast<const float2 *>(pc + k * RANK + d);
        const float c0 = pcv.x + (a0.x + a1.x), c1 = pcv.y + (a0.y + a1.y);
        *reinterpret_cast<uint32_t *>(cop + t * COP_LD + d) = (uint32_t)f2bf(c0) | ((uint32_t)f2bf(c1) << 16);
        if ((d >> 5) == rank) *reinterpret_cast<float2 *>(&cown[t][d & 31]) = make_float2(c0, c1);
    }
}

// gather_e issued as asynchronous copies (one commit group; the caller waits
// with cp_async_wait<0> before reading e).
__device__ __forceinline__ void gather_e_async(const Params &p, const int *x, const int *anch, float *e, int CH,
                                               int cb, int tid, int nth, uint64_t policy)
{
    const int N = p.N, B = p.B, V = p.V, total = N * CH / 4;
    for (int i = tid; i < total; i += nth) {
        const int j = i / (CH / 4), q = i % (CH / 4), k = j % B, s = j / B;
        int tk = k == 0 ? anch[s] : x[j - 1];
        if (tk < 0 || tk >= V) tk = 0;                         // reported at the start
        cp_async16(reinterpret_cast<float4 *>(e) + i, reinterpret_cast<const float4 *>(p.Ep + (size_t)tk * RANK + cb) + q,
                   16u, policy);
    }
    cp_async_commit();
}

__device__ __forceinline__ void trans_role(const Params &p, SmallCtl *c, uint8_t *base, unsigned long long t_start)
{
    TsShared &sh = *reinterpret_cast<TsShared *>(base);
    const int rank = blockIdx.x - p.S, d0 = rank * 32;
    const int N = p.N, B = p.B, b = p.b, V = p.V;
    const bool full = B <= FULL_C_MAX_B;                   // this CTA forms all of c
    const int CH = full ? RANK : 32, cb = full ? 0 : d0;   // channels kept, first one
    const int TRI = B * (B - 1) / 2;
    uint16_t *cop = reinterpret_cast<uint16_t *>(base + TS_HEAD);
    uint16_t *uop = cop + 32 * COP_LD;
    float *e = reinterpret_cast<float *>(uop + 32 * UOP_LD);   // [32][CH]
    float *pc = e + 32 * CH;                                   // [32][CH]
    uint16_t *Lp = reinterpret_cast<uint16_t *>(pc + 32 * CH);  // [TRI][CH]
    const int tid = threadIdx.x, nth = blockDim.x, warp = tid / 32, lane = tid % 32;
    const int g = lane >> 2, tq = lane & 3, khalf = (warp >> 2) & 1;
    const bool lead = rank == 0;

    // static operands: W_1 / W_2 fragments and L's strictly lower part for the
    // kept channels (warps 0-7).  Meanwhile warps 8 and 9 run the B = 16 mix
    // once on scratch operands, so that its code (a non-inlined function) is
    // cached before the first pass needs it (cop and cown are rewritten before
    // their first use; e, pc and Lp hold whatever is there).
    MlpFrags fr;
    if (warp < 8) {
        load_mlp_frags(p, rank, fr);
        for (int i = tid; i < TRI * CH / 8; i += 256) {          // 16-byte pieces of the kept channels
            const int q = i / (CH / 8), c8 = i % (CH / 8);
            reinterpret_cast<uint4 *>(Lp)[i] = __ldg(reinterpret_cast<const uint4 *>(p.Lpk + (size_t)q * RANK + cb) + c8);
        }
    } else if (full && B == FULL_C_MAX_B) {
        const int d = 2 * (tid & 127);
        if (warp == 8) mix_block16<0>(e, Lp, pc, cop, sh.cown, d, -1, B - 1, 0, rank);
        else mix_block16<1>(e, Lp, pc, cop, sh.cown, d, -1, B - 1, 0, rank);
    }
    if (tid < N) { sh.tpos[tid] = tid % B; sh.tseq[tid] = tid / B; }
    // Y^(0) from the draft; the lead CTA writes the state of the first pass
    if (tid < N) {
        int y = 0;
        if (p.draft) {
            y = p.draft[tid];
            if (y < 0 || y >= V) {
                if (lead) atomicOr(reinterpret_cast<int *>(&c->status.v), ST_BOUNDS);
                y = 0;
            }
        }
        sh.x[tid] = y;
        sh.tok[tid] = p.sequential ? tid * B : tid;           // the first pass: all positions, or position 0
    }
    const int n0 = p.sequential ? b : N;                       // tokens the first pass evaluates
    if (lead) {
        if (tid < n0) p.act_tok[tid] = p.sequential ? tid * B : tid;
        if (tid < N) {
            if (p.draft) p.tokens[tid] = sh.x[tid];
        }
        if (tid < b) {
            SeqState s{};
            s.active = 1; s.m = -1; s.iters = 0; s.converged = 0;
            s.off = p.sequential ? tid : tid * B; s.cnt = p.sequential ? 1 : B;
            p.st[tid] = s;
            if (p.anchor[tid] < 0 || p.anchor[tid] >= V) atomicOr(reinterpret_cast<int *>(&c->status.v), ST_BOUNDS);
            if (p.iters) p.iters[tid] = 0;
            if (p.converged) p.converged[tid] = 0;
        }
        if (tid == 0) { p.ctl[CTL_NACT] = n0; p.ctl[CTL_DONE] = 0; p.ctl[CTL_PASS] = 0; p.ctl[CTL_EVAL] = n0; }
        if (tid < 64) p.best64[tid] = 0ull;                    // both parities, before pass 0's z
    }
    if (tid < b) {
        SeqState s{};
        s.active = 1; s.m = -1; s.iters = 0; s.converged = 0;
        s.off = p.sequential ? tid : tid * B; s.cnt = p.sequential ? 1 : B;
        sh.st[tid] = s;
        sh.anch[tid] = p.anchor[tid];
        const float T = p.temperature[tid];
        sh.invT[tid] = T > 0.0f ? 1.0f / T : 0.0f;
    }
    if (lead && tid == 0 && p.trace) trace_mark(p.trace, 250, t_start);
    if (tid == 0) sh.go = wait_count(c, &c->pre_done.v, (unsigned)p.S, p.wait_ns);
    __syncthreads();
    if (!sh.go) return;
    if (lead && tid == 0 && p.trace) trace_mark(p.trace, 251, t_start);
    if (!p.draft) {
        // Y^(0) = argmax s (Algorithm 1), from the Read CTAs' partials
        for (int t = warp; t < N; t += nth / 32) {
            const Partial q = ldcg_partial(p.rmax + (size_t)t * RMAX_SEG + lane);
            float best = q.best;
            int idx = q.idx;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float ob = __shfl_xor_sync(0xffffffffu, best, o);
                const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
                if (ob > best || (ob == best && oi < idx)) { best = ob; idx = oi; }
            }
            if (lane == 0) {
                if (idx < 0 || idx >= V) idx = 0;
                sh.x[t] = idx;
                if (lead) p.tokens[t] = idx;
            }
        }
    }
    // Pc = (I + L) P (Eq. mix) of the kept channels, from the Read CTAs
    for (int i = tid; i < N * CH / 4; i += nth) {
        const int t = i / (CH / 4), q = i % (CH / 4);
        reinterpret_cast<float4 *>(pc)[i] = __ldcg(reinterpret_cast<const float4 *>(p.pcx + (size_t)t * RANK + cb) + q);
    }
    __syncthreads();
    if (lead && tid == 0 && p.trace) trace_mark(p.trace, 3, t_start);

    float *zf = p.z_final ? p.z_final : p.zbuf;
    uint16_t *zpack = static_cast<uint16_t *>(p.zpack);
    const uint64_t eprow_policy = policy_evict_first();       // E' rows are read once per pass
    int n = n0;                                                // evaluated tokens of this pass
    for (int pass = 0;; ++pass) {
        const unsigned long long t_pass = globaltimer_ns();
        const int trs = (lead && tid == 0 && p.trace && pass < 3) ? 210 + 8 * pass : 0;
        if (trs) trace_mark(p.trace, trs, t_pass);
        const bool first_c = pass == 0 && p.draft && !p.sequential;   // c formed by the Read CTAs
        if (!first_c) {
            if (pass > 0) cp_async_wait<0>();                  // issued at the end of the previous pass
            else gather_e(p, sh.x, sh.anch, e, CH, cb, tid, nth);
            __syncthreads();
        }
        if (trs) trace_mark(p.trace, trs + 1, t_pass);
        // Mix for the evaluated tokens; c enters W_1 rounded to bf16.
        if (first_c) {
            for (int i = tid; i < n * (RANK / 4); i += nth) {
                const int t = i / (RANK / 4), q = i % (RANK / 4);
                const float4 v = __ldcg(reinterpret_cast<const float4 *>(p.c0x + (size_t)t * RANK) + q);
                *reinterpret_cast<uint2 *>(cop + t * COP_LD + 4 * q) =
                    make_uint2((uint32_t)f2bf(v.x) | ((uint32_t)f2bf(v.y) << 16),
                               (uint32_t)f2bf(v.z) | ((uint32_t)f2bf(v.w) << 16));
                if ((q >> 3) == rank) *reinterpret_cast<float4 *>(&sh.cown[t][4 * (q & 7)]) = v;
            }
            for (int i = tid; i < ((n + 15) / 16 * 16 - n) * RANK; i += nth)
                cop[(n + i / RANK) * COP_LD + i % RANK] = 0;
            __syncthreads();
            if (trs) trace_mark(p.trace, trs + 2, t_pass);
        } else if (full) {
            // thread (channel pair 2 cp, 2 cp + 1; half kh of the positions,
            // dealt ABBA from the last one so that both halves get about the
            // same number of L terms): a block's E' values sit in registers,
            // the j loop is unrolled (B <= 16) with unconditional loads (row
            // k(k-1)/2 + j2 stays inside the 120 rows reserved for Lp) and the
            // terms j2 >= k selected away, and two partial sums per channel
            // shorten the dependency chains
            const int cp = tid & 127, kh = tid >> 7, d = 2 * cp;
            if (B == FULL_C_MAX_B) {
                for (int s = 0; s < b; ++s) {
                    const SeqState st = sh.st[s];
                    if (!st.active) continue;
                    if (kh == 0)
                        mix_block16<0>(e + s * B * CH, Lp, pc + s * B * CH, cop, sh.cown, d, st.m, st.m + st.cnt,
                                       st.off, rank);
                    else if (kh == 1)
                        mix_block16<1>(e + s * B * CH, Lp, pc + s * B * CH, cop, sh.cown, d, st.m, st.m + st.cnt,
                                       st.off, rank);
                }
            } else if (kh < 2)
                for (int s = 0; s < b; ++s) {
                    const SeqState st = sh.st[s];
                    if (!st.active) continue;
                    float2 er[FULL_C_MAX_B];
#pragma unroll
                    for (int j2 = 0; j2 < FULL_C_MAX_B; ++j2)
                        er[j2] = j2 < B ? *reinterpret_cast<const float2 *>(e + (s * B + j2) * CH + d)
                                        : make_float2(0.0f, 0.0f);
#pragma unroll 1
                    for (int k = st.m + 1; k <= st.m + st.cnt; ++k) {
                        if ((((B - 1 - k + 1) >> 1) & 1) != kh) continue;
                        const int t = st.off + k - st.m - 1;
                        float2 a0 = *reinterpret_cast<const float2 *>(e + (s * B + k) * CH + d);
                        float2 a1 = make_float2(0.0f, 0.0f);
                        const uint32_t *lrow = reinterpret_cast<const uint32_t *>(Lp + (k * (k - 1) / 2) * CH + d);
                        uint32_t lw2[FULL_C_MAX_B - 1];
#pragma unroll
                        for (int j2 = 0; j2 < FULL_C_MAX_B - 1; ++j2) lw2[j2] = lrow[j2 * (CH / 2)];
#pragma unroll
                        for (int j2 = 0; j2 < FULL_C_MAX_B - 1; ++j2) {
                                const uint32_t lw = j2 < k ? lw2[j2] : 0u;
                                const float lx = __uint_as_float(lw << 16), ly = __uint_as_float(lw & 0xFFFF0000u);
                                if (j2 & 1) {
                                    a1.x = fmaf(lx, er[j2].x, a1.x);
                                    a1.y = fmaf(ly, er[j2].y, a1.y);
                                } else {
                                    a0.x = fmaf(lx, er[j2].x, a0.x);
                                    a0.y = fmaf(ly, er[j2].y, a0.y);
                                }
                            }
                        const float2 pcv = *reinterpret_cast<const float2 *>(pc + (s * B + k) * CH + d);
                        const float cx0 = pcv.x + (a0.x + a1.x), cx1 = pcv.y + (a0.y + a1.y);
                        *reinterpret_cast<uint32_t *>(cop + t * COP_LD + d) =
                            (uint32_t)f2bf(cx0) | ((uint32_t)f2bf(cx1) << 16);
                        if ((d >> 5) == rank) *reinterpret_cast<float2 *>(&sh.cown[t][d & 31]) = make_float2(cx0, cx1);
                    }
                }
        } else {
            // thread (channel dd of the own 32, token phase t0)
            const int tstep = nth / CH;                        // 10 token phases
            const int dd = tid % CH, t0 = tid / CH;
            if (t0 < tstep)
                for (int t = t0; t < n; t += tstep) {
                    const int tok = sh.tok[t], s = sh.tseq[tok], k = sh.tpos[tok];
                    float a = e[tok * CH + dd];
                    const uint16_t *lrow = Lp + (k * (k - 1) / 2) * CH + dd;
                    const float *erow = e + (s * B) * CH + dd;
                    for (int j2 = 0; j2 < k; ++j2) a = fmaf(bf2f(lrow[j2 * CH]), erow[j2 * CH], a);
                    a = pc[tok * CH + dd] + a;
                    sh.cown[t][dd] = a;
                    p.cx[(size_t)t * RANK + d0 + dd] = f2bf(a);
                }
        }
        if (first_c) {
        } else if (full) {
            // rows past n of the last 16-row tile: zero operands
            for (int i = tid; i < ((n + 15) / 16 * 16 - n) * RANK; i += nth)
                cop[(n + i / RANK) * COP_LD + i % RANK] = 0;
            __syncthreads();
            if (trs) trace_mark(p.trace, trs + 2, t_pass);
        } else {
            __syncthreads();
            if (tid == 0) {
                red_add_release_gpu(&c->c_ready.v, 1u);
                sh.go = wait_count(c, &c->c_ready.v, (unsigned)(8 * (pass + (p.draft && !p.sequential ? 0 : 1))),
                                   p.wait_ns);
                if (trs) trace_mark(p.trace, trs + 2, t_pass);
            }
            __syncthreads();
            if (!sh.go) break;
            for (int i = tid; i < 32 * (RANK / 8); i += nth) {
                const int t = i / (RANK / 8), cc = i % (RANK / 8);
                uint4 v = make_uint4(0, 0, 0, 0);
                if (t < n) v = __ldcg(reinterpret_cast<const uint4 *>(p.cx + (size_t)t * RANK) + cc);
                *reinterpret_cast<uint4 *>(cop + t * COP_LD + 8 * cc) = v;
            }
            __syncthreads();
        }
        // u = sigma(W_1 c), rows [64 rank, +64): warp w -> 8 rows
        if (warp < 8) {
            for (int mt = 0; mt * 16 < n; ++mt) {
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
                const int f = 64 * rank + 8 * warp + 2 * tq;
                const int t0 = mt * 16 + g, t1 = t0 + 8;
                if (t0 < n)
                    *reinterpret_cast<uint32_t *>(p.ux + (size_t)t0 * 2 * RANK + f) =
                        (uint32_t)f2bf(act_fn(p.act, acc[0])) | ((uint32_t)f2bf(act_fn(p.act, acc[1])) << 16);
                if (t1 < n)
                    *reinterpret_cast<uint32_t *>(p.ux + (size_t)t1 * 2 * RANK + f) =
                        (uint32_t)f2bf(act_fn(p.act, acc[2])) | ((uint32_t)f2bf(act_fn(p.act, acc[3])) << 16);
            }
        }
        __syncthreads();
        if (tid == 0) {
            red_add_release_gpu(&c->u_ready.v, 1u);
            sh.go = wait_count(c, &c->u_ready.v, (unsigned)(8 * (pass + 1)), p.wait_ns);
            if (trs) trace_mark(p.trace, trs + 3, t_pass);
        }
        __syncthreads();
        if (!sh.go) break;
        // every Trans CTA has read the previous pass's keys (before its u was
        // published): clear them for the pass after this one (same parity)
        if (lead && pass > 0 && tid < 32) p.best64[32 * ((pass - 1) & 1) + tid] = 0ull;
        {
            // the rows of W_2's 16-row tiles: u of the evaluated tokens, zeros
            // past n; four loads in flight per thread
            const int total = (n + 15) / 16 * 16 * (2 * RANK / 8);
            for (int i0 = tid; i0 < total; i0 += 4 * nth) {
                uint4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int i = i0 + u * nth, t = i / (2 * RANK / 8), cc = i % (2 * RANK / 8);
                    v[u] = make_uint4(0, 0, 0, 0);
                    if (i < total && t < n) v[u] = __ldcg(reinterpret_cast<const uint4 *>(p.ux + (size_t)t * 2 * RANK) + cc);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int i = i0 + u * nth, t = i / (2 * RANK / 8), cc = i % (2 * RANK / 8);
                    if (i < total) *reinterpret_cast<uint4 *>(uop + t * UOP_LD + 8 * cc) = v[u];
                }
            }
        }
        __syncthreads();
        // z = c + W_2 u for channels [32 rank, +32): warp w -> 8 channels, K half w / 4
        if (warp < 8) {
            for (int mt = 0; mt * 16 < n; ++mt) {
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
                const int col = 8 * (warp & 3) + 2 * tq, t0 = mt * 16 + g;
                sh.zhalf[khalf][t0][col] = acc[0];
                sh.zhalf[khalf][t0][col + 1] = acc[1];
                sh.zhalf[khalf][t0 + 8][col] = acc[2];
                sh.zhalf[khalf][t0 + 8][col + 1] = acc[3];
            }
        }
        __syncthreads();
        for (int i = tid; i < n * 32; i += nth) {
            const int t = i / 32, dd = i % 32, tok = sh.tok[t];
            const float z = sh.cown[t][dd] + (sh.zhalf[0][t][dd] + sh.zhalf[1][t][dd]);
            zf[(size_t)tok * RANK + d0 + dd] = z;
            zpack[(size_t)t * RANK + d0 + dd] = f2bf(z);
        }
        __syncthreads();                                       // (the Read CTAs fence before their TMA of z)
        if (tid == 0) {
            red_add_release_gpu(&c->z_ready.v, 1u);
            if (lead && p.trace) trace_mark(p.trace, 8 + 4 * pass, t_pass);
            sh.go = wait_count(c, &c->read_done.v, (unsigned)(p.S * (pass + 1)), p.wait_ns);
        }
        __syncthreads();
        if (!sh.go) break;
        const unsigned long long t_end = globaltimer_ns();
        if (lead && tid == 0 && p.trace && pass < 2) trace_mark(p.trace, 240 + 4 * pass, t_end);
        // ---- end of the pass, in every Trans CTA (identical results; the lead
        // CTA publishes them): combine the Read partials of each evaluated
        // token, apply Algorithm 1's stopping rule, pack the next pass
        if (warp == 0) {
            // greedy tokens: the Read CTAs left one argmax key per token
            const int t = lane;
            if (t < n && sh.invT[sh.tok[t] / B] <= 0.0f) {
                const int tok = sh.tok[t];
                float best;
                int idx;
                argmax_unkey(__ldcg(p.best64 + 32 * (pass & 1) + t), best, idx);
                sh.ynew[t] = idx;
                sh.yold[t] = sh.x[tok];
                if (lead) {
                    if (p.lse) p.lse[tok] = __int_as_float(0x7fc00000);
                    if (p.logit_sel) p.logit_sel[tok] = best;
                    p.tokens[tok] = idx;
                    record_traj(p, tok, pass, idx);
                }
            }
        }
        // T > 0 tokens: warp w combines the partials of tokens w, w + 10, ...
        for (int t = warp; t < n; t += nth / 32) {
            const int tok = sh.tok[t];
            const float invT = sh.invT[tok / B];               // warp-uniform
            if (invT <= 0.0f) continue;
            const TokenResult res = reduce_token(p, t, tok, invT, p.seed[tok / B]);
            if (lane == 0) {
                sh.ynew[t] = res.y;
                sh.yold[t] = sh.x[tok];
                if (lead) {
                    if (p.lse) p.lse[tok] = res.lse;
                    if (p.logit_sel) p.logit_sel[tok] = res.sel;
                    p.tokens[tok] = res.y;
                    record_traj(p, tok, pass, res.y);
                }
            }
        }
        if (lead && lane == 0 && p.trace && pass < 2) trace_mark(p.trace, 240 + 4 * pass + 1, t_end);
        __syncthreads();
        if (lead && tid == 0 && p.trace && pass < 2) trace_mark(p.trace, 240 + 4 * pass + 2, t_end);
        // the new tokens, then the next pass's E' rows in flight while the
        // stopping rule and the packing run
        for (int t = tid; t < n; t += nth) sh.x[sh.tok[t]] = sh.ynew[t];
        __syncthreads();
        gather_e_async(p, sh.x, sh.anch, e, CH, cb, tid, nth, eprow_policy);
        if (warp == 0) {
            // lane q: block q (b <= 32)
            SeqState ns{};
            int cnt = 0;
            if (lane < b) {
                const SeqState st = sh.st[lane];
                ns = st.active ? converge_state(p, st, sh.ynew, sh.yold, st.off - st.m - 1) : st;
                if (st.active && lead) {
                    if (p.iters) p.iters[lane] = ns.iters;
                    if (p.converged) p.converged[lane] = ns.converged;
                }
                cnt = eval_count(p, ns);
            }
            int incl = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += v;
            }
            const int total = __shfl_sync(0xffffffffu, incl, 31);
            if (lane < b) {
                ns.off = incl - cnt;
                ns.cnt = cnt;
                sh.st[lane] = ns;
                for (int q = 0; q < cnt; ++q) sh.tok2[ns.off + q] = lane * B + ns.m + 1 + q;
            }
            if (lane == 0) {
                sh.n2 = total;
                sh.more = total > 0 && pass + 1 < p.K_max;
            }
        }
        __syncthreads();
        if (lead && tid == 0 && p.trace && pass < 2) trace_mark(p.trace, 240 + 4 * pass + 3, t_end);
        n = sh.n2;
        const bool more = sh.more;
        if (tid < n) sh.tok[tid] = sh.tok2[tid];
        if (lead) {
            if (tid < n) p.act_tok[tid] = sh.tok2[tid];
            if (tid == 0) {
                p.ctl[CTL_NACT] = n;
                p.ctl[CTL_PASS] = pass + 1;
                if (more) p.ctl[CTL_EVAL] += n;
            }
        }
        __syncthreads();
        if (lead && tid == 0 && p.trace) trace_mark(p.trace, 8 + 4 * pass + 2, t_end);
        if (!more) {
            cp_async_wait<0>();                                // no copy may land after the CTA leaves
            if (lead && tid == 0) raise_stop(c, 0);            // after the lead's writes
            break;
        }
    }
}

}  // namespace

const size_t kRefineSmallSmemBytes = SMALL_SMEM;

// grid S + 8 (cooperative), TV_THREADS threads, SMALL_SMEM dynamic shared memory,
// one CTA per SM (10 warps: 3 on some of the 4 sub-partitions, hence <= 168
// registers per thread).
__global__ void __launch_bounds__(TV_THREADS, 1)
    k_refine_small(const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tmap_wrb,
                   const __grid_constant__ CUtensorMap tmap_wr32, const __grid_constant__ CUtensorMap tmap_z,
                   const __grid_constant__ CUtensorMap tmap_f, const __grid_constant__ CUtensorMap tmap_h)
{
    const unsigned long long t_start = globaltimer_ns();
    // a kernel launched after this one with programmatic dependent launch may
    // start now (the acceptance's first kernel reads none of our outputs; a
    // dependent must wait with griddepcontrol.wait before reading them)
    pdl_trigger();
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    SmallCtlArea *area = p.sctl;
    const int par = (int)(__ldcg(&area->parity.v) & 1u);
    SmallCtl *c = &area->blk[par];
    if (blockIdx.x == 0 && threadIdx.x < (int)(sizeof(SmallCtl) / sizeof(CtlLine))) {
        // the next call's block (this call's other one) starts from zero
        CtlLine *nxt = reinterpret_cast<CtlLine *>(&area->blk[par ^ 1]);
        nxt[threadIdx.x].v = 0;
    }
    if ((int)blockIdx.x < p.S) read_role(p, &tmap_wrb, &tmap_wr32, &tmap_z, &tmap_f, &tmap_h, c, base, t_start);
    else trans_role(p, c, base, t_start);
    __syncthreads();
    if (threadIdx.x == 0) leave(p, area, c, par);
}

// Folded hidden projection (Fuse is linear): F[o][i] = sum_e W_in[o][e] W_h[e][i]
// for o < r and sum_e W_in[o - r][r + e] W_g[e][i] for o >= r, fp32 accumulation,
// stored as two bf16 terms: Fhl[0] = hi = bf16(F), Fhl[1] = lo = bf16(F - hi)
// (F - hi is exact in fp32; hi + lo is F to about 2^-17 relative).
// grid (ceil(H / 256), 2r / 8), 256 threads.
__global__ void __launch_bounds__(256) k_fold_hidden(const uint16_t *W_h, const uint16_t *W_g, const uint16_t *W_in,
                                                     uint16_t *Fhl, int H)
{
    __shared__ float win[8][RANK];
    const int o0 = blockIdx.y * 8, i = blockIdx.x * 256 + threadIdx.x;
    const bool gpart = o0 >= RANK;
    for (int q = threadIdx.x; q < 8 * RANK; q += 256) {
        const int rr = q / RANK, e = q % RANK, o = o0 + rr;
        win[rr][e] = bf2f(W_in[(size_t)(o % RANK) * 3 * RANK + (gpart ? RANK : 0) + e]);
    }
    __syncthreads();
    if (i >= H) return;
    const uint16_t *W = gpart ? W_g : W_h;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int e = 0; e < RANK; ++e) {
        const float x = bf2f(W[(size_t)e * H + i]);
#pragma unroll
        for (int rr = 0; rr < 8; ++rr) acc[rr] = fmaf(win[rr][e], x, acc[rr]);
    }
#pragma unroll
    for (int rr = 0; rr < 8; ++rr) {
        const uint16_t hi = f2bf(acc[rr]);
        Fhl[(size_t)(o0 + rr) * H + i] = hi;
        Fhl[(size_t)(2 * RANK + o0 + rr) * H + i] = f2bf(acc[rr] - bf2f(hi));
    }
}

// Packs L's strictly lower part channel-innermost: Lpk[k(k-1)/2 + j][d] =
// L[d][k][j] (j < k), so that a warp reading one (k, j) for 32 consecutive
// channels reads 64 contiguous bytes.  grid (ceil(B(B-1)/2 / 8)), 256 threads.
__global__ void __launch_bounds__(256) k_pack_L(const uint16_t *L, uint16_t *Lpk, int B)
{
    const int TRI = B * (B - 1) / 2, d = threadIdx.x;
    for (int q = blockIdx.x * 8; q < min(TRI, blockIdx.x * 8 + 8); ++q) {
        int k = 1;
        while ((k + 1) * k / 2 <= q) ++k;
        const int j = q - k * (k - 1) / 2;
        Lpk[(size_t)q * RANK + d] = L[((size_t)d * B + k) * B + j];
    }
}

}  // namespace xp
