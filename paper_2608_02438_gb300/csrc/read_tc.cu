// read_tc.cu -- Read + Correct + selection on the 5th-generation tensor cores.
//
// Computes, for every evaluated token z_k (the W_r operand, bf16) and every
// vocabulary id v,  l_k,v = s_k,v + (W_r z_k)_v  (Sec. 4.1, Eq. read and
// Eq. correct) and folds it straight into the token's selection state
// (Algorithm 1's argmax at T = 0, the group draw of the hierarchical
// Gumbel-max at T > 0).  The logits never travel to HBM.
//
// GEMM view: D[token, v] = z[token, :] . W_r[v, :], M = tokens (128 per tile),
// N = vocabulary (256 per tile), K = r = 256.  Tokens sit in TMEM lanes so that
// each epilogue thread owns one token and reduces over vocabulary columns
// without any cross-thread traffic.
//
// Roles (576 threads, one CTA per SM, persistent over a contiguous vocabulary
// range):
//   warp 0      TMA producer: the token tile (A, kept for the whole range) and
//               a 2-stage ring of W_r K-chunks (B, 32 KB each)
//   warp 1      TMEM allocator and tcgen05.mma issuer (one thread)
//   warps 2-17  epilogue: tcgen05.ld 32 columns, add s (a 2-slot cp.async ring
//               per thread), select_group; 4 warps per SM sub-partition, so
//               that the dependent chains of the fold are hidden
// Two TMEM accumulators of 256 columns let the MMA of tile t+1 overlap the
// epilogue of tile t.  The 4 warps of a TMEM lane quarter split the 8 groups of
// a tile.  With <= 32 evaluated tokens the 32 token rows are replicated into
// all four TMEM lane quarters, and warps 0-7 of the epilogue take one 32-id
// group each (the others only hand the accumulators back).
#include "common.cuh"
#include "kernels.h"

namespace xp {

constexpr int TC_BM = 128;
constexpr int TC_BN = 256;
constexpr int TC_BK = 64;                     // one 128-byte swizzle row of bf16
constexpr int TC_KCH = RANK / TC_BK;          // 4 K-chunks
constexpr int TC_STAGES = 2;                  // W_r stays in L2 (evict_last): 2 stages in flight suffice
constexpr int TC_SPF = 2;                     // s groups in flight per epilogue thread (cp.async ring)
constexpr int TC_EPI_WARPS = 16;                // 4 per SM sub-partition (latency hiding)
constexpr int TC_WPQ = TC_EPI_WARPS / 4;       // epilogue warps per TMEM lane quarter
constexpr int TC_THREADS = 32 * (2 + TC_EPI_WARPS);
constexpr uint32_t TC_A_CHUNK = TC_BM * TC_BK * 2;       // 16 KB
constexpr uint32_t TC_A_BYTES = TC_A_CHUNK * TC_KCH;      // 64 KB
constexpr uint32_t TC_B_STAGE = TC_BN * TC_BK * 2;       // 32 KB
constexpr uint32_t TC_TMEM_COLS = 2 * TC_BN;              // two accumulators
constexpr uint32_t TC_IDESC = idesc_bf16(TC_BM, TC_BN);

struct TcShared {
    uint64_t full[TC_STAGES];
    uint64_t empty[TC_STAGES];
    uint64_t a_full, a_empty;
    uint64_t tfull[2], tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    SelState st[TC_EPI_WARPS][32];
};

constexpr uint32_t TC_S_BYTES = TC_SPF * 4 * (TC_EPI_WARPS * 32) * 16;   // [slot][chunk][thread] 16 B
constexpr size_t TC_SMEM_BYTES = 1024 + TC_A_BYTES + TC_STAGES * TC_B_STAGE + TC_S_BYTES + sizeof(TcShared);
const size_t kReadTcSmemBytes = TC_SMEM_BYTES;
const int kReadTcThreads = TC_THREADS;

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, %0;" ::"n"(TC_EPI_WARPS * 32) : "memory"); }

// Named barrier over the 8 epilogue warps that also ORs a predicate, so that
// every epilogue warp takes the same decision to stop after an abort.
__device__ __forceinline__ bool epi_bar_or(bool pred)
{
    uint32_t res;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, %2, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(res)
        : "r"((uint32_t)pred), "n"(TC_EPI_WARPS * 32)
        : "memory");
    return res != 0;
}

// s[v0 .. v0 + 31] of one token as raw bf16 pairs (zeros past V or for an
// invalid thread); streaming loads (s is read once, evict it first).
__device__ __forceinline__ void load_s_group(uint4 (&r)[4], const uint16_t *row, int v0, int V, bool valid)
{
    if (valid && v0 + GROUP <= V) {
        const uint4 *src = reinterpret_cast<const uint4 *>(row + v0);
#pragma unroll
        for (int c = 0; c < 4; ++c) r[c] = __ldcs(src + c);
        return;
    }
    uint32_t w[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        const int j = v0 + 2 * q;
        const uint32_t lo = (valid && j < V) ? row[j] : 0u;
        const uint32_t hi = (valid && j + 1 < V) ? row[j + 1] : 0u;
        w[q] = lo | (hi << 16);
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) r[c] = make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
}

__global__ void __launch_bounds__(TC_THREADS, 1)
    k_read_tc(const Params *__restrict__ pp, const __grid_constant__ CUtensorMap tmap_wr,
              const __grid_constant__ CUtensorMap tmap_z, int V)
{
    const unsigned long long t_start = globaltimer_ns();
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = base;
    uint8_t *sB = base + TC_A_BYTES;
    uint4 *sS = reinterpret_cast<uint4 *>(sB + TC_STAGES * TC_B_STAGE);   // epilogue s ring
    TcShared &sh = *reinterpret_cast<TcShared *>(sB + TC_STAGES * TC_B_STAGE + TC_S_BYTES);
    const Params &p = *pp;
    const int NVT = (V + TC_BN - 1) / TC_BN;
    const int S = gridDim.x, r = blockIdx.x;
    const int vt0 = (int)((long long)NVT * r / S), vt1 = (int)((long long)NVT * (r + 1) / S);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < TC_STAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        mbar_init(&sh.a_full, 1);
        mbar_init(&sh.a_empty, 1);
        for (int i = 0; i < 2; ++i) { mbar_init(&sh.tfull[i], 1); mbar_init(&sh.tempty[i], TC_EPI_WARPS); }
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, TC_TMEM_COLS); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;

    // W_r does not depend on the previous kernel: start streaming the first
    // stages before waiting for it (programmatic dependent launch)
    const int pre = min(TC_STAGES, (vt1 - vt0) * TC_KCH);
    const uint64_t keep = policy_evict_last();   // W_r is re-read by every pass of the call
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_wr);
        tma_prefetch_desc(&tmap_z);
        // the rest of this CTA's rows of W_r (contiguous: 512 bytes a row) go to
        // L2 now, so that they stream while the previous kernel finishes
        const uint32_t row_bytes = RANK * 2;
        const char *wr = static_cast<const char *>(p.W_r);
        for (int vt = vt0; vt < vt1; ++vt) {
            const int rows = min(TC_BN, V - vt * TC_BN);
            for (int r0 = 0; r0 < rows; r0 += 64)
                prefetch_l2_bulk(wr + (size_t)(vt * TC_BN + r0) * row_bytes, (uint32_t)min(64, rows - r0) * row_bytes);
        }
        for (int i = 0; i < pre; ++i) {
            mbar_expect_tx(&sh.full[i], TC_B_STAGE);
            tma_load_2d_hint(sB + i * TC_B_STAGE, &tmap_wr, &sh.full[i], (i % TC_KCH) * TC_BK,
                             (vt0 + i / TC_KCH) * TC_BN, keep);
        }
    }
    pdl_wait();
    const unsigned long long t_wait = globaltimer_ns();
    const int n = p.ctl[CTL_NACT];
    const bool tr0 = p.trace && p.ctl[CTL_PASS] == 0;   // phase marks of the first pass
    const bool small = n <= 32;
    const int MT = n == 0 ? 0 : (small ? 1 : (n + TC_BM - 1) / TC_BM);
    if (n == 0 && warp == 0 && lane == 0) {
        // nothing to evaluate: let the early copies land before tearing down
        int dummy = 0;
        for (int i = 0; i < pre; ++i) mbar_wait(&sh.full[i], 0, &dummy, 10000000ull);
    }

    if (warp == 0) {
        // ------------------------------------------------------- producer
        if (lane == 0) {
            int stage = 0, skip = pre;
            uint32_t phase = 0, pending = 0, pend_par = 0;
            for (int i = 0; i < pre; ++i) pending |= 1u << i;
            for (int j = 0; j < MT && !*abort; ++j) {
                if (!mbar_wait(&sh.a_empty, (j & 1) ^ 1, abort)) break;
                mbar_expect_tx(&sh.a_full, TC_A_BYTES);
                for (int kc = 0; kc < TC_KCH; ++kc)
                    for (int q = 0; q < 4; ++q)
                        tma_load_2d(sA + kc * TC_A_CHUNK + q * 4096, &tmap_z, &sh.a_full, kc * TC_BK,
                                    small ? 0 : j * TC_BM + 32 * q);
                for (int vt = vt0; vt < vt1 && !*abort; ++vt)
                    for (int kc = 0; kc < TC_KCH; ++kc) {
                        if (skip > 0) {       // issued before the dependency wait
                            --skip;
                            if (++stage == TC_STAGES) { stage = 0; phase ^= 1; }
                            continue;
                        }
                        if (!mbar_wait(&sh.empty[stage], phase ^ 1, abort)) break;
                        mbar_expect_tx(&sh.full[stage], TC_B_STAGE);
                        tma_load_2d_hint(sB + stage * TC_B_STAGE, &tmap_wr, &sh.full[stage], kc * TC_BK,
                                         vt * TC_BN, keep);
                        pending |= 1u << stage;
                        pend_par = (pend_par & ~(1u << stage)) | (phase << stage);
                        if (++stage == TC_STAGES) { stage = 0; phase ^= 1; }
                    }
            }
            if (*abort) {
                // let the copies already issued land before the CTA goes away
                for (int st = 0; st < TC_STAGES; ++st)
                    if (pending & (1u << st)) {
                        int dummy = 0;
                        mbar_wait(&sh.full[st], (pend_par >> st) & 1, &dummy, 10000000ull);
                    }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            int stage = 0, t = 0;
            uint32_t phase = 0;
            for (int j = 0; j < MT && !*abort; ++j) {
                if (!mbar_wait(&sh.a_full, j & 1, abort)) break;
                tc_fence_after();
                if (tr0 && j == 0) trace_mark(p.trace, 201, t_wait);
                const uint32_t a0 = smem_u32(sA);
                for (int vt = vt0; vt < vt1 && !*abort; ++vt, ++t) {
                    const int buf = t & 1;
                    if (!mbar_wait(&sh.tempty[buf], ((t >> 1) & 1) ^ 1, abort)) break;
                    tc_fence_after();
                    const uint32_t d = tmem + buf * TC_BN;
                    for (int kc = 0; kc < TC_KCH; ++kc) {
                        if (!mbar_wait(&sh.full[stage], phase, abort)) break;
                        tc_fence_after();
                        const uint32_t b0 = smem_u32(sB + stage * TC_B_STAGE);
#pragma unroll
                        for (int kk = 0; kk < TC_BK / 16; ++kk)
                            tc_mma_bf16(d, smem_desc_sw128(a0 + kc * TC_A_CHUNK + kk * 32),
                                        smem_desc_sw128(b0 + kk * 32), TC_IDESC, (kc | kk) != 0);
                        tc_commit(&sh.empty[stage]);
                        if (++stage == TC_STAGES) { stage = 0; phase ^= 1; }
                    }
                    tc_commit(&sh.tfull[buf]);
                }
                tc_commit(&sh.a_empty);
            }
            // every MMA issued above has finished before the CTA tears down
            tc_commit(&sh.drain);
            int dummy = 0;
            mbar_wait(&sh.drain, 0, &dummy, 100000000ull);
            if (tr0) trace_mark(p.trace, 202, t_wait);
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int ew = warp - 2;
        const int q = warp & 3;              // TMEM lane quarter this warp may access
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        // large: the TC_WPQ warps of a lane quarter split the 8 groups of a
        // tile; small (<= 32 tokens, replicated in every quarter): warp ew < 8
        // takes group ew, the others only hand the accumulators back
        const int g_first = small ? (ew & 7) : (ew >> 2) * (8 / TC_WPQ);
        const int g_count = small ? (ew < 8 ? 1 : 0) : 8 / TC_WPQ;
        int t = 0;
        for (int j = 0; j < MT; ++j) {
            bool ok = true;
            const int slot = small ? lane : q * 32 + lane;
            const int i = small ? lane : j * TC_BM + slot;
            const bool valid = i < n;
            int tok = 0, pos = 0, seq = 0;
            float invT = 0.0f;
            unsigned long long seed = 0;
            if (valid) {
                tok = p.act_tok[i];
                seq = tok / p.B;
                pos = tok % p.B;
                const float T = p.temperature[seq];
                invT = T > 0.0f ? 1.0f / T : 0.0f;
                seed = p.seed[seq];
            }
            const uint16_t *srow = static_cast<const uint16_t *>(p.s) + (size_t)tok * p.V;
            SelState sel;
            sel.init();
            // (tile, group) work items in order; s of item i + 1 is loaded
            // while item i is processed
            const int items = (vt1 - vt0) * g_count;
            // s is read once: evict it first, so that W_r (re-read for every
            // token tile, evict_last) stays in L2.  (An L2 bulk prefetch of s
            // ahead of the ring measured slower: many small prefetches.)
            const uint64_t once = policy_evict_first();
            float gn[4] = {0.f, 0.f, 0.f, 0.f};     // T > 0: Gumbel noise of the tile's group quad
            // s of item k into ring slot k % TC_SPF (cp.async, L2 only; zero-filled
            // past V or for an invalid thread), one commit group per item
            const int et = threadIdx.x - 64;
            // the next item to issue, walked forward without divisions
            int is_k = 0, is_vt = vt0, is_gl = g_first;
            auto issue_next = [&]() {
                if (is_k < items) {
                    const int v0 = is_vt * TC_BN + is_gl * GROUP;
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const int vv = v0 + 8 * c;
                        const bool in = valid && vv < p.V;
                        cp_async16(&sS[((is_k % TC_SPF) * 4 + c) * (TC_EPI_WARPS * 32) + et], in ? srow + vv : srow,
                                   in ? 16u : 0u, once);
                    }
                }
                cp_async_commit();
                ++is_k;
                if (++is_gl == g_first + g_count) { is_gl = g_first; ++is_vt; }
            };
#pragma unroll
            for (int k = 0; k < TC_SPF - 1; ++k) issue_next();
            if (g_count == 0)
                for (int vt = vt0; vt < vt1; ++vt) {
                    const int buf = t & 1;
                    if (!mbar_wait(&sh.tfull[buf], (t >> 1) & 1, abort)) { ok = false; break; }
                    tc_fence_after();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sh.tempty[buf]);
                    ++t;
                }
            int vt = vt0, gl = g_first;                  // the item being folded
            for (int it = 0; it < items; ++it) {
                const int buf = t & 1;
                if (gl == g_first) {
                    if (valid && invT > 0.0f)
                        group_noise4(seed, (uint32_t)(vt * (TC_BN / GROUP) + g_first) >> 2, (uint32_t)pos, p.offset, gn);
                    if (!mbar_wait(&sh.tfull[buf], (t >> 1) & 1, abort)) { ok = false; break; }
                    tc_fence_after();
                }
                issue_next();                           // item it + TC_SPF - 1
                cp_async_wait<TC_SPF - 1>();        // item it has landed
                uint4 cur[4];
#pragma unroll
                for (int c = 0; c < 4; ++c) cur[c] = sS[((it % TC_SPF) * 4 + c) * (TC_EPI_WARPS * 32) + et];
                const int v0 = vt * TC_BN + gl * GROUP;
                const int nv = min(GROUP, p.V - v0);
                float acc[GROUP];
                tmem_ld32(tmem + lane_base + buf * TC_BN + gl * GROUP, acc);
                if (valid && nv > 0) {
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const uint32_t ww[4] = {cur[c].x, cur[c].y, cur[c].z, cur[c].w};
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            acc[c * 8 + 2 * q] += __uint_as_float(ww[q] << 16);
                            acc[c * 8 + 2 * q + 1] += __uint_as_float(ww[q] & 0xFFFF0000u);
                        }
                    }
                    if (p.logits) {
                        float *dst = p.logits + (size_t)tok * p.V + v0;
#pragma unroll
                        for (int jj = 0; jj < GROUP; ++jj)
                            if (jj < nv) dst[jj] = acc[jj];
                    }
                    select_group(sel, acc, v0, nv, invT, gn[(v0 / GROUP) & 3]);
                }
                if (gl == g_first + g_count - 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sh.tempty[buf]);
                    ++t;
                    gl = g_first;
                    ++vt;
                } else {
                    ++gl;
                }
            }
            cp_async_wait<0>();                      // nothing in flight into the ring
            sh.st[ew][lane] = sel;
            const bool stop = epi_bar_or(!ok || *abort);
            if (!stop) {
                if (small) {
                    if (ew == 0 && lane < n) {
                        RPartial a = sh.st[0][lane].partial();
                        for (int w = 1; w < TC_EPI_WARPS; ++w) merge_rpartial(a, sh.st[w][lane].partial(), invT > 0.0f);
                        p.part[(size_t)lane * p.S + r] = a;
                    }
                } else if (ew < 4 && valid) {
                    RPartial a = sh.st[ew][lane].partial();
                    for (int w = 1; w < TC_WPQ; ++w) merge_rpartial(a, sh.st[ew + 4 * w][lane].partial(), invT > 0.0f);
                    p.part[(size_t)i * p.S + r] = a;
                }
            }
            epi_bar();
            if (stop) break;
        }
    }
    if (tr0 && threadIdx.x == 64) trace_mark(p.trace, 203, t_wait);
    pdl_trigger();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TC_TMEM_COLS);
    }
    if (threadIdx.x == 0 && sh.abort) set_status(p.status, ST_TIMEOUT);
    if (threadIdx.x == 0 && p.trace) trace_mark(p.trace, 8 + 4 * p.ctl[CTL_PASS] + 1, t_start);
}

}  // namespace xp
