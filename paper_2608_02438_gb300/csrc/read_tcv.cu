// read_tcv.cu -- Read + Correct + selection for small batches (<= 32 evaluated
// tokens), vocabulary rows as the MMA's M dimension.
//
// Same result as k_read_tc (Sec. 4.1 Eq. read / correct, Algorithm 1's argmax,
// the T > 0 group draw), but D[v, t] = W_r[v, :] . z[t, :] with M = 128
// vocabulary rows, N = 32 token columns, K = r = 256: with at most 32 tokens
// this does 1/8 of the tensor work of a 128-token tile.  TMEM lane quarter q of
// an accumulator holds vocabulary rows 32 q .. 32 q + 31 of the block, i.e.
// exactly one 32-id group.
//
// Roles (320 threads, one CTA per SM, persistent over a contiguous range of
// 128-row vocabulary blocks):
//   warp 0      TMA producer: z (the 32 x 256 B operand, kept) and an 8-stage
//               ring of W_r K-chunks (16 KB each)
//   warp 1      TMEM allocator and tcgen05.mma issuer
//   warps 2-9   epilogue: quarter q = warp % 4, half h = (warp - 2) / 4 takes
//               every other block; the 32 x 32 accumulator tile of a quarter
//               is transposed through shared memory so that lane t folds the
//               group of token t (select_group), with its s segment read from
//               global memory one block ahead
// Four TMEM accumulators of 32 columns decouple the MMA from the epilogue.
#include "common.cuh"
#include "kernels.h"
#include "reduce_common.cuh"
#include "tcv_common.cuh"

namespace xp {

struct TvShared {
    uint64_t full[TV_STAGES];
    uint64_t empty[TV_STAGES];
    uint64_t z_full;
    uint64_t tfull[TV_NBUF], tempty[TV_NBUF];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    int tok[TV_BN], pos[TV_BN];
    float invT[TV_BN];
    unsigned long long seed[TV_BN];
    SelState st[TV_EPI_WARPS][32];
    float tile[TV_EPI_WARPS][TV_BN][33];      // per-warp transpose: [token][vocabulary row]
    int last;                                 // this CTA finished last: it reduces the pass
    int ynew[TV_BN], yold[TV_BN];             // per evaluated token: new / previous token
    SeqState seq[TV_BN];                      // block states at the start of the pass (b <= 32)
    int passes;
};

constexpr size_t TV_SMEM_BYTES = 1024 + TV_STAGES * TV_A_STAGE + TV_Z_BYTES + sizeof(TvShared);
const size_t kReadTcvSmemBytes = TV_SMEM_BYTES;
const int kReadTcvThreads = TV_THREADS;

__global__ void __launch_bounds__(TV_THREADS, 1)
    k_read_tcv(const Params *__restrict__ pp, const __grid_constant__ CUtensorMap tmap_wr128,
               const __grid_constant__ CUtensorMap tmap_z, int V, int fuse, cudaGraphConditionalHandle handle)
{
    const unsigned long long t_start = globaltimer_ns();
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = base;                                   // W_r stages
    uint8_t *sZ = base + TV_STAGES * TV_A_STAGE;          // z, 4 K-chunks
    TvShared &sh = *reinterpret_cast<TvShared *>(sZ + TV_Z_BYTES);
    const Params &p = *pp;
    const int NVB = (V + TV_BM - 1) / TV_BM;
    const int S = gridDim.x, r = blockIdx.x;
    const int vb0 = (int)((long long)NVB * r / S), vb1 = (int)((long long)NVB * (r + 1) / S);
    const int nblk = vb1 - vb0;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < TV_STAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        mbar_init(&sh.z_full, 1);
        for (int i = 0; i < TV_NBUF; ++i) { mbar_init(&sh.tfull[i], 1); mbar_init(&sh.tempty[i], 4); }
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, TV_TMEM_COLS); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;

    // W_r does not depend on the previous kernel: start streaming it before
    // waiting for that kernel (programmatic dependent launch)
    const int pre = min(TV_STAGES, nblk * TV_KCH);
    const uint64_t keep = policy_evict_last();
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_wr128);
        tma_prefetch_desc(&tmap_z);
        const char *wr = static_cast<const char *>(p.W_r);
        const int rows = min(vb1 * TV_BM, V) - vb0 * TV_BM;
        for (int r0 = 0; r0 < rows; r0 += 64)
            prefetch_l2_bulk(wr + (size_t)(vb0 * TV_BM + r0) * RANK * 2, (uint32_t)min(64, rows - r0) * RANK * 2);
        for (int i = 0; i < pre; ++i) {
            mbar_expect_tx(&sh.full[i], TV_A_STAGE);
            tma_load_2d_hint(sA + i * TV_A_STAGE, &tmap_wr128, &sh.full[i], (i % TV_KCH) * TV_BK,
                             (vb0 + i / TV_KCH) * TV_BM, keep);
        }
    }
    pdl_wait();
    const unsigned long long t_wait = globaltimer_ns();
    const int n = min(p.ctl[CTL_NACT], TV_BN);
    const bool tr0 = p.trace && p.ctl[CTL_PASS] == 0;
    if (n == 0 && warp == 0 && lane == 0) {
        int dummy = 0;
        for (int i = 0; i < pre; ++i) mbar_wait(&sh.full[i], 0, &dummy, 10000000ull);
    }
    const int blocks = n == 0 ? 0 : nblk;

    if (warp == 0) {
        // ------------------------------------------------------- producer
        if (lane == 0 && blocks > 0) {
            mbar_expect_tx(&sh.z_full, TV_Z_BYTES);
            for (int kc = 0; kc < TV_KCH; ++kc) tma_load_2d(sZ + kc * TV_Z_CHUNK, &tmap_z, &sh.z_full, kc * TV_BK, 0);
            int stage = 0, skip = pre;
            uint32_t phase = 0, pending = 0, pend_par = 0;
            for (int i = 0; i < pre; ++i) pending |= 1u << i;
            for (int i = 0; i < blocks && !*abort; ++i)
                for (int kc = 0; kc < TV_KCH; ++kc) {
                    if (skip > 0) {
                        --skip;
                        if (++stage == TV_STAGES) { stage = 0; phase ^= 1; }
                        continue;
                    }
                    if (!mbar_wait(&sh.empty[stage], phase ^ 1, abort)) break;
                    mbar_expect_tx(&sh.full[stage], TV_A_STAGE);
                    tma_load_2d_hint(sA + stage * TV_A_STAGE, &tmap_wr128, &sh.full[stage], kc * TV_BK,
                                     (vb0 + i) * TV_BM, keep);
                    pending |= 1u << stage;
                    pend_par = (pend_par & ~(1u << stage)) | (phase << stage);
                    if (++stage == TV_STAGES) { stage = 0; phase ^= 1; }
                }
            if (*abort) {
                int dummy = 0;
                for (int st = 0; st < TV_STAGES; ++st)
                    if (pending & (1u << st)) mbar_wait(&sh.full[st], (pend_par >> st) & 1, &dummy, 10000000ull);
                mbar_wait(&sh.z_full, 0, &dummy, 10000000ull);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0 && blocks > 0) {
            int stage = 0;
            uint32_t phase = 0;
            if (mbar_wait(&sh.z_full, 0, abort)) {
                tc_fence_after();
                if (tr0) trace_mark(p.trace, 201, t_wait);
                const uint32_t z0 = smem_u32(sZ);
                for (int i = 0; i < blocks && !*abort; ++i) {
                    const int buf = i % TV_NBUF;
                    if (!mbar_wait(&sh.tempty[buf], ((i / TV_NBUF) & 1) ^ 1, abort)) break;
                    tc_fence_after();
                    const uint32_t d = tmem + buf * TV_BN;
                    for (int kc = 0; kc < TV_KCH; ++kc) {
                        if (!mbar_wait(&sh.full[stage], phase, abort)) break;
                        tc_fence_after();
                        const uint32_t a0 = smem_u32(sA + stage * TV_A_STAGE);
#pragma unroll
                        for (int kk = 0; kk < TV_BK / 16; ++kk)
                            tc_mma_bf16(d, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(z0 + kc * TV_Z_CHUNK + kk * 32),
                                        TV_IDESC, (kc | kk) != 0);
                        tc_commit(&sh.empty[stage]);
                        if (++stage == TV_STAGES) { stage = 0; phase ^= 1; }
                    }
                    tc_commit(&sh.tfull[buf]);
                }
            }
            tc_commit(&sh.drain);
            int dummy = 0;
            mbar_wait(&sh.drain, 0, &dummy, 100000000ull);
            if (tr0) trace_mark(p.trace, 202, t_wait);
        }
    } else if (blocks > 0) {
        // ------------------------------------------------------ epilogue
        const int ew = warp - 2, q = warp & 3, half = ew >> 2;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        if (ew == 0) {
            const int t = lane;
            int tok = 0, seq = 0, pos = 0;
            float invT = 0.0f;
            unsigned long long seed = 0;
            if (t < n) {
                tok = p.act_tok[t];
                seq = tok / p.B;
                pos = tok % p.B;
                const float T = p.temperature[seq];
                invT = T > 0.0f ? 1.0f / T : 0.0f;
                seed = p.seed[seq];
            }
            sh.tok[t] = tok;
            sh.pos[t] = pos;
            sh.invT[t] = invT;
            sh.seed[t] = seed;
            if (fuse) {
                // what the fused end of the pass needs, read once up front
                if (t < n) sh.yold[t] = p.tokens[tok];
                if (t < p.b) sh.seq[t] = p.st[t];
                if (t == 0) sh.passes = p.ctl[CTL_PASS];
            }
        }
        tv_epi_bar();
        // lane t owns token t: its s row segment of the next block is loaded
        // (16-byte pieces) while the current block is processed
        const int my_tok = sh.tok[lane], my_pos = sh.pos[lane];
        const float my_invT = sh.invT[lane];
        const unsigned long long my_seed = sh.seed[lane];
        const bool tvalid = lane < n;
        const uint16_t *srow = static_cast<const uint16_t *>(p.s) + (size_t)my_tok * V;
        float (*tile)[33] = sh.tile[ew];
        SelState sel;
        sel.init();
        bool ok = true;
        uint4 cur[4], nxt[4];
        if (half < blocks) load_s_group(cur, srow, (vb0 + half) * TV_BM + q * 32, V, tvalid);
        for (int i = half; i < blocks; i += 2) {
            const int buf = i % TV_NBUF;
            const int v0 = (vb0 + i) * TV_BM + q * 32;          // this warp's group
            if (i + 2 < blocks) load_s_group(nxt, srow, (vb0 + i + 2) * TV_BM + q * 32, V, tvalid);
            if (!mbar_wait(&sh.tfull[buf], (i / TV_NBUF) & 1, abort)) { ok = false; break; }
            tc_fence_after();
            float acc[TV_BN];
            tmem_ld32(tmem + lane_base + buf * TV_BN, acc);     // lane: vocabulary row, acc[t]: token t
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.tempty[buf]);
#pragma unroll
            for (int t2 = 0; t2 < TV_BN; ++t2) tile[t2][lane] = acc[t2];
            __syncwarp();
            const int nv = min(GROUP, V - v0);
            if (tvalid && nv > 0) {
                float l[GROUP];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const uint32_t ww[4] = {cur[c].x, cur[c].y, cur[c].z, cur[c].w};
#pragma unroll
                    for (int e2 = 0; e2 < 4; ++e2) {
                        l[c * 8 + 2 * e2] = tile[lane][c * 8 + 2 * e2] + __uint_as_float(ww[e2] << 16);
                        l[c * 8 + 2 * e2 + 1] = tile[lane][c * 8 + 2 * e2 + 1] + __uint_as_float(ww[e2] & 0xFFFF0000u);
                    }
                }
                if (p.logits) {
                    float *dst = p.logits + (size_t)my_tok * V + v0;
#pragma unroll
                    for (int jj = 0; jj < GROUP; ++jj)
                        if (jj < nv) dst[jj] = l[jj];
                }
                const float gz = my_invT > 0.0f ? group_noise(my_seed, (uint32_t)(v0 / GROUP), (uint32_t)my_pos, p.offset) : 0.0f;
                select_group(sel, l, v0, nv, my_invT, gz);
            }
            __syncwarp();
#pragma unroll
            for (int c = 0; c < 4; ++c) cur[c] = nxt[c];
        }
        sh.st[ew][lane] = sel;
        const bool stop = tv_epi_bar_or(!ok || *abort);
        if (!stop && ew == 0 && lane < n) {
            RPartial a = sh.st[0][lane].partial();
            for (int w = 1; w < TV_EPI_WARPS; ++w) merge_rpartial(a, sh.st[w][lane].partial(), my_invT > 0.0f);
            p.part[(size_t)lane * p.S + r] = a;
        }
    }
    if (tr0 && threadIdx.x == 64) trace_mark(p.trace, 203, t_wait);
    const int tr_slot = 8 + 4 * p.ctl[CTL_PASS] + 1;
    pdl_trigger();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TV_TMEM_COLS);
    }
    if (threadIdx.x == 0 && sh.abort) set_status(p.status, ST_TIMEOUT);
    if (fuse && n > 0) {
        // end of the pass, fused: the last CTA to finish combines the
        // partials of every evaluated token, applies Algorithm 1's stopping
        // rule to each block and packs the next pass
        if (threadIdx.x == 0) {
            __threadfence();
            sh.last = atomicAdd(&p.ctl[CTL_DONE], 1) == S - 1;
        }
        __syncthreads();
        if (sh.last) {
            __threadfence();
            const unsigned long long t_last = globaltimer_ns();
            if (tr0 && threadIdx.x == 0) trace_mark(p.trace, 204, t_wait);
            for (int t = warp; t < n; t += TV_THREADS / 32) {
                const int tok = sh.tok[t];
                const TokenResult res = reduce_token(p, t, tok, sh.invT[t], sh.seed[t]);
                if (lane == 0) {
                    sh.ynew[t] = res.y;
                    if (p.lse) p.lse[tok] = res.lse;
                    if (p.logit_sel) p.logit_sel[tok] = res.sel;
                    p.tokens[tok] = res.y;
                    record_traj(p, tok, sh.passes, res.y);
                }
            }
            __syncthreads();
            if (tr0 && threadIdx.x == 0) trace_mark(p.trace, 205, t_last);
            if (warp == 0) converge_pack_small(p, sh.seq, sh.ynew, sh.yold, sh.passes, handle);
            if (tr0 && threadIdx.x == 0) trace_mark(p.trace, 207, t_last);
        }
    }
    if (threadIdx.x == 0 && p.trace) trace_mark(p.trace, tr_slot, t_start);
}

}  // namespace xp
