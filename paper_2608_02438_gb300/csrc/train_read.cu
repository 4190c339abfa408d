// train_read.cu -- the Read GEMM of the refiner training step (Sec. 4.3) on
// tcgen05, fused with the softmax / total-variation arithmetic of the loss
// L(p) = sum_k w_k [a_ce (-log p_k(y*_k)) + a_l1 |p_k - p^t_k|_1]
// and of its gradient.  The logits l = s + W_r z of all rows are recomputed by
// every pass instead of being stored (N x V floats would cost more HBM traffic
// than re-reading s and t).
//
// Rows: the refiner runs twice per position (teacher-forced inputs and the
// consistency inputs argmax s); a 128-row tile holds 64 positions, rows 0-63
// the teacher-forced forward and rows 64-127 the consistency forward of the
// same positions, so that one s / t tile of those 64 positions serves both.
//
// k_train_tok -- token-major: D[row, v] = z_row . W_r[v], M = 128 rows, N = 64
// vocabulary ids, K = r.  CTA (split, tile) takes one row tile and a
// contiguous range of vocabulary tiles.  Modes:
//   TR_STATS  per row the running max / log2-sum of l (log2 domain) and l at y*
//   TR_TV     per row sum_v min(p, q), the part where p < q and where p = q
//             (compared in the log domain: one exp2 per element), and per
//             position the same sum for the drafter's p^b = softmax(s)
//   TR_DZ     dl = p (A0 + A1 sgn(p - q)) - A2 [v = y*] as a bf16 tile in
//             shared memory, then dz += dl W_r on the tensor core (W_r tile
//             read MN-major); each split stores its dz slice at the end
// k_train_voc -- vocabulary-major: D[v, row] = W_r[v] . z_row, M = 128 ids,
// N = 64 rows (32 positions x both forwards); the same dl (transposed) feeds
// dW_r[v, :] += dl^T Z (Z tile read MN-major), accumulated in TMEM over every
// row of the step and added into gW_r once per vocabulary tile.
#include "common.cuh"
#include "kernels.h"

namespace xp {

namespace {

constexpr float L2E = 1.4426950408889634f;

// ---------------------------------------------------------------- k_train_tok
constexpr int TR_BM = 128;
constexpr int TR_BN = 64;
constexpr int TR_BSTAGES = 3;
constexpr int TR_SSTAGES = 2;
constexpr int TR_EPI_WARPS = 8;                            // 2 per TMEM lane quarter: 32 ids each
constexpr int TR_THREADS = 32 * (2 + TR_EPI_WARPS);
constexpr uint32_t TR_A_CHUNK = TR_BM * 64 * 2;            // 16 KB: 128 rows x 64 of r
constexpr uint32_t TR_A_BYTES = 4 * TR_A_CHUNK;            // 64 KB
constexpr uint32_t TR_B_CHUNK = TR_BN * 64 * 2;            // 8 KB: 64 ids x 64 of r
constexpr uint32_t TR_B_STAGE = 4 * TR_B_CHUNK;            // 32 KB: one vocabulary tile of W_r
constexpr uint32_t TR_ST_TILE = 64 * TR_BN * 2;            // 8 KB: 64 positions x 64 ids of s (or t)
constexpr uint32_t TR_S_STAGE = 2 * TR_ST_TILE;            // s and t
constexpr uint32_t TR_D_BUF = TR_BM * TR_BN * 2;           // 16 KB: dl tile, bf16, K-major (K = ids)
constexpr uint32_t TR_IDESC_F = idesc_bf16(TR_BM, TR_BN);
constexpr uint32_t TR_IDESC_D = idesc_bf16_mn(TR_BM, RANK, false, true);
constexpr uint32_t TR_TMEM_COLS = 512;                     // l: 2 x 64 at 0; dz: 256 at 256
constexpr uint32_t TR_DZ_COL = 256;

struct TrShared {
    uint64_t a_full;
    uint64_t full[TR_BSTAGES], empty[TR_BSTAGES];
    uint64_t sfull[TR_SSTAGES], sempty[TR_SSTAGES];
    uint64_t tfull[2], tempty[2];
    uint64_t dfull[2], dempty[2];
    uint64_t zdone, drain;
    uint32_t tmem_base;
    int abort;
};

constexpr size_t TR_SMEM = 1024 + TR_A_BYTES + TR_BSTAGES * TR_B_STAGE + TR_SSTAGES * TR_S_STAGE + 2 * TR_D_BUF +
                           sizeof(TrShared);

__device__ __forceinline__ void tr_epi_bar()
{
    asm volatile("bar.sync 1, %0;" ::"n"(TR_EPI_WARPS * 32) : "memory");
}

// 32 consecutive bf16 of row `pr` of a 64-wide SW128 tile (chunks 4h .. 4h+3)
__device__ __forceinline__ void ld_tile32(const uint8_t *tile, int pr, int h, uint4 (&r)[4])
{
#pragma unroll
    for (int c = 0; c < 4; ++c)
        r[c] = *reinterpret_cast<const uint4 *>(tile + pr * 128 + (((4 * h + c) ^ (pr & 7)) << 4));
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ void unpack32(const uint4 (&r)[4], float (&x)[32])
{
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        const uint32_t w[4] = {r[c].x, r[c].y, r[c].z, r[c].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            x[8 * c + 2 * q] = bf_lo(w[q]);
            x[8 * c + 2 * q + 1] = bf_hi(w[q]);
        }
    }
}

// log2-domain running log-sum-exp: value = s * 2^m
__device__ __forceinline__ void lse2_add32(float &m, float &s, const float (&x)[32])
{
    float gm = x[0];
#pragma unroll
    for (int j = 1; j < 32; ++j) gm = fmaxf(gm, x[j]);
    const float M = fmaxf(m, gm);
    if (M == -INFINITY) return;
    float acc = 0.0f;
#pragma unroll
    for (int j = 0; j < 32; ++j) acc += ex2_approx(x[j] - M);
    s = s * ex2_approx(m - M) + acc;
    m = M;
}

__device__ __forceinline__ void lse2_merge(float &m, float &s, float om, float os)
{
    const float M = fmaxf(m, om);
    if (M == -INFINITY) return;
    s = s * ex2_approx(m - M) + os * ex2_approx(om - M);
    m = M;
}

}  // namespace

const size_t kTrainTokSmemBytes = TR_SMEM;
const int kTrainTokThreads = TR_THREADS;

// grid (splits, NR / 128), TR_THREADS threads, TR_SMEM bytes.
__global__ void __launch_bounds__(TR_THREADS, 1)
    k_train_tok(const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,
                const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,
                const __grid_constant__ CUtensorMap tmap_t, int mode)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = base;
    uint8_t *sB = sA + TR_A_BYTES;
    uint8_t *sS = sB + TR_BSTAGES * TR_B_STAGE;
    uint8_t *sD = sS + TR_SSTAGES * TR_S_STAGE;
    TrShared &sh = *reinterpret_cast<TrShared *>(sD + 2 * TR_D_BUF);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int j = blockIdx.y, sv = blockIdx.x;
    const int vt0 = (int)((long long)p.nvt * sv / p.splits), vt1 = (int)((long long)p.nvt * (sv + 1) / p.splits);
    const int items = vt1 - vt0;
    const bool dzm = mode == TR_DZ;

    if (threadIdx.x == 0) {
        mbar_init(&sh.a_full, 1);
        for (int i = 0; i < TR_BSTAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        for (int i = 0; i < TR_SSTAGES; ++i) { mbar_init(&sh.sfull[i], 1); mbar_init(&sh.sempty[i], TR_EPI_WARPS); }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sh.tfull[i], 1);
            mbar_init(&sh.tempty[i], TR_EPI_WARPS);
            mbar_init(&sh.dfull[i], TR_EPI_WARPS);
            mbar_init(&sh.dempty[i], 1);
        }
        mbar_init(&sh.zdone, 1);
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, TR_TMEM_COLS); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;
    const unsigned long long lim = p.wait_ns;

    if (warp == 0) {
        // ------------------------------------------------------- producer
        if (lane == 0 && items > 0) {
            tma_prefetch_desc(&tmap_z);
            tma_prefetch_desc(&tmap_w);
            tma_prefetch_desc(&tmap_s);
            tma_prefetch_desc(&tmap_t);
            const uint64_t keep = policy_evict_last(), once = policy_evict_first();
            const bool need_t = mode != TR_STATS;
            mbar_expect_tx(&sh.a_full, TR_A_BYTES);
            for (int c = 0; c < 4; ++c) tma_load_2d(sA + c * TR_A_CHUNK, &tmap_z, &sh.a_full, c * 64, j * TR_BM);
            uint32_t pend_b = 0, par_b = 0, pend_s = 0, par_s = 0;
            for (int it = 0; it < items && !*abort; ++it) {
                const int vt = vt0 + it;
                const int st = it % TR_BSTAGES;
                const uint32_t ph = (uint32_t)((it / TR_BSTAGES) & 1);
                if (!mbar_wait(&sh.empty[st], ph ^ 1, abort, lim)) break;
                mbar_expect_tx(&sh.full[st], TR_B_STAGE);
                for (int c = 0; c < 4; ++c)
                    tma_load_2d_hint(sB + st * TR_B_STAGE + c * TR_B_CHUNK, &tmap_w, &sh.full[st], c * 64, vt * TR_BN,
                                     keep);
                pend_b |= 1u << st;
                par_b = (par_b & ~(1u << st)) | (ph << st);
                const int ss = it & 1;
                const uint32_t sph = (uint32_t)((it >> 1) & 1);
                if (!mbar_wait(&sh.sempty[ss], sph ^ 1, abort, lim)) break;
                mbar_expect_tx(&sh.sfull[ss], need_t ? TR_S_STAGE : TR_ST_TILE);
                tma_load_2d_hint(sS + ss * TR_S_STAGE, &tmap_s, &sh.sfull[ss], vt * TR_BN, j * 64, once);
                if (need_t)
                    tma_load_2d_hint(sS + ss * TR_S_STAGE + TR_ST_TILE, &tmap_t, &sh.sfull[ss], vt * TR_BN, j * 64,
                                     once);
                pend_s |= 1u << ss;
                par_s = (par_s & ~(1u << ss)) | (sph << ss);
            }
            if (*abort) {
                // no copy may still be landing when the CTA leaves
                int dummy = 0;
                mbar_wait(&sh.a_full, 0, &dummy, 100000000ull);
                for (int st = 0; st < TR_BSTAGES; ++st)
                    if (pend_b & (1u << st)) mbar_wait(&sh.full[st], (par_b >> st) & 1, &dummy, 100000000ull);
                for (int ss = 0; ss < TR_SSTAGES; ++ss)
                    if (pend_s & (1u << ss)) mbar_wait(&sh.sfull[ss], (par_s >> ss) & 1, &dummy, 100000000ull);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0 && items > 0) {
            const uint32_t a0 = smem_u32(sA), b0 = smem_u32(sB), d0 = smem_u32(sD);
            // dz += dl(u) W_r(u): A = the dl tile (K-major over ids), B = the W_r
            // tile read MN-major (N = r along the 128-byte rows, K = ids)
            auto dz_step = [&](int u) -> bool {
                const int db = u & 1;
                if (!mbar_wait(&sh.dfull[db], (uint32_t)((u >> 1) & 1), abort, lim)) return false;
                tc_fence_after();
                const uint32_t bs = b0 + (u % TR_BSTAGES) * TR_B_STAGE;
#pragma unroll
                for (int kk = 0; kk < TR_BN / 16; ++kk)
                    tc_mma_bf16(tmem + TR_DZ_COL, smem_desc_sw128(d0 + db * TR_D_BUF + kk * 32),
                                smem_desc_sw128_mn(bs + kk * 2048, TR_B_CHUNK), TR_IDESC_D, (u | kk) != 0);
                tc_commit(&sh.empty[u % TR_BSTAGES]);
                tc_commit(&sh.dempty[db]);
                return true;
            };
            bool ok = mbar_wait(&sh.a_full, 0, abort, lim);
            if (ok) tc_fence_after();
            for (int it = 0; it < items && ok; ++it) {
                const int st = it % TR_BSTAGES, buf = it & 1;
                if (!mbar_wait(&sh.full[st], (uint32_t)((it / TR_BSTAGES) & 1), abort, lim) ||
                    !mbar_wait(&sh.tempty[buf], (uint32_t)(((it >> 1) & 1) ^ 1), abort, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t bs = b0 + st * TR_B_STAGE;
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc_mma_bf16(tmem + buf * TR_BN, smem_desc_sw128(a0 + c * TR_A_CHUNK + kk * 32),
                                    smem_desc_sw128(bs + c * TR_B_CHUNK + kk * 32), TR_IDESC_F, (c | kk) != 0);
                tc_commit(&sh.tfull[buf]);
                if (!dzm) tc_commit(&sh.empty[st]);
                else if (it > 0 && !dz_step(it - 1)) ok = false;
            }
            if (ok && dzm) ok = dz_step(items - 1);
            if (ok && dzm) tc_commit(&sh.zdone);
            // every MMA issued above has finished before the CTA tears down
            tc_commit(&sh.drain);
            int dummy = 0;
            mbar_wait(&sh.drain, 0, &dummy, 100000000ull);
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int ew = warp - 2, q = warp & 3, g = ew >> 2;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const int row = q * 32 + lane, f = row >> 6, pl = row & 63;
        const int i = j * 64 + pl;                 // position
        const int rowg = j * TR_BM + row;          // paired row
        const bool valid = i < p.P;
        const int y = valid ? p.ystar[i] : -1;
        float lp2 = 0.f, lq2 = 0.f, ls2 = 0.f, A0 = 0.f, A1 = 0.f, A2 = 0.f;
        if (valid && mode != TR_STATS) {
            lp2 = p.lse_p2[rowg];
            lq2 = p.lse_q2[i];
            ls2 = p.lse_s2[i];
        }
        if (valid && dzm) {
            const RowCoef rc = p.coef[rowg];
            A0 = rc.A0;
            A1 = rc.A1;
            A2 = rc.A2;
        }
        // the anchor term's share: the teacher-forced row takes the even
        // 32-id group of each tile, the consistency row the odd one
        const bool anchor = (f == g);
        float r0 = -INFINITY, r1 = 0.f, r2 = 0.f, r3 = 0.f;   // STATS: m, s; TV: sum min, lt, eq, anchor
        if (mode == TR_TV) r0 = 0.f;
        bool ok = true;
        for (int it = 0; it < items; ++it) {
            const int buf = it & 1;
            const uint32_t ph = (uint32_t)((it >> 1) & 1);
            if (!mbar_wait(&sh.tfull[buf], ph, abort, lim) || !mbar_wait(&sh.sfull[buf], ph, abort, lim)) {
                ok = false;
                break;
            }
            tc_fence_after();
            float acc[32];
            tmem_ld32(tmem + lane_base + buf * TR_BN + g * 32, acc);
            uint4 sr[4], tr[4];
            const uint8_t *stile = sS + buf * TR_S_STAGE;
            ld_tile32(stile, pl, g, sr);
            if (mode != TR_STATS) ld_tile32(stile + TR_ST_TILE, pl, g, tr);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&sh.tempty[buf]);
                mbar_arrive(&sh.sempty[buf]);
            }
            const int v0 = (vt0 + it) * TR_BN + g * 32;
            const int nv = min(32, p.V - v0);
            float sv32[32];
            unpack32(sr, sv32);
            if (mode == TR_STATS) {
                if (valid) {
                    float x[32];
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) {
                        const float l = acc[jj] + sv32[jj];
                        x[jj] = jj < nv ? l * L2E : -INFINITY;
                        if (v0 + jj == y) p.ly[rowg] = l;
                    }
                    lse2_add32(r0, r1, x);
                }
            } else {
                float tv32[32];
                unpack32(tr, tv32);
                if (mode == TR_TV) {
                    if (valid) {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) {
                            if (jj < nv) {
                                const float a2 = fmaf(acc[jj] + sv32[jj], L2E, -lp2);
                                const float b2 = fmaf(tv32[jj], L2E, -lq2);
                                const float m = ex2_approx(fminf(a2, b2));
                                r0 += m;
                                r1 += a2 < b2 ? m : 0.f;
                                r2 += a2 == b2 ? m : 0.f;
                                if (anchor) r3 += ex2_approx(fminf(fmaf(sv32[jj], L2E, -ls2), b2));
                            }
                        }
                    }
                } else {
                    uint32_t w[16];
#pragma unroll
                    for (int jj = 0; jj < 32; jj += 2) {
                        float d2[2];
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int jv = jj + e;
                            const float a2 = fmaf(acc[jv] + sv32[jv], L2E, -lp2);
                            const float b2 = fmaf(tv32[jv], L2E, -lq2);
                            const float pv = ex2_approx(a2);
                            const float sg = a2 > b2 ? 1.f : (a2 < b2 ? -1.f : 0.f);
                            float d = pv * fmaf(A1, sg, A0) - (v0 + jv == y ? A2 : 0.f);
                            d2[e] = (jv < nv && valid) ? d : 0.f;
                        }
                        w[jj / 2] = pack_bf16x2(d2[0], d2[1]);
                    }
                    if (!mbar_wait(&sh.dempty[buf], ph ^ 1, abort, lim)) { ok = false; break; }
                    uint8_t *dt = sD + buf * TR_D_BUF + row * 128;
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        *reinterpret_cast<uint4 *>(dt + (((4 * g + c) ^ (row & 7)) << 4)) =
                            make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sh.dfull[buf]);
                }
            }
        }
        if (!dzm) {
            // merge the two id groups of each row, one partial per (split, row)
            float4 *scr = reinterpret_cast<float4 *>(sD);
            if (g == 1) scr[row] = make_float4(r0, r1, r2, r3);
            tr_epi_bar();
            if (g == 0 && valid && ok && !*abort) {
                const float4 o = scr[row];
                if (mode == TR_STATS) lse2_merge(r0, r1, o.x, o.y);
                else { r0 += o.x; r1 += o.y; r2 += o.z; r3 += o.w; }
                p.part[(size_t)sv * p.NR + rowg] = make_float4(r0, r1, r2, r3);
            }
        } else if (ok && items > 0) {
            if (mbar_wait(&sh.zdone, 0, abort, lim)) {
                tc_fence_after();
#pragma unroll 1
                for (int c4 = 0; c4 < 4; ++c4) {
                    float v[32];
                    tmem_ld32(tmem + lane_base + TR_DZ_COL + g * 128 + c4 * 32, v);
                    float4 *dst = reinterpret_cast<float4 *>(p.dzp + ((size_t)sv * p.NR + rowg) * RANK + g * 128 +
                                                             c4 * 32);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = valid ? make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3])
                                       : make_float4(0.f, 0.f, 0.f, 0.f);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TR_TMEM_COLS);
    }
    if (threadIdx.x == 0 && sh.abort) set_status(p.status, ST_TIMEOUT);
}


// ---------------------------------------------------------------- k_train_voc
namespace {

constexpr int TV_BM = 128;                                 // vocabulary ids
constexpr int TV_BN = 64;                                  // rows per step: 32 positions x 2 forwards
constexpr int TV_EPI_WARPS = 8;                            // 2 per lane quarter: teacher / consistency half
constexpr int TV_THREADS = 32 * (2 + TV_EPI_WARPS);
constexpr uint32_t TV_W_CHUNK = TV_BM * 64 * 2;            // 16 KB: 128 ids x 64 of r
constexpr uint32_t TV_W_BYTES = 4 * TV_W_CHUNK;            // 64 KB
constexpr uint32_t TV_Z_CHUNK = TV_BN * 64 * 2;            // 8 KB: 64 rows x 64 of r
constexpr uint32_t TV_Z_BYTES = 4 * TV_Z_CHUNK;            // 32 KB
constexpr uint32_t TV_ST_BOX = 32 * 64 * 2;                // 4 KB: 32 positions x 64 ids
constexpr uint32_t TV_ST_TILE = 2 * TV_ST_BOX;             // s (or t) of 32 positions x 128 ids
constexpr uint32_t TV_INFO = TV_BN * sizeof(RowCoef);      // 2 KB
constexpr uint32_t TV_STEP = TV_Z_BYTES + 2 * TV_ST_TILE + TV_INFO;   // one ring stage
constexpr uint32_t TV_D_BUF = TV_BM * TV_BN * 2;           // 16 KB: dl^T tile (K-major over rows)
constexpr uint32_t TV_IDESC_F = idesc_bf16(TV_BM, TV_BN);
constexpr uint32_t TV_IDESC_D = idesc_bf16_mn(TV_BM, RANK, false, true);
constexpr uint32_t TV_TMEM_COLS = 512;                     // l^T: 2 x 64 at 0; dW_r: 256 at 256
constexpr uint32_t TV_DW_COL = 256;

struct TvShared {
    uint64_t a_full, a_empty;
    uint64_t zfull[2], zempty[2];
    uint64_t tfull[2], tempty[2];
    uint64_t dfull[2], dempty[2];
    uint64_t wfull, wempty, drain;
    uint32_t tmem_base;
    int abort;
};

constexpr size_t TV_SMEM = 1024 + TV_W_BYTES + 2 * TV_STEP + 2 * TV_D_BUF + sizeof(TvShared);

}  // namespace

const size_t kTrainVocSmemBytes = TV_SMEM;
const int kTrainVocThreads = TV_THREADS;

// grid min(SMs, ceil(V / 128)) (persistent over vocabulary tiles), TV_THREADS
// threads, TV_SMEM bytes.  tmap_w: W_r boxes of 128 rows; tmap_z: Z boxes of 32
// rows; tmap_s / tmap_t: boxes of 64 ids x 32 positions.
__global__ void __launch_bounds__(TV_THREADS, 1)
    k_train_voc(const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,
                const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,
                const __grid_constant__ CUtensorMap tmap_t)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sW = base;
    uint8_t *sR = sW + TV_W_BYTES;                 // step ring: Z, s, t, row coefficients
    uint8_t *sD = sR + 2 * TV_STEP;
    TvShared &sh = *reinterpret_cast<TvShared *>(sD + 2 * TV_D_BUF);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int nvt = (p.V + TV_BM - 1) / TV_BM;
    const int nsteps = (p.P + 31) / 32;

    if (threadIdx.x == 0) {
        mbar_init(&sh.a_full, 1);
        mbar_init(&sh.a_empty, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sh.zfull[i], 1);
            mbar_init(&sh.zempty[i], 1 + TV_EPI_WARPS);    // the dW MMA's commit + every epilogue warp
            mbar_init(&sh.tfull[i], 1);
            mbar_init(&sh.tempty[i], TV_EPI_WARPS);
            mbar_init(&sh.dfull[i], TV_EPI_WARPS);
            mbar_init(&sh.dempty[i], 1);
        }
        mbar_init(&sh.wfull, 1);
        mbar_init(&sh.wempty, TV_EPI_WARPS);
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
    const unsigned long long lim = p.wait_ns;

    if (warp == 0) {
        // ------------------------------------------------------- producer
        if (lane == 0 && nsteps > 0) {
            tma_prefetch_desc(&tmap_z);
            tma_prefetch_desc(&tmap_w);
            tma_prefetch_desc(&tmap_s);
            tma_prefetch_desc(&tmap_t);
            const uint64_t once = policy_evict_first();
            const char *wr = static_cast<const char *>(p.W_r);
            int gu = 0, lt = 0;
            uint32_t pend = 0, par = 0;
            bool pend_a = false;
            for (int vt = blockIdx.x; vt < nvt && !*abort; vt += gridDim.x, ++lt) {
                // the next tile's W_r rows go to L2 while this one is consumed
                const int nx = vt + gridDim.x;
                if (nx < nvt)
                    prefetch_l2_bulk(wr + (size_t)nx * TV_BM * RANK * 2,
                                     (uint32_t)min(TV_BM, p.V - nx * TV_BM) * RANK * 2);
                if (!mbar_wait(&sh.a_empty, (uint32_t)((lt & 1) ^ 1), abort, lim)) break;
                mbar_expect_tx(&sh.a_full, TV_W_BYTES);
                for (int c = 0; c < 4; ++c) tma_load_2d(sW + c * TV_W_CHUNK, &tmap_w, &sh.a_full, c * 64, vt * TV_BM);
                pend_a = true;
                for (int u = 0; u < nsteps; ++u, ++gu) {
                    const int zs = gu & 1;
                    const uint32_t ph = (uint32_t)((gu >> 1) & 1);
                    if (!mbar_wait(&sh.zempty[zs], ph ^ 1, abort, lim)) break;
                    uint8_t *st = sR + zs * TV_STEP;
                    mbar_expect_tx(&sh.zfull[zs], TV_STEP);
                    const int jt = u >> 1, hh = u & 1;
                    const int rt = jt * 128 + 32 * hh;               // teacher-forced rows of the step
                    for (int c = 0; c < 4; ++c) {
                        tma_load_2d(st + c * TV_Z_CHUNK, &tmap_z, &sh.zfull[zs], c * 64, rt);
                        tma_load_2d(st + c * TV_Z_CHUNK + 4096, &tmap_z, &sh.zfull[zs], c * 64, rt + 64);
                    }
                    for (int h2 = 0; h2 < 2; ++h2) {
                        tma_load_2d_hint(st + TV_Z_BYTES + h2 * TV_ST_BOX, &tmap_s, &sh.zfull[zs],
                                         vt * TV_BM + 64 * h2, 32 * u, once);
                        tma_load_2d_hint(st + TV_Z_BYTES + TV_ST_TILE + h2 * TV_ST_BOX, &tmap_t, &sh.zfull[zs],
                                         vt * TV_BM + 64 * h2, 32 * u, once);
                    }
                    uint8_t *info = st + TV_Z_BYTES + 2 * TV_ST_TILE;
                    bulk_load_1d(info, p.coef + rt, 32 * sizeof(RowCoef), &sh.zfull[zs]);
                    bulk_load_1d(info + 32 * sizeof(RowCoef), p.coef + rt + 64, 32 * sizeof(RowCoef), &sh.zfull[zs]);
                    pend |= 1u << zs;
                    par = (par & ~(1u << zs)) | (ph << zs);
                }
            }
            if (*abort) {
                int dummy = 0;
                if (pend_a) mbar_wait(&sh.a_full, (uint32_t)((lt - 1) & 1), &dummy, 100000000ull);
                for (int zs = 0; zs < 2; ++zs)
                    if (pend & (1u << zs)) mbar_wait(&sh.zfull[zs], (par >> zs) & 1, &dummy, 100000000ull);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0 && nsteps > 0) {
            const uint32_t w0 = smem_u32(sW), r0 = smem_u32(sR), d0 = smem_u32(sD);
            int gu = 0, lt = 0;
            bool ok = true;
            // dW_r += dl^T(v) Z(v): A = the dl^T tile (K-major over rows), B = the
            // step's Z tile read MN-major (N = r along the 128-byte rows, K = rows)
            auto dw_step = [&](int v, bool first) -> bool {
                const int db = v & 1;
                if (!mbar_wait(&sh.dfull[db], (uint32_t)((v >> 1) & 1), abort, lim)) return false;
                if (first && !mbar_wait(&sh.wempty, (uint32_t)((lt & 1) ^ 1), abort, lim)) return false;
                tc_fence_after();
                const uint32_t zb = r0 + (v & 1) * TV_STEP;
#pragma unroll
                for (int kk = 0; kk < TV_BN / 16; ++kk)
                    tc_mma_bf16(tmem + TV_DW_COL, smem_desc_sw128(d0 + db * TV_D_BUF + kk * 32),
                                smem_desc_sw128_mn(zb + kk * 2048, TV_Z_CHUNK), TV_IDESC_D, !(first && kk == 0));
                tc_commit(&sh.zempty[v & 1]);
                tc_commit(&sh.dempty[db]);
                return true;
            };
            for (int vt = blockIdx.x; vt < nvt && ok; vt += gridDim.x, ++lt) {
                if (!mbar_wait(&sh.a_full, (uint32_t)(lt & 1), abort, lim)) { ok = false; break; }
                tc_fence_after();
                for (int u = 0; u < nsteps; ++u, ++gu) {
                    const int zs = gu & 1, buf = gu & 1;
                    if (!mbar_wait(&sh.zfull[zs], (uint32_t)((gu >> 1) & 1), abort, lim) ||
                        !mbar_wait(&sh.tempty[buf], (uint32_t)(((gu >> 1) & 1) ^ 1), abort, lim)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t zb = r0 + zs * TV_STEP;
#pragma unroll
                    for (int c = 0; c < 4; ++c)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc_mma_bf16(tmem + buf * TV_BN, smem_desc_sw128(w0 + c * TV_W_CHUNK + kk * 32),
                                        smem_desc_sw128(zb + c * TV_Z_CHUNK + kk * 32), TV_IDESC_F, (c | kk) != 0);
                    tc_commit(&sh.tfull[buf]);
                    if (u == nsteps - 1) tc_commit(&sh.a_empty);
                    if (u > 0 && !dw_step(gu - 1, u == 1)) { ok = false; break; }
                }
                if (!ok) break;
                if (!dw_step(gu - 1, nsteps == 1)) { ok = false; break; }
                tc_commit(&sh.wfull);
            }
            tc_commit(&sh.drain);
            int dummy = 0;
            mbar_wait(&sh.drain, 0, &dummy, 100000000ull);
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int ew = warp - 2, q = warp & 3, g = ew >> 2;     // g: 0 teacher-forced rows, 1 consistency rows
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const int vr = q * 32 + lane;                          // id row of the tile
        const int h2 = vr >> 6, cc = vr & 63;                  // s / t box and column within it
        int gu = 0, lt = 0;
        bool ok = nsteps > 0;
        for (int vt = blockIdx.x; vt < nvt && ok; vt += gridDim.x, ++lt) {
            const int v = vt * TV_BM + vr;
            const bool vvalid = v < p.V;
            for (int u = 0; u < nsteps; ++u, ++gu) {
                const int buf = gu & 1;
                const uint32_t ph = (uint32_t)((gu >> 1) & 1);
                if (!mbar_wait(&sh.tfull[buf], ph, abort, lim) || !mbar_wait(&sh.zfull[buf], ph, abort, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                float acc[32];
                tmem_ld32(tmem + lane_base + buf * TV_BN + g * 32, acc);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sh.tempty[buf]);
                const uint8_t *st = sR + buf * TV_STEP;
                const uint8_t *sbox = st + TV_Z_BYTES + h2 * TV_ST_BOX;
                const RowCoef *info = reinterpret_cast<const RowCoef *>(st + TV_Z_BYTES + 2 * TV_ST_TILE) + g * 32;
                const int coff = (cc & 7) * 2;
                uint32_t w[16];
#pragma unroll
                for (int c = 0; c < 32; c += 2) {
                    float d2[2];
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const int pr = c + e;                  // position within the step
                        const int off = pr * 128 + (((cc >> 3) ^ (pr & 7)) << 4) + coff;
                        const float sv = bf2f(*reinterpret_cast<const uint16_t *>(sbox + off));
                        const float tv = bf2f(*reinterpret_cast<const uint16_t *>(sbox + TV_ST_TILE + off));
                        const RowCoef rc = info[pr];
                        const float a2 = fmaf(acc[pr] + sv, L2E, -rc.lse_p2);
                        const float b2 = fmaf(tv, L2E, -rc.lse_q2);
                        const float pv = ex2_approx(a2);
                        const float sg = a2 > b2 ? 1.f : (a2 < b2 ? -1.f : 0.f);
                        const float d = pv * fmaf(rc.A1, sg, rc.A0) - (v == rc.y ? rc.A2 : 0.f);
                        d2[e] = vvalid ? d : 0.f;
                    }
                    w[c / 2] = pack_bf16x2(d2[0], d2[1]);
                }
                if (!mbar_wait(&sh.dempty[buf], ph ^ 1, abort, lim)) { ok = false; break; }
                uint8_t *dt = sD + buf * TV_D_BUF + vr * 128;
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    *reinterpret_cast<uint4 *>(dt + (((4 * g + c) ^ (vr & 7)) << 4)) =
                        make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&sh.dfull[buf]);
                    mbar_arrive(&sh.zempty[buf]);
                }
            }
            if (!ok) break;
            // this tile's dW_r rows: add into gW_r, then hand the accumulator back
            if (!mbar_wait(&sh.wfull, (uint32_t)(lt & 1), abort, lim)) { ok = false; break; }
            tc_fence_after();
#pragma unroll 1
            for (int c4 = 0; c4 < 4; ++c4) {
                float wv[32];
                tmem_ld32(tmem + lane_base + TV_DW_COL + g * 128 + c4 * 32, wv);
                if (vvalid) {
                    float4 *dst = reinterpret_cast<float4 *>(p.gW_r + (size_t)v * RANK + g * 128 + c4 * 32);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        float4 o = dst[e];
                        o.x += wv[4 * e];
                        o.y += wv[4 * e + 1];
                        o.z += wv[4 * e + 2];
                        o.w += wv[4 * e + 3];
                        dst[e] = o;
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.wempty);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TV_TMEM_COLS);
    }
    if (threadIdx.x == 0 && sh.abort) set_status(p.status, ST_TIMEOUT);
}

}  // namespace xp
