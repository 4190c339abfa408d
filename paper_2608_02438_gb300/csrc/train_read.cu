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
// k_train_tok -- token-major: D[row, v] = z_row . W_r[v], M = 128 rows, N = 128
// vocabulary ids in TR_STATS, 64 in TR_TV and TR_DZ, K = r.  CTA (split, tile) takes one row tile and a
// contiguous range of vocabulary tiles.  The row tile Z sits in tensor memory
// as the A operand (with N = 64, re-reading a 4 KB A block from shared memory
// for every MMA would cost more than the product), so shared memory holds
// only the W_r and s / t rings.  Modes:
//   TR_STATS  per row the running max / log2-sum of l (log2 domain)
//   TR_TV     per row sum_v min(p, q), the part where p < q and where p = q
//             (compared in the log domain: one exp2 per element), and per
//             position the same sum for the drafter's p^b = softmax(s)
//   TR_DZ     dl = p A(sgn(p - q)) as a bf16 tile in shared memory, then
//             dz += dl W_r on the tensor core (W_r tile read MN-major); each
//             split stores its dz slice at the end
// k_train_voc -- vocabulary-major: D[v, row] = W_r[v] . z_row, M = 128 ids,
// N = 64 rows (32 positions x both forwards); the same dl (transposed) feeds
// dW_r[v, :] += dl^T Z (Z tile read MN-major), accumulated in TMEM over every
// row of the step and added into gW_r once per vocabulary tile.
// The s and t tiles stream from HBM: the producers prefetch them into L2 a
// few tiles ahead (tensor-map prefetch) so that the TMA loads of the rings
// hit L2.  The -A2 [v = y*] term of dL/dl and l at y* are left to the small
// kernels (k_train_dz, k_train_stats_fin), so the loops here carry no id test.
#include "train_common.cuh"
#include "kernels.h"

namespace xp {

namespace {

constexpr float L2E = 1.4426950408889634f;

// ---------------------------------------------------------------- k_train_tok
constexpr int TR_BM = 128;
constexpr int TR_BN = 64;                                  // ids per tile in TR_DZ (128 in the other modes)
constexpr int TR_BMAX = 4;                                 // most W_r ring stages
constexpr int TR_SMAX = 8;                                 // most s / t ring stages
constexpr int TR_PF = 8;                                   // s / t tiles prefetched into L2 ahead
constexpr int TR_EPI_WARPS = 16;                           // 2 sets (item parity) x 4 lane quarters x 2 id groups
constexpr int TR_SET = TR_EPI_WARPS / 2;                   // the warps that take one item
constexpr int TR_THREADS = 32 * (2 + TR_EPI_WARPS);
constexpr uint32_t TR_BOX = 64 * 64 * 2;                   // 8 KB: a TMA box of 64 rows x 64 bf16 (128 B)
constexpr uint32_t TR_D_BUF = TR_BM * TR_BN * 2;           // 16 KB: dl tile, bf16, K-major (K = ids)
constexpr uint32_t TR_RINGS = 224 * 1024;                  // W_r ring, s / t ring (and the dl tiles in TR_DZ)
constexpr uint32_t TR_IDESC_D = idesc_bf16_mn(TR_BM, RANK, false, true);
constexpr int TR_NBUF = 4;                                 // most l accumulators in flight
// TMEM: the l accumulators (tr_nbuf) of bn columns from 0, then the Z tile (128
// columns: 256 bf16 per lane, two per column), then in TR_DZ dz (256) at 256
constexpr uint32_t TR_TMEM_COLS = 512;
constexpr uint32_t TR_DZ_COL = 256;

struct TrShared {
    uint64_t a_full;
    uint64_t full[TR_BMAX], empty[TR_BMAX];
    uint64_t sfull[TR_SMAX], sempty[TR_SMAX];
    uint64_t tfull[TR_NBUF], tempty[TR_NBUF];
    uint64_t dfull[2], dempty[2];
    uint64_t zdone, drain;
    uint32_t tmem_base;
    int abort;
};

constexpr size_t TR_SMEM = 1024 + TR_RINGS + sizeof(TrShared);
static_assert(TR_SMEM <= 232448, "k_train_tok shared memory");

// The rings of each mode (TR_RINGS holds them): W_r stages (the W_r loads
// from L2 take about 2 us under load, so their ring depth sets the pace; the
// s / t tiles are prefetched into L2 and need fewer), s / t stage bytes and
// stages, and the two dl tiles in TR_DZ.
// 128-id tiles where the epilogue is light (the log-sum-exp pass: the MMA of a
// 16-instruction tile costs the same for N = 64 and N = 128), 64 otherwise
__host__ __device__ constexpr int tr_bn(int mode) { return mode == TR_STATS ? 2 * TR_BN : TR_BN; }
__host__ __device__ constexpr uint32_t tr_bstage(int mode) { return 4u * tr_bn(mode) * 128u; }   // a W_r tile
__host__ __device__ constexpr int tr_bstages(int mode) { return mode == TR_STATS ? 2 : 4; }
__host__ __device__ constexpr int tr_nbuf(int mode) { return mode == TR_TV ? 4 : 2; }
static_assert(tr_nbuf(TR_STATS) * 2 * 64 + 128 <= 512 && tr_nbuf(TR_TV) * 64 + 128 <= 512 &&
                  tr_nbuf(TR_DZ) * 64 + 128 <= 256,
              "tensor memory: accumulators + Z (+ dz)");
__host__ __device__ constexpr uint32_t tr_st_tile(int mode) { return (uint32_t)tr_bn(mode) * 64u * 2u; }   // s or t
__host__ __device__ constexpr uint32_t tr_stage_bytes(int mode)
{
    return mode == TR_STATS ? tr_st_tile(mode) : 2 * tr_st_tile(mode);
}
__host__ __device__ constexpr int tr_stages(int mode)
{
    return (int)((TR_RINGS - tr_bstages(mode) * tr_bstage(mode) - (mode == TR_DZ ? 2 * TR_D_BUF : 0)) /
                 tr_stage_bytes(mode));
}
static_assert(tr_stages(TR_STATS) <= TR_SMAX && tr_stages(TR_TV) >= 2 && tr_stages(TR_DZ) >= 2 &&
                  tr_stages(TR_TV) <= TR_SMAX && tr_stages(TR_DZ) <= TR_SMAX && tr_bstages(TR_DZ) <= TR_BMAX,
              "ring depths");

__device__ __forceinline__ void tr_epi_bar()
{
    asm volatile("bar.sync 1, %0;" ::"n"(TR_EPI_WARPS * 32) : "memory");
}

// log2-domain running log-sum-exp over 16 values: value = s * 2^m.  The max
// and the sum run as trees (short dependent chains).
__device__ __forceinline__ void lse2_add16(float &m, float &s, const float (&x)[16])
{
    float t[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) t[j] = fmaxf(x[j], x[j + 8]);
#pragma unroll
    for (int w = 4; w >= 1; w >>= 1)
#pragma unroll
        for (int j = 0; j < w; ++j) t[j] = fmaxf(t[j], t[j + w]);
    const float M = fmaxf(m, t[0]);
    if (M == -INFINITY) return;
    float e[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) e[j] = ex2_approx(x[j] - M) + ex2_approx(x[j + 8] - M);
#pragma unroll
    for (int w = 4; w >= 1; w >>= 1)
#pragma unroll
        for (int j = 0; j < w; ++j) e[j] += e[j + w];
    s = s * ex2_approx(m - M) + e[0];
    m = M;
}

__device__ __forceinline__ void lse2_merge(float &m, float &s, float om, float os)
{
    const float M = fmaxf(m, om);
    if (M == -INFINITY) return;
    s = s * ex2_approx(m - M) + os * ex2_approx(om - M);
    m = M;
}

// dL/dl_v without the y* term: p A(sgn(p - q)); A(0) = (Apos + Aneg) / 2
__device__ __forceinline__ float dl_value(float a2, float b2, float Apos, float Aneg)
{
    const float A = a2 > b2 ? Apos : (a2 < b2 ? Aneg : 0.5f * (Apos + Aneg));
    return ex2_approx(a2) * A;
}

}  // namespace

const size_t kTrainTokSmemBytes = TR_SMEM;
const int kTrainTokThreads = TR_THREADS;

// The token-major kernel for one mode (compiled once per mode, so that its
// tile width, ring depths and epilogue are constants).  tmap_w: W_r as (64
// columns, rows, 4 K chunks), boxes of 64 x bn x 4 (one copy per tile);
// tmap_s / tmap_t: boxes of 64 ids x 64 positions.
template <int mode>
__device__ __forceinline__ void train_tok_body(const TrainParams &p, const CUtensorMap &tmap_w,
                                               const CUtensorMap &tmap_s, const CUtensorMap &tmap_t)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sB = base;
    TrShared &sh = *reinterpret_cast<TrShared *>(sB + TR_RINGS);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int j = blockIdx.y, sv = blockIdx.x;
    constexpr int bn = tr_bn(mode);                // ids per tile
    const int nvtm = (p.V + bn - 1) / bn;
    const int vt0 = (int)((long long)nvtm * sv / p.splits), vt1 = (int)((long long)nvtm * (sv + 1) / p.splits);
    const int items = vt1 - vt0;
    constexpr bool dzm = mode == TR_DZ;
    constexpr int NB = tr_bstages(mode), NS = tr_stages(mode);
    constexpr uint32_t BST = tr_bstage(mode), BCH = (uint32_t)tr_bn(mode) * 128, STT = tr_st_tile(mode);
    constexpr int NBUF = tr_nbuf(mode);
    constexpr uint32_t ZC = NBUF * bn;             // TMEM column of the Z tile
    constexpr uint32_t SB = tr_stage_bytes(mode);
    uint8_t *sS = sB + NB * BST;                   // s / t ring after the W_r ring
    uint8_t *sD = sS + NS * SB;                    // TR_DZ: the two dl tiles after the s / t ring

    if (threadIdx.x == 0) {
        mbar_init(&sh.a_full, TR_EPI_WARPS);       // every epilogue warp stores its part of Z
        for (int i = 0; i < NB; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        for (int i = 0; i < NS; ++i) { mbar_init(&sh.sfull[i], 1); mbar_init(&sh.sempty[i], TR_SET); }
        for (int i = 0; i < TR_NBUF; ++i) {
            mbar_init(&sh.tfull[i], 1);
            mbar_init(&sh.tempty[i], TR_SET);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sh.dfull[i], TR_SET);
            mbar_init(&sh.dempty[i], 1);
        }
        mbar_init(&sh.zdone, 1);
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, TR_TMEM_COLS); tmem_relinquish(); }
    pdl_trigger();                 // the next kernel may start its set-up
    pdl_wait();                    // Z, the statistics and the coefficients are complete
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;
    const unsigned long long lim = p.wait_ns;

    if (warp == 0) {
        // ------------------------------------------------------- producer
        if (lane == 0 && items > 0) {
            tma_prefetch_desc(&tmap_w);
            tma_prefetch_desc(&tmap_s);
            tma_prefetch_desc(&tmap_t);
            const uint64_t keep = policy_evict_last(), once = policy_evict_first();
            constexpr bool need_t = mode != TR_STATS;
            auto prefetch_st = [&](int it) {
                for (int x = 0; x < bn; x += 64) {
                    tma_prefetch_2d(&tmap_s, (vt0 + it) * bn + x, j * 64);
                    if (need_t) tma_prefetch_2d(&tmap_t, (vt0 + it) * bn + x, j * 64);
                }
            };
            for (int it = 0; it < min(TR_PF, items); ++it) prefetch_st(it);
            uint32_t pend_b = 0, par_b = 0, pend_s = 0, par_s = 0;
            int ss = 0;
            uint32_t sph = 0;
            for (int it = 0; it < items && !*abort; ++it) {
                const int vt = vt0 + it;
                if (it + TR_PF < items) prefetch_st(it + TR_PF);
                const int st = it % NB;
                const uint32_t ph = (uint32_t)((it / NB) & 1);
                if (!mbar_wait_spin(&sh.empty[st], ph ^ 1, abort, lim)) break;
                mbar_expect_tx(&sh.full[st], BST);   // tmap_w: (64 columns, rows, K chunk), boxes of bn rows
                tma_load_w3d(sB + st * BST, &tmap_w, &sh.full[st], vt * bn, keep);
                pend_b |= 1u << st;
                par_b = (par_b & ~(1u << st)) | (ph << st);
                if (!mbar_wait_spin(&sh.sempty[ss], sph ^ 1, abort, lim)) break;
                mbar_expect_tx(&sh.sfull[ss], SB);
                for (int x = 0; x < bn; x += 64) {   // boxes of 64 ids x 64 positions
                    tma_load_2d_hint(sS + ss * SB + x * 128, &tmap_s, &sh.sfull[ss], vt * bn + x, j * 64, once);
                    if (need_t)
                        tma_load_2d_hint(sS + ss * SB + STT + x * 128, &tmap_t, &sh.sfull[ss], vt * bn + x, j * 64,
                                         once);
                }
                pend_s |= 1u << ss;
                par_s = (par_s & ~(1u << ss)) | (sph << ss);
                if (++ss == NS) { ss = 0; sph ^= 1; }
            }
            if (*abort) {
                // no copy may still be landing when the CTA leaves
                int dummy = 0;
                for (int st = 0; st < NB; ++st)
                    if (pend_b & (1u << st)) mbar_wait_spin(&sh.full[st], (par_b >> st) & 1, &dummy, 100000000ull);
                for (int s2 = 0; s2 < NS; ++s2)
                    if (pend_s & (1u << s2)) mbar_wait_spin(&sh.sfull[s2], (par_s >> s2) & 1, &dummy, 100000000ull);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0 && items > 0) {
            const uint32_t b0 = smem_u32(sB), d0 = smem_u32(sD);
            // descriptors formed once, advanced per MMA
            const uint64_t bdesc0 = smem_desc_sw128(b0), ddesc0 = smem_desc_sw128(d0);
            const uint64_t bmn0 = smem_desc_sw128_mn(b0, BCH);
            // dz += dl(u) W_r(u): A = the dl tile (K-major over ids), B = the W_r
            // tile read MN-major (N = r along the 128-byte rows, K = ids)
            auto dz_step = [&](int u) -> bool {
                const int db = u & 1;
                if (!mbar_wait_spin(&sh.dfull[db], (uint32_t)((u >> 1) & 1), abort, lim)) return false;
                tc_fence_after();
                const uint64_t bs = smem_desc_advance(bmn0, (u % NB) * BST);
                const uint64_t ds = smem_desc_advance(ddesc0, db * TR_D_BUF);
#pragma unroll
                for (int kk = 0; kk < TR_BN / 16; ++kk)
                    tc_mma_bf16(tmem + TR_DZ_COL, smem_desc_advance(ds, kk * 32), smem_desc_advance(bs, kk * 2048),
                                TR_IDESC_D, (u | kk) != 0);
                tc_commit(&sh.empty[u % NB]);
                tc_commit(&sh.dempty[db]);
                return true;
            };
            bool ok = mbar_wait_spin(&sh.a_full, 0, abort, lim);
            if (ok) tc_fence_after();
            const uint32_t idesc_f = idesc_bf16(TR_BM, bn);
            // TR_TV: two tiles at a time, their MMA chains interleaved (two
            // accumulators), so that consecutive MMAs do not depend on one another
            constexpr bool pairs = mode == TR_TV;
            for (int it = 0; pairs && it + 1 < items && ok; it += 2) {
                const int st0 = it % NB, st1 = (it + 1) % NB, q0 = it % NBUF, q1 = (it + 1) % NBUF;
                if (!mbar_wait_spin(&sh.full[st0], (uint32_t)((it / NB) & 1), abort, lim) ||
                    !mbar_wait_spin(&sh.full[st1], (uint32_t)(((it + 1) / NB) & 1), abort, lim) ||
                    !mbar_wait_spin(&sh.tempty[q0], (uint32_t)(((it / NBUF) & 1) ^ 1), abort, lim) ||
                    !mbar_wait_spin(&sh.tempty[q1], (uint32_t)((((it + 1) / NBUF) & 1) ^ 1), abort, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t bs0 = smem_desc_advance(bdesc0, st0 * BST), bs1 = smem_desc_advance(bdesc0, st1 * BST);
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        tc_mma_bf16_ts(tmem + q0 * bn, tmem + ZC + c * 32 + kk * 8,
                                       smem_desc_advance(bs0, c * BCH + kk * 32), idesc_f, (c | kk) != 0);
                        tc_mma_bf16_ts(tmem + q1 * bn, tmem + ZC + c * 32 + kk * 8,
                                       smem_desc_advance(bs1, c * BCH + kk * 32), idesc_f, (c | kk) != 0);
                    }
                tc_commit(&sh.tfull[q0]);
                tc_commit(&sh.tfull[q1]);
                tc_commit(&sh.empty[st0]);
                tc_commit(&sh.empty[st1]);
            }
            for (int it = pairs ? (items & ~1) : 0; it < items && ok; ++it) {
                const int st = it % NB, buf = it % NBUF;
                if (!mbar_wait_spin(&sh.full[st], (uint32_t)((it / NB) & 1), abort, lim) ||
                    !mbar_wait_spin(&sh.tempty[buf], (uint32_t)(((it / NBUF) & 1) ^ 1), abort, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t bs = smem_desc_advance(bdesc0, st * BST);
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc_mma_bf16_ts(tmem + buf * bn, tmem + ZC + c * 32 + kk * 8,
                                       smem_desc_advance(bs, c * BCH + kk * 32), idesc_f, (c | kk) != 0);
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
        // warp set `set` takes the items of its parity (accumulators it %
        // NBUF, dl tile `set`); within a set, warp (q, g) the 32 rows of lane
        // quarter q and ids [g bn / 2, (g + 1) bn / 2) of the tile, 16 at a time
        const int ew = warp - 2, q = warp & 3, g = (ew >> 2) & 1, set = ew >> 3;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const int row = q * 32 + lane, f = row >> 6, pl = row & 63;
        const int i = j * 64 + pl;                 // position
        const int rowg = j * TR_BM + row;          // paired row
        const bool valid = i < p.P;
        float lp2 = 0.f, lq2 = 0.f, ls2 = 0.f, Apos = 0.f, Aneg = 0.f;
        if (valid && mode != TR_STATS) {
            lp2 = p.lse_p2[rowg];
            lq2 = p.lse_q2[i];
            ls2 = p.lse_s2[i];
        }
        if (valid && dzm) {
            const RowCoef rc = p.coef[rowg];
            Apos = rc.Apos;
            Aneg = rc.Aneg;
        }
        // Z into TMEM: warp (q, g, set) stores K elements 64 cb .. 64 cb + 63
        // (columns ZC + 32 cb ..) of its 32 rows, cb = 2 set + g
        {
            const int cb = 2 * set + g;
            const uint4 *src = reinterpret_cast<const uint4 *>(p.zop + (size_t)rowg * RANK + 64 * cb);
            uint32_t zr[32];
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint4 v = src[c];
                zr[4 * c] = v.x;
                zr[4 * c + 1] = v.y;
                zr[4 * c + 2] = v.z;
                zr[4 * c + 3] = v.w;
            }
            tmem_st32(tmem + lane_base + ZC + 32 * cb, zr);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.a_full);
        }
        // the anchor term's share: the teacher-forced row takes the first half
        // of each tile's ids, the consistency row the second
        const bool anchor = (f == g);
        // STATS: running (m, s); TV: 2-way partial sums of min(p, q), of the
        // part where p < q (+ half of where p = q), and of the anchor's min(p^b, q)
        float m2 = -INFINITY, s2 = 0.f;
        float r0[2] = {0.f, 0.f}, r1[2] = {0.f, 0.f}, r3[2] = {0.f, 0.f};
        bool ok = true;
        constexpr int nq = bn / 32;                // 16-id pieces per warp and tile
        for (int it = set; it < items; it += 2) {
            const int buf = it % NBUF;
            const uint32_t ph = (uint32_t)((it >> 1) & 1);      // phase of the dl tile `set`
            const int ss = it % NS;
            if (!mbar_wait_spin(&sh.tfull[buf], (uint32_t)((it / NBUF) & 1), abort, lim) ||
                !mbar_wait_spin(&sh.sfull[ss], (uint32_t)((it / NS) & 1), abort, lim)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint8_t *stile = sS + ss * SB;
            const int v0 = (vt0 + it) * bn + g * (bn / 2);
            const int nv = valid ? min(bn / 2, p.V - v0) : 0;
            uint32_t w[16];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                if (h >= nq) break;
                const int idoff = g * (bn / 2) + 16 * h;        // first id of the piece within the tile
                float acc[16];
                tmem_ld16(tmem + lane_base + buf * bn + idoff, acc);
                // the piece's 16 ids of s (and t): two 16-byte chunks of row pl
                // of the 64-id box idoff / 64
                uint4 sr[2], tr[2];
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    const int off = (idoff >> 6) * (int)TR_BOX + pl * 128 +
                                    (((((idoff & 63) >> 3) + c) ^ (pl & 7)) << 4);
                    sr[c] = *reinterpret_cast<const uint4 *>(stile + off);
                    if (mode != TR_STATS) tr[c] = *reinterpret_cast<const uint4 *>(stile + STT + off);
                }
                float sv[16], tv[16];
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    const uint32_t ws_[4] = {sr[c].x, sr[c].y, sr[c].z, sr[c].w};
                    const uint32_t wt_[4] = {tr[c].x, tr[c].y, tr[c].z, tr[c].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        sv[8 * c + 2 * e] = __uint_as_float(ws_[e] << 16);
                        sv[8 * c + 2 * e + 1] = __uint_as_float(ws_[e] & 0xFFFF0000u);
                        tv[8 * c + 2 * e] = __uint_as_float(wt_[e] << 16);
                        tv[8 * c + 2 * e + 1] = __uint_as_float(wt_[e] & 0xFFFF0000u);
                    }
                }
                const int nh = nv - 16 * h;              // ids of this piece that exist (<= 0: none)
                if (mode == TR_STATS) {
                    if (nh > 0) {
                        float x[16];
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) x[jj] = jj < nh ? (acc[jj] + sv[jj]) * L2E : -INFINITY;
                        lse2_add16(m2, s2, x);
                    }
                } else if (mode == TR_TV) {
                    if (nh >= 16) {
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) {
                            const float a2 = fmaf(acc[jj] + sv[jj], L2E, -lp2);
                            const float b2 = fmaf(tv[jj], L2E, -lq2);
                            const float m = ex2_approx(fminf(a2, b2));
                            r0[jj & 1] += m;
                            r1[jj & 1] += a2 < b2 ? m : (a2 == b2 ? 0.5f * m : 0.f);
                            if (anchor) r3[jj & 1] += ex2_approx(fminf(fmaf(sv[jj], L2E, -ls2), b2));
                        }
                    } else if (nh > 0) {
                        // the vocabulary's last tile: the same, masked
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) {
                            if (jj < nh) {
                                const float a2 = fmaf(acc[jj] + sv[jj], L2E, -lp2);
                                const float b2 = fmaf(tv[jj], L2E, -lq2);
                                const float m = ex2_approx(fminf(a2, b2));
                                r0[jj & 1] += m;
                                r1[jj & 1] += a2 < b2 ? m : (a2 == b2 ? 0.5f * m : 0.f);
                                if (anchor) r3[jj & 1] += ex2_approx(fminf(fmaf(sv[jj], L2E, -ls2), b2));
                            }
                        }
                    }
                } else {
#pragma unroll
                    for (int jj = 0; jj < 16; jj += 2) {
                        float d2[2];
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int jv = jj + e;
                            const float a2 = fmaf(acc[jv] + sv[jv], L2E, -lp2);
                            const float b2 = fmaf(tv[jv], L2E, -lq2);
                            d2[e] = jv < nh ? dl_value(a2, b2, Apos, Aneg) : 0.f;
                        }
                        w[8 * (h & 1) + jj / 2] = pack_bf16x2(d2[0], d2[1]);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&sh.tempty[buf]);
                mbar_arrive(&sh.sempty[ss]);
            }
            if (dzm) {
                if (!mbar_wait_spin(&sh.dempty[set], ph ^ 1, abort, lim)) { ok = false; break; }
                uint8_t *dt = sD + set * TR_D_BUF + row * 128;
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    *reinterpret_cast<uint4 *>(dt + (((4 * g + c) ^ (row & 7)) << 4)) =
                        make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sh.dfull[set]);
            }
        }
        if (!dzm) {
            // merge the four warps of each row (2 id groups x 2 sets), one
            // partial per (split, row); the ring is free once every item is read
            const float4 o4 = mode == TR_STATS ? make_float4(m2, s2, 0.f, 0.f)
                                               : make_float4(r0[0] + r0[1], r1[0] + r1[1], 0.f, r3[0] + r3[1]);
            tr_epi_bar();
            float4 *scr = reinterpret_cast<float4 *>(sS);
            const int slot = 2 * set + g;
            if (slot != 0) scr[(slot - 1) * TR_BM + row] = o4;
            tr_epi_bar();
            if (slot == 0 && valid && ok && !*abort) {
                float4 a = o4;
                for (int k = 0; k < 3; ++k) {
                    const float4 o = scr[k * TR_BM + row];
                    if (mode == TR_STATS) lse2_merge(a.x, a.y, o.x, o.y);
                    else { a.x += o.x; a.y += o.y; a.w += o.w; }
                }
                p.part[(size_t)sv * p.NR + rowg] = a;
            }
        } else if (ok && items > 0) {
            if (mbar_wait_spin(&sh.zdone, 0, abort, lim)) {
                tc_fence_after();
                // the 4 warps of a lane quarter take 64 of the 256 columns each
                const int c0 = (2 * set + g) * 64;
#pragma unroll 1
                for (int c4 = 0; c4 < 2; ++c4) {
                    float v[32];
                    tmem_ld32(tmem + lane_base + TR_DZ_COL + c0 + c4 * 32, v);
                    float4 *dst =
                        reinterpret_cast<float4 *>(p.dzp + ((size_t)sv * p.NR + rowg) * RANK + c0 + c4 * 32);
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

// grid (splits, NR / 128), TR_THREADS threads, TR_SMEM bytes; one kernel per
// mode.  tmap_z is not read (Z goes to tensor memory from p.zop).
__global__ void __launch_bounds__(TR_THREADS, 1)
    k_train_tok_stats(const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,
                      const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,
                      const __grid_constant__ CUtensorMap tmap_t)
{
    train_tok_body<TR_STATS>(p, tmap_w, tmap_s, tmap_t);
}
__global__ void __launch_bounds__(TR_THREADS, 1)
    k_train_tok_tv(const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,
                   const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,
                   const __grid_constant__ CUtensorMap tmap_t)
{
    train_tok_body<TR_TV>(p, tmap_w, tmap_s, tmap_t);
}
__global__ void __launch_bounds__(TR_THREADS, 1)
    k_train_tok_dz(const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,
                   const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,
                   const __grid_constant__ CUtensorMap tmap_t)
{
    train_tok_body<TR_DZ>(p, tmap_w, tmap_s, tmap_t);
}

// ---------------------------------------------------------------- k_train_voc
namespace {

constexpr int TV_BM = 128;                                 // vocabulary ids
constexpr int TV_BN = 64;                                  // rows per step: 32 positions x 2 forwards
constexpr int TV_PF = 4;                                   // steps whose s / t are prefetched into L2 ahead
constexpr int TV_EPI_WARPS = 16;                           // 2 sets (step parity) x 4 lane quarters x 2 row halves
constexpr int TV_SET = TV_EPI_WARPS / 2;
constexpr int TV_THREADS = 32 * (2 + TV_EPI_WARPS);
constexpr int TV_ZS = 4;                                   // Z ring (freed by the step's dW MMA)
constexpr int TV_SS = 3;                                   // s / t / coefficient ring (freed by the epilogue)
constexpr uint32_t TV_Z_CHUNK = TV_BN * 64 * 2;            // 8 KB: 64 rows x 64 of r
constexpr uint32_t TV_Z_BYTES = 4 * TV_Z_CHUNK;            // 32 KB
constexpr uint32_t TV_ST_BOX = 32 * 64 * 2;                // 4 KB: 32 positions x 64 ids
constexpr uint32_t TV_ST_TILE = 2 * TV_ST_BOX;             // s (or t) of 32 positions x 128 ids
constexpr uint32_t TV_INFO = TV_BN * sizeof(RowCoef);      // 1 KB
constexpr uint32_t TV_S_STAGE = 2 * TV_ST_TILE + 1024;     // s, t, row coefficients (1024-byte aligned)
constexpr uint32_t TV_D_BUF = TV_BM * TV_BN * 2;           // 16 KB: dl^T tile (K-major over rows)
constexpr uint32_t TV_IDESC_F = idesc_bf16(TV_BM, TV_BN);
constexpr uint32_t TV_IDESC_D = idesc_bf16_mn(TV_BM, RANK, false, true);
// TMEM: l^T accumulators 2 x 64 from 0, the W_r tile (A operand: 128 ids x
// 256 bf16, two per column) at 128, dW_r (256) at 256
constexpr uint32_t TV_TMEM_COLS = 512;
constexpr uint32_t TV_WR_COL = 128;
constexpr uint32_t TV_DW_COL = 256;
static_assert(TV_INFO <= 1024, "row coefficients of a step");

struct TvShared {
    uint64_t a_full, a_empty;                  // the W_r tile in TMEM: written (16 warps), read by the last F
    uint64_t zfull[TV_ZS], zempty[TV_ZS];
    uint64_t sfull[TV_SS], sempty[TV_SS];
    uint64_t tfull[2], tempty[2];
    uint64_t dfull[2], dempty[2];
    uint64_t wfull, wempty, drain;
    uint32_t tmem_base;
    int abort;
};

constexpr size_t TV_SMEM = 1024 + TV_ZS * TV_Z_BYTES + TV_SS * TV_S_STAGE + 2 * TV_D_BUF + sizeof(TvShared);
static_assert(TV_SMEM <= 232448, "k_train_voc shared memory");

}  // namespace

const size_t kTrainVocSmemBytes = TV_SMEM;
const int kTrainVocThreads = TV_THREADS;

// grid min(SMs, ceil(V / 128)) (persistent over vocabulary tiles), TV_THREADS
// threads, TV_SMEM bytes.  tmap_z: Z boxes of 32 rows; tmap_s / tmap_t: boxes
// of 64 ids x 32 positions.  tmap_w is not read (the W_r tile goes to tensor
// memory from p.W_r).
__global__ void __launch_bounds__(TV_THREADS, 1)
    k_train_voc(const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,
                const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,
                const __grid_constant__ CUtensorMap tmap_t)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sZ = base;                            // Z ring
    uint8_t *sS = sZ + TV_ZS * TV_Z_BYTES;         // s / t / coefficient ring
    uint8_t *sD = sS + TV_SS * TV_S_STAGE;         // dl^T tiles, one per warp set
    TvShared &sh = *reinterpret_cast<TvShared *>(sD + 2 * TV_D_BUF);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int nvt = (p.V + TV_BM - 1) / TV_BM;
    const int nsteps = (p.P + 31) / 32;

    if (threadIdx.x == 0) {
        mbar_init(&sh.a_full, TV_EPI_WARPS);
        mbar_init(&sh.a_empty, 1);
        for (int i = 0; i < TV_ZS; ++i) {
            mbar_init(&sh.zfull[i], 1);
            mbar_init(&sh.zempty[i], 1);               // the step's dW MMA
        }
        for (int i = 0; i < TV_SS; ++i) {
            mbar_init(&sh.sfull[i], 1);
            mbar_init(&sh.sempty[i], TV_SET);          // the step's epilogue warps
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sh.tfull[i], 1);
            mbar_init(&sh.tempty[i], TV_SET);
            mbar_init(&sh.dfull[i], TV_SET);
            mbar_init(&sh.dempty[i], 1);
        }
        mbar_init(&sh.wfull, 1);
        mbar_init(&sh.wempty, TV_EPI_WARPS);
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, TV_TMEM_COLS); tmem_relinquish(); }
    pdl_trigger();                 // the next kernel may start its set-up
    pdl_wait();                    // Z and the coefficients are complete
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
            tma_prefetch_desc(&tmap_s);
            tma_prefetch_desc(&tmap_t);
            const uint64_t once = policy_evict_first();
            const char *wr = static_cast<const char *>(p.W_r);
            auto prefetch_wr = [&](int vt) {      // a W_r tile into L2 (the epilogue loads it into TMEM)
                if (vt < nvt)
                    prefetch_l2_bulk(wr + (size_t)vt * TV_BM * RANK * 2, (uint32_t)min(TV_BM, p.V - vt * TV_BM) * RANK * 2);
            };
            // the L2 prefetch cursor of s / t runs TV_PF steps ahead of the loads
            int pf_vt = blockIdx.x, pf_u = 0;
            auto advance_pf = [&]() {
                if (pf_vt >= nvt) return;
                for (int h2 = 0; h2 < 2; ++h2) {
                    tma_prefetch_2d(&tmap_s, pf_vt * TV_BM + 64 * h2, 32 * pf_u);
                    tma_prefetch_2d(&tmap_t, pf_vt * TV_BM + 64 * h2, 32 * pf_u);
                }
                if (++pf_u == nsteps) { pf_u = 0; pf_vt += gridDim.x; }
            };
            prefetch_wr(blockIdx.x);
            for (int k = 0; k < TV_PF; ++k) advance_pf();
            int gu = 0;
            uint32_t pend_z = 0, par_z = 0, pend_s = 0, par_s = 0;
            const char *gw = reinterpret_cast<const char *>(p.gW_r);
            for (int vt = blockIdx.x; vt < nvt && !*abort; vt += gridDim.x) {
                prefetch_wr(vt + gridDim.x);
                for (int u = 0; u < nsteps && !*abort; ++u, ++gu) {
                    advance_pf();
                    if (u == max(0, nsteps - 4)) {
                        // this tile's gW_r rows (fp32, added into at the tile's end)
                        // into L2, a few steps before the drain needs them
                        const uint32_t rows = (uint32_t)min(TV_BM, p.V - vt * TV_BM);
                        for (uint32_t r0 = 0; r0 < rows; r0 += 32)
                            prefetch_l2_bulk(gw + ((size_t)vt * TV_BM + r0) * RANK * 4,
                                             min(32u, rows - r0) * RANK * 4);
                    }
                    const int jt = u >> 1, hh = u & 1;
                    const int rt = jt * 128 + 32 * hh;               // teacher-forced rows of the step
                    const int zs = gu % TV_ZS;
                    const uint32_t zph = (uint32_t)((gu / TV_ZS) & 1);
                    if (!mbar_wait_spin(&sh.zempty[zs], zph ^ 1, abort, lim)) break;
                    uint8_t *zt = sZ + zs * TV_Z_BYTES;
                    mbar_expect_tx(&sh.zfull[zs], TV_Z_BYTES);
                    for (int c = 0; c < 4; ++c) {
                        tma_load_2d(zt + c * TV_Z_CHUNK, &tmap_z, &sh.zfull[zs], c * 64, rt);
                        tma_load_2d(zt + c * TV_Z_CHUNK + 4096, &tmap_z, &sh.zfull[zs], c * 64, rt + 64);
                    }
                    pend_z |= 1u << zs;
                    par_z = (par_z & ~(1u << zs)) | (zph << zs);
                    const int ss = gu % TV_SS;
                    const uint32_t sph = (uint32_t)((gu / TV_SS) & 1);
                    if (!mbar_wait_spin(&sh.sempty[ss], sph ^ 1, abort, lim)) break;
                    uint8_t *stg = sS + ss * TV_S_STAGE;
                    mbar_expect_tx(&sh.sfull[ss], 2 * TV_ST_TILE + TV_INFO);
                    for (int h2 = 0; h2 < 2; ++h2) {
                        tma_load_2d_hint(stg + h2 * TV_ST_BOX, &tmap_s, &sh.sfull[ss], vt * TV_BM + 64 * h2, 32 * u, once);
                        tma_load_2d_hint(stg + TV_ST_TILE + h2 * TV_ST_BOX, &tmap_t, &sh.sfull[ss], vt * TV_BM + 64 * h2,
                                         32 * u, once);
                    }
                    uint8_t *info = stg + 2 * TV_ST_TILE;
                    bulk_load_1d(info, p.coef + rt, 32 * sizeof(RowCoef), &sh.sfull[ss]);
                    bulk_load_1d(info + 32 * sizeof(RowCoef), p.coef + rt + 64, 32 * sizeof(RowCoef), &sh.sfull[ss]);
                    pend_s |= 1u << ss;
                    par_s = (par_s & ~(1u << ss)) | (sph << ss);
                }
            }
            if (*abort) {
                // no copy may still be landing when the CTA leaves
                int dummy = 0;
                for (int k = 0; k < TV_ZS; ++k)
                    if (pend_z & (1u << k)) mbar_wait_spin(&sh.zfull[k], (par_z >> k) & 1, &dummy, 100000000ull);
                for (int k = 0; k < TV_SS; ++k)
                    if (pend_s & (1u << k)) mbar_wait_spin(&sh.sfull[k], (par_s >> k) & 1, &dummy, 100000000ull);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        // Issues, in order, the l^T products F(k) and the dW_r products D(k)
        // of the CTA's steps k = tile * nsteps + u, whichever is ready first:
        // F(k) needs Z(k) landed, accumulator k % 2 handed back and (first
        // step of a tile) the tile's W_r rows in TMEM; D(k) needs the dl^T
        // tile of step k and (first step of a tile) the previous tile's dW_r
        // drained.  F runs ahead of D while the epilogue works.
        if (lane == 0 && nsteps > 0) {
            const uint32_t z0 = smem_u32(sZ), d0 = smem_u32(sD);
            // descriptors formed once, advanced per MMA
            const uint64_t zdesc0 = smem_desc_sw128(z0), ddesc0 = smem_desc_sw128(d0);
            const uint64_t zmn0 = smem_desc_sw128_mn(z0, TV_Z_CHUNK);
            const int ntiles = ((int)blockIdx.x < nvt) ? (nvt - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
            const int total = ntiles * nsteps;
            int kf = 0, kd = 0;
            bool ok = true;
            unsigned long long stall0 = 0;          // when the current stall began (bounded by wait_ns)
            uint32_t spins = 0;
            while (kd < total && ok) {
                bool progressed = false;
                if (kf < total) {
                    const int lt = kf / nsteps, u = kf - lt * nsteps;
                    const int zs = kf % TV_ZS, buf = kf & 1;
                    if ((u != 0 || mbar_try_wait(&sh.a_full, (uint32_t)(lt & 1))) &&
                        mbar_try_wait(&sh.zfull[zs], (uint32_t)((kf / TV_ZS) & 1)) &&
                        mbar_try_wait(&sh.tempty[buf], (uint32_t)(((kf >> 1) & 1) ^ 1))) {
                        tc_fence_after();
                        const uint64_t zb = smem_desc_advance(zdesc0, zs * TV_Z_BYTES);
#pragma unroll
                        for (int c = 0; c < 4; ++c)
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                tc_mma_bf16_ts(tmem + buf * TV_BN, tmem + TV_WR_COL + c * 32 + kk * 8,
                                               smem_desc_advance(zb, c * TV_Z_CHUNK + kk * 32), TV_IDESC_F,
                                               (c | kk) != 0);
                        tc_commit(&sh.tfull[buf]);
                        if (u == nsteps - 1) tc_commit(&sh.a_empty);
                        ++kf;
                        progressed = true;
                    }
                }
                if (kd < kf) {
                    const int lt = kd / nsteps, u = kd - lt * nsteps;
                    const int db = kd & 1;
                    if (mbar_try_wait(&sh.dfull[db], (uint32_t)((kd >> 1) & 1)) &&
                        (u != 0 || mbar_try_wait(&sh.wempty, (uint32_t)((lt & 1) ^ 1)))) {
                        tc_fence_after();
                        const uint64_t zb = smem_desc_advance(zmn0, (kd % TV_ZS) * TV_Z_BYTES);
                        const uint64_t ds = smem_desc_advance(ddesc0, db * TV_D_BUF);
#pragma unroll
                        for (int kk = 0; kk < TV_BN / 16; ++kk)
                            tc_mma_bf16(tmem + TV_DW_COL, smem_desc_advance(ds, kk * 32), smem_desc_advance(zb, kk * 2048),
                                        TV_IDESC_D, !(u == 0 && kk == 0));
                        tc_commit(&sh.zempty[kd % TV_ZS]);
                        tc_commit(&sh.dempty[db]);
                        if (u == nsteps - 1) tc_commit(&sh.wfull);
                        ++kd;
                        progressed = true;
                    }
                }
                if (progressed) {
                    spins = 0;
                } else if ((++spins & 63u) == 0) {
                    const unsigned long long now = globaltimer();
                    if (spins == 64) stall0 = now;
                    if (*abort) ok = false;
                    else if (now - stall0 > lim) { *abort = 1; ok = false; }
                }
            }
            tc_commit(&sh.drain);
            int dummy = 0;
            mbar_wait(&sh.drain, 0, &dummy, 100000000ull);
        }
    } else {
        // ------------------------------------------------------ epilogue
        // warp set `set` takes the steps of its parity; within a set, warp
        // (q, g) the 32 ids of lane quarter q and the 32 rows of half g
        // (0 teacher-forced, 1 consistency), in two halves of 16.  At each
        // vocabulary tile every warp first stores its part of the tile's W_r
        // rows into TMEM (K block 2 set + g), then drains the previous tile's
        // dW_r (64 columns each) while the MMA starts on the new tile.
        const int ew = warp - 2, q = warp & 3, g = (ew >> 2) & 1, set = ew >> 3;
        const int cb = 2 * set + g;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const int vr = q * 32 + lane;                          // id row of the tile
        const int h2 = vr >> 6, cc = vr & 63;                  // s / t box and column within it
        const int coff = (cc & 7) * 2;
        int gu = 0, lt = 0;
        bool ok = nsteps > 0;
        // adds the dW_r rows of tile `pvt` (the lt'-th of this CTA) into gW_r
        auto drain = [&](int pvt, int plt) -> bool {
            if (!mbar_wait_spin(&sh.wfull, (uint32_t)(plt & 1), abort, lim)) return false;
            tc_fence_after();
            const int pv = pvt * TV_BM + vr;
#pragma unroll 1
            for (int c4 = 0; c4 < 4; ++c4) {
                float4 *dst = reinterpret_cast<float4 *>(p.gW_r + (size_t)pv * RANK + 64 * cb + 16 * c4);
                float4 o[4];
                if (pv < p.V) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) o[e] = dst[e];   // loads in flight before the TMEM read
                }
                float wv[16];
                tmem_ld16(tmem + lane_base + TV_DW_COL + 64 * cb + c4 * 16, wv);
                if (pv < p.V) {
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        dst[e] = make_float4(o[e].x + wv[4 * e], o[e].y + wv[4 * e + 1], o[e].z + wv[4 * e + 2],
                                             o[e].w + wv[4 * e + 3]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.wempty);
            return true;
        };
        for (int vt = blockIdx.x; vt < nvt && ok; vt += gridDim.x, ++lt) {
            const int v = vt * TV_BM + vr;
            const bool vvalid = v < p.V;
            // this tile's W_r rows into TMEM, once the previous tile's last F is done
            if (!mbar_wait_spin(&sh.a_empty, (uint32_t)((lt & 1) ^ 1), abort, lim)) { ok = false; break; }
            {
                uint32_t wrw[32];
                if (vvalid) {
                    const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.W_r) +
                                                                       (size_t)v * RANK + 64 * cb);
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const uint4 x = src[c];
                        wrw[4 * c] = x.x;
                        wrw[4 * c + 1] = x.y;
                        wrw[4 * c + 2] = x.z;
                        wrw[4 * c + 3] = x.w;
                    }
                } else {
#pragma unroll
                    for (int c = 0; c < 32; ++c) wrw[c] = 0u;
                }
                tc_fence_after();
                tmem_st32(tmem + lane_base + TV_WR_COL + 32 * cb, wrw);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sh.a_full);
            }
            if (lt > 0 && !drain(vt - (int)gridDim.x, lt - 1)) { ok = false; break; }
            for (int u = 0; u < nsteps; ++u, ++gu) {
                if ((gu & 1) != set) continue;
                const int buf = set;
                const uint32_t ph = (uint32_t)((gu >> 1) & 1);
                const int ss = gu % TV_SS;
                if (!mbar_wait_spin(&sh.tfull[buf], ph, abort, lim) ||
                    !mbar_wait_spin(&sh.sfull[ss], (uint32_t)((gu / TV_SS) & 1), abort, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint8_t *stg = sS + ss * TV_S_STAGE;
                const uint8_t *sbox = stg + h2 * TV_ST_BOX;
                const float4 *info = reinterpret_cast<const float4 *>(stg + 2 * TV_ST_TILE) + g * 32;
                uint32_t w[16];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float acc[16];
                    tmem_ld16(tmem + lane_base + buf * TV_BN + g * 32 + h * 16, acc);
#pragma unroll
                    for (int c = 0; c < 16; c += 2) {
                        float d2[2];
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int pr = 16 * h + c + e;     // position within the step
                            const int off = pr * 128 + (((cc >> 3) ^ (pr & 7)) << 4) + coff;
                            const float sv = bf2f(*reinterpret_cast<const uint16_t *>(sbox + off));
                            const float tv = bf2f(*reinterpret_cast<const uint16_t *>(sbox + TV_ST_TILE + off));
                            const float4 rc = info[pr];      // lse_p2, lse_q2, Apos, Aneg
                            const float a2 = fmaf(acc[c + e] + sv, L2E, -rc.x);
                            const float b2 = fmaf(tv, L2E, -rc.y);
                            d2[e] = vvalid ? dl_value(a2, b2, rc.z, rc.w) : 0.f;
                        }
                        w[8 * h + c / 2] = pack_bf16x2(d2[0], d2[1]);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&sh.tempty[buf]);
                    mbar_arrive(&sh.sempty[ss]);
                }
                if (!mbar_wait_spin(&sh.dempty[buf], ph ^ 1, abort, lim)) { ok = false; break; }
                uint8_t *dt = sD + buf * TV_D_BUF + vr * 128;
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    *reinterpret_cast<uint4 *>(dt + (((4 * g + c) ^ (vr & 7)) << 4)) =
                        make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sh.dfull[buf]);
            }
        }
        // the last tile's dW_r
        if (ok && lt > 0) drain(blockIdx.x + (lt - 1) * (int)gridDim.x, lt - 1);
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
