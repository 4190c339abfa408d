// trans_tc.cu -- Fuse (token slot), Mix and Trans of one pass on the graph
// path for bf16 refiners with more than 32 evaluated tokens (Sec. 4.1,
// Eq. fuse / mix / mlp), the two Trans products on tcgen05.
//
//   k_mix_c     per block and 32-channel slice: e_j = E'[x_{j-1}] for the
//               block's positions, c_k = Pc_k + e_k + sum_{j<k} L_kj e_j for
//               the positions the pass evaluates; c goes to cbuf (fp32, the
//               residual of Eq. mlp) and, rounded to bf16, to zpack (the
//               W_1 operand; the W_2 kernel later overwrites it with z)
//   k_trans_tc  D = A B^T on tcgen05, M = 128 evaluated tokens, N = 32
//               output units, K = 256 (W_1) or 512 (W_2):
//                 mode 1: A = bf16(c), B = W_1 rows; u = bf16(sigma(D)) to ubuf
//                 mode 2: A = u, B = W_2 rows; z = c + D to z_final (fp32, at
//                         the token's position) and bf16(z) to zpack (the
//                         Read's operand)
// Roles of k_trans_tc (192 threads): warp 0 TMA producer (an 8-stage ring of
// A and B K-chunks), warp 1 TMEM allocator and MMA issuer, warps 2-5
// epilogue (one TMEM lane quarter each).  Tiles whose first token is past
// the pass's count exit after the dependency wait, before any copy.
#include "common.cuh"
#include "kernels.h"

namespace xp {

namespace {

constexpr int TT_BM = 128;                     // tokens (M)
constexpr int TT_BN = 32;                      // output units (N): many CTAs for a few token tiles
constexpr int TT_BK = 64;
constexpr int TT_STAGES = 8;                   // every K-chunk of W_2 (K = 512) in flight at once
constexpr uint32_t TT_A_STAGE = TT_BM * TT_BK * 2;    // 16 KB
constexpr uint32_t TT_B_STAGE = TT_BN * TT_BK * 2;    // 4 KB
constexpr uint32_t TT_STAGE = TT_A_STAGE + TT_B_STAGE;
constexpr uint32_t TT_IDESC = idesc_bf16(TT_BM, TT_BN);

struct TtShared {
    uint64_t full[TT_STAGES], empty[TT_STAGES];
    uint64_t tfull;
    uint32_t tmem_base;
    int abort;
    int n;
};

}  // namespace

const size_t kTransTcSmemBytes = 1024 + TT_STAGES * TT_STAGE + sizeof(TtShared);

// grid (8, b), 256 threads.  CTA `rank` of block s: channels [32 rank, +32).
__global__ void __launch_bounds__(256) k_mix_c(const Params *__restrict__ pp)
{
    pdl_trigger();                     // the W_1 kernel may start its prologue
    pdl_wait();                        // the previous pass (or the precompute) is complete
    const Params &p = *pp;
    const int rank = blockIdx.x, s = blockIdx.y, B = p.B;
    const SeqState st = p.st[s];
    if (!st.active) return;
    const int m = st.m, cnt = st.cnt, off = st.off;
    const int d0 = rank * 32;
    __shared__ float e[MAX_B][32];
    for (int i = threadIdx.x; i < B * 32; i += blockDim.x) {
        const int j = i / 32, dd = i % 32;
        int x = j == 0 ? p.anchor[s] : p.tokens[(size_t)s * B + j - 1];
        if (x < 0 || x >= p.V) x = 0;   // reported by k_init
        e[j][dd] = p.Ep[(size_t)x * RANK + d0 + dd];
    }
    __syncthreads();
    uint16_t *cop = static_cast<uint16_t *>(p.zpack);
    for (int i = threadIdx.x; i < cnt * 32; i += blockDim.x) {
        const int t = i / 32, dd = i % 32, k = m + 1 + t, d = d0 + dd;
        const uint16_t *lp = p.Lpk + (size_t)(k * (k - 1) / 2) * RANK + d;
        float acc = p.Pc[((size_t)s * B + k) * RANK + d] + e[k][dd];
#pragma unroll
        for (int j = 0; j < MAX_B; ++j)
            if (j < k) acc = fmaf(bf2f(lp[(size_t)j * RANK]), e[j][dd], acc);
        const size_t o = (size_t)(off + t) * RANK + d;
        p.cbuf[o] = acc;
        cop[o] = f2bf(acc);
    }
}

// grid (ceil(N / 128), units / 32), 192 threads, kTransTcSmemBytes.
__global__ void __launch_bounds__(192, 1)
    k_trans_tc(const Params *__restrict__ pp, const __grid_constant__ CUtensorMap tmap_a,
               const __grid_constant__ CUtensorMap tmap_b, int K, int mode)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    TtShared &sh = *reinterpret_cast<TtShared *>(base + TT_STAGES * TT_STAGE);
    const Params &p = *pp;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int t0 = blockIdx.x * TT_BM, n0 = blockIdx.y * TT_BN;
    const int nch = K / TT_BK;
    pdl_trigger();                     // the next kernel may start its prologue
    if (threadIdx.x == 0) {
        for (int i = 0; i < TT_STAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        mbar_init(&sh.tfull, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, TT_BN); tmem_relinquish(); }
    pdl_wait();                        // the operands of this pass are complete
    if (threadIdx.x == 0) sh.n = p.ctl[CTL_NACT];
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;
    const int n = sh.n;
    const bool live = t0 < n;          // uniform over the CTA

    if (live && warp == 0) {
        if (lane == 0) {
            tma_prefetch_desc(&tmap_a);
            tma_prefetch_desc(&tmap_b);
            uint32_t pending = 0, pend_par = 0;
            for (int c = 0; c < nch; ++c) {
                const int st = c % TT_STAGES;
                const uint32_t ph = (uint32_t)((c / TT_STAGES) & 1);
                if (!mbar_wait(&sh.empty[st], ph ^ 1, abort)) break;
                uint8_t *sa = base + st * TT_STAGE;
                mbar_expect_tx(&sh.full[st], TT_STAGE);
                tma_load_2d(sa, &tmap_a, &sh.full[st], c * TT_BK, t0);
                tma_load_2d(sa + TT_A_STAGE, &tmap_b, &sh.full[st], c * TT_BK, n0);
                pending |= 1u << st;
                pend_par = (pend_par & ~(1u << st)) | (ph << st);
            }
            // no copy may still be landing when the CTA leaves
            int dummy = 0;
            for (int st = 0; st < TT_STAGES; ++st)
                if (pending & (1u << st)) mbar_wait(&sh.full[st], (pend_par >> st) & 1, &dummy, 100000000ull);
        }
    } else if (live && warp == 1) {
        if (lane == 0) {
            bool ok = true;
            for (int c = 0; c < nch && ok; ++c) {
                const int st = c % TT_STAGES;
                if (!mbar_wait(&sh.full[st], (uint32_t)((c / TT_STAGES) & 1), abort)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a0 = smem_u32(base + st * TT_STAGE), b0 = a0 + TT_A_STAGE;
#pragma unroll
                for (int kk = 0; kk < TT_BK / 16; ++kk)
                    tc_mma_bf16(tmem, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + kk * 32), TT_IDESC,
                                (c | kk) != 0);
                tc_commit(&sh.empty[st]);
            }
            tc_commit(&sh.tfull);      // also when stopped: the epilogue must not hang
        }
    } else if (live && warp >= 2) {
        // epilogue: warp (quarter q = warp % 4) -> tokens 32 q .. +31 of the tile
        const int q = warp & 3;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const bool got = mbar_wait(&sh.tfull, 0, abort);
        if (got) {
            tc_fence_after();
            const int t = t0 + q * 32 + lane;
            const bool valid = t < n;
            int tok = 0;
            if (mode == 2 && valid) tok = p.act_tok[t];
            float *zf = p.z_final ? p.z_final : p.zbuf;
#pragma unroll
            for (int g = 0; g < TT_BN / 32; ++g) {
                float v[32];
                tmem_ld32(tmem + lane_base + g * 32, v);
                if (!valid) continue;
                const int col = n0 + g * 32;
                if (mode == 1) {
                    uint32_t w[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = (uint32_t)f2bf(act_fn(p.act, v[2 * j])) |
                               ((uint32_t)f2bf(act_fn(p.act, v[2 * j + 1])) << 16);
                    uint4 *dst = reinterpret_cast<uint4 *>(p.ubuf + (size_t)t * 2 * RANK + col);
#pragma unroll
                    for (int c = 0; c < 4; ++c) dst[c] = make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                } else {
                    const float4 *cr = reinterpret_cast<const float4 *>(p.cbuf + (size_t)t * RANK + col);
                    float4 *zr = reinterpret_cast<float4 *>(zf + (size_t)tok * RANK + col);
                    uint32_t w[16];
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const float4 cv = cr[c];
                        const float4 z = make_float4(cv.x + v[4 * c], cv.y + v[4 * c + 1], cv.z + v[4 * c + 2],
                                                     cv.w + v[4 * c + 3]);
                        zr[c] = z;
                        w[2 * c] = (uint32_t)f2bf(z.x) | ((uint32_t)f2bf(z.y) << 16);
                        w[2 * c + 1] = (uint32_t)f2bf(z.z) | ((uint32_t)f2bf(z.w) << 16);
                    }
                    uint4 *dst = reinterpret_cast<uint4 *>(static_cast<uint16_t *>(p.zpack) + (size_t)t * RANK + col);
#pragma unroll
                    for (int c = 0; c < 4; ++c) dst[c] = make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TT_BN);
    }
    if (threadIdx.x == 0 && sh.abort) set_status(p.status, ST_TIMEOUT);
}

}  // namespace xp
