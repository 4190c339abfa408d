// pre_tc.cu -- the hidden projection of Fuse on tcgen05 for large batches.
//
// U[t][o] = sum_k h[t][k] F[o][k] with F = [W_in[:, 0:r] W_h ; W_in[:, r:2r] W_g]
// (Sec. 4.1, Eq. fuse: Fuse is linear, so the h and g slots are folded through
// W_in once per refiner; g's slot is the block mean of F_g h_k, taken by the
// Fuse/Mix precompute).  F is stored as two bf16 terms hi + lo, run as a
// doubled K loop into the same accumulator: bf16 operands (exact products),
// fp32 accumulation in TMEM.  Each CTA computes one 128-token x 256-row tile
// over one K-slice and writes it as a split-K partial Upart[slice][t][o].
//
// Roles (320 threads): warp 0 TMA producer (a 4-stage ring of h and W
// K-chunks), warp 1 TMEM allocator and MMA issuer, warps 2-9 epilogue
// (tcgen05.ld, fp32 stores).  grid (ceil(N / 128), 2 (W_h, W_g), slices).
#include "common.cuh"
#include "kernels.h"

namespace xp {

namespace {

constexpr int PT_BM = 128;                    // tokens (M)
constexpr int PT_BN = 256;                    // rows of W_h or W_g (N)
constexpr int PT_BK = 64;
constexpr int PT_STAGES = 4;
constexpr uint32_t PT_A_STAGE = PT_BM * PT_BK * 2;   // 16 KB of h
constexpr uint32_t PT_B_STAGE = PT_BN * PT_BK * 2;   // 32 KB of W
constexpr uint32_t PT_STAGE = PT_A_STAGE + PT_B_STAGE;
constexpr uint32_t PT_IDESC = idesc_bf16(PT_BM, PT_BN);

struct PtShared {
    uint64_t full[PT_STAGES], empty[PT_STAGES];
    uint64_t tfull;
    uint32_t tmem_base;
    int abort;
};

}  // namespace

const size_t kPreTcSmemBytes = 1024 + PT_STAGES * PT_STAGE + sizeof(PtShared);

__global__ void __launch_bounds__(320, 1)
    k_pre_tc(const Params *__restrict__ pp, const __grid_constant__ CUtensorMap tmap_h,
             const __grid_constant__ CUtensorMap tmap_fhi, const __grid_constant__ CUtensorMap tmap_flo, int kslice)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    PtShared &sh = *reinterpret_cast<PtShared *>(base + PT_STAGES * PT_STAGE);
    const Params &p = *pp;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int t0 = blockIdx.x * PT_BM, which = blockIdx.y, ks = blockIdx.z;
    const int kb = ks * kslice, ke = min(p.H, kb + kslice);
    const int nch = (ke - kb + PT_BK - 1) / PT_BK;         // K-chunks of the slice, each taken twice (hi, lo)

    if (threadIdx.x == 0) {
        for (int i = 0; i < PT_STAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        mbar_init(&sh.tfull, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, PT_BN); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_desc(&tmap_h);
            tma_prefetch_desc(&tmap_fhi);
            tma_prefetch_desc(&tmap_flo);
            uint32_t pending = 0, pend_par = 0;
            for (int c = 0; c < 2 * nch; ++c) {
                const int st = c % PT_STAGES;
                const uint32_t ph = (uint32_t)((c / PT_STAGES) & 1);
                if (!mbar_wait(&sh.empty[st], ph ^ 1, abort)) break;
                uint8_t *sa = base + st * PT_STAGE;
                mbar_expect_tx(&sh.full[st], PT_STAGE);
                const int kc = kb + (c % nch) * PT_BK;
                tma_load_2d(sa, &tmap_h, &sh.full[st], kc, t0);
                tma_load_2d(sa + PT_A_STAGE, c < nch ? &tmap_fhi : &tmap_flo, &sh.full[st], kc, which * RANK);
                pending |= 1u << st;
                pend_par = (pend_par & ~(1u << st)) | (ph << st);
            }
            // no copy may still be landing when the CTA leaves
            int dummy = 0;
            for (int st = 0; st < PT_STAGES; ++st)
                if (pending & (1u << st)) mbar_wait(&sh.full[st], (pend_par >> st) & 1, &dummy, 100000000ull);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            bool ok = true;
            for (int c = 0; c < 2 * nch && ok; ++c) {
                const int st = c % PT_STAGES;
                if (!mbar_wait(&sh.full[st], (uint32_t)((c / PT_STAGES) & 1), abort)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a0 = smem_u32(base + st * PT_STAGE), b0 = a0 + PT_A_STAGE;
#pragma unroll
                for (int kk = 0; kk < PT_BK / 16; ++kk)
                    tc_mma_bf16(tmem, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + kk * 32), PT_IDESC,
                                (c | kk) != 0);
                tc_commit(&sh.empty[st]);
            }
            tc_commit(&sh.tfull);                  // also when stopped: the epilogue must not hang
        }
    } else {
        // epilogue: warp (quarter q = warp % 4, half h) -> tokens 32 q .. +31,
        // rows 128 h .. +127 of the tile
        const int q = warp & 3, half = (warp - 2) >> 2;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const bool got = mbar_wait(&sh.tfull, 0, abort);
        if (got) {
            tc_fence_after();
            const int t = t0 + q * 32 + lane;
            float *dst = p.Upart + ((size_t)ks * p.N + t) * 2 * RANK + which * RANK + half * 128;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float v[32];
                tmem_ld32(tmem + lane_base + half * 128 + c * 32, v);
                if (t < p.N && nch > 0) {
#pragma unroll
                    for (int j = 0; j < 32; j += 4)
                        *reinterpret_cast<float4 *>(dst + c * 32 + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                } else if (t < p.N) {
#pragma unroll
                    for (int j = 0; j < 32; j += 4)
                        *reinterpret_cast<float4 *>(dst + c * 32 + j) = make_float4(0.f, 0.f, 0.f, 0.f);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, PT_BN);
    }
    if (threadIdx.x == 0 && sh.abort) set_status(p.status, ST_TIMEOUT);
}

}  // namespace xp
