// train_gemm.cu -- the dense products of the refiner training step (Sec. 4.3)
// other than the Read: the projections of Fuse (W_h h, W_g h, W_in [..]) and
// Trans (W_1, W_2) forward, and their input and weight gradients backward.
//
// D[M, N] = A[M, K] B[N, K]^T on tcgen05, tile 128 x 64, K in chunks of 64
// through a 6-stage TMA ring.  Each operand is either K-major (its rows run
// along M or N, as a weight or an activation used as is) or MN-major (its rows
// run along K: an activation read transposed for a weight gradient, or a
// weight read transposed for an input gradient); an MN-major tile is two (A)
// or one (B) TMA boxes of 64 elements x 64 K rows, read with the MN-major
// shared-memory descriptor, so no transposed copy is ever made.
// grid.z splits K; split products are added atomically (GM_ADD) or stored
// one slice per split (GM_PART) for a reduction in a fixed order.
//
// Roles (192 threads): warp 0 TMA producer, warp 1 TMEM allocator and MMA
// issuer, warps 2-5 epilogue (one TMEM lane quarter each, 32 rows).
#include "train_common.cuh"
#include "kernels.h"

namespace xp {

namespace {

constexpr int G_BM = 128, G_BN = 64, G_BK = 64, G_STAGES = 6;
constexpr uint32_t G_A_STAGE = G_BM * G_BK * 2;   // 16 KB
constexpr uint32_t G_B_STAGE = G_BN * G_BK * 2;   // 8 KB
constexpr uint32_t G_STAGE = G_A_STAGE + G_B_STAGE;

struct GShared {
    uint64_t full[G_STAGES], empty[G_STAGES];
    uint64_t tfull;
    uint32_t tmem_base;
    int abort;
};

}  // namespace

const size_t kGemmSmemBytes = 1024 + G_STAGES * G_STAGE + sizeof(GShared);

// grid (ceil(M / 128), ceil(N / 64), K splits), 192 threads, kGemmSmemBytes.
// ta: A K-major [M][K] boxes {64, 128}, or MN-major [K][M] boxes {64, 64};
// tb: B K-major [N][K] or MN-major [K][N], boxes {64, 64}.
__global__ void __launch_bounds__(192, 1)
    k_gemm(const __grid_constant__ GemmArgs g, const __grid_constant__ CUtensorMap ta,
           const __grid_constant__ CUtensorMap tb)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    GShared &sh = *reinterpret_cast<GShared *>(base + G_STAGES * G_STAGE);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int m0 = blockIdx.x * G_BM, n0 = blockIdx.y * G_BN;
    const int nk = (g.K + G_BK - 1) / G_BK;
    const int kc0 = blockIdx.z * g.kchunks, kc1 = min(nk, kc0 + g.kchunks);
    const int nc = kc1 - kc0;
    const uint32_t idesc = idesc_bf16_mn(G_BM, G_BN, g.a_mn != 0, g.b_mn != 0);

    if (threadIdx.x == 0) {
        for (int i = 0; i < G_STAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        mbar_init(&sh.tfull, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, G_BN); tmem_relinquish(); }
    if (threadIdx.x == 0) {
        tma_prefetch_desc(&ta);
        tma_prefetch_desc(&tb);
    }
    pdl_trigger();                 // the next kernel may start its set-up
    pdl_wait();                    // the operands of this product are complete
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;

    if (warp == 0) {
        if (lane == 0 && nc > 0) {
            uint32_t pending = 0, pend_par = 0;
            for (int c = 0; c < nc; ++c) {
                const int st = c % G_STAGES;
                const uint32_t ph = (uint32_t)((c / G_STAGES) & 1);
                if (!mbar_wait_spin(&sh.empty[st], ph ^ 1, abort)) break;
                uint8_t *sa = base + st * G_STAGE, *sb = sa + G_A_STAGE;
                const int k = (kc0 + c) * G_BK;
                mbar_expect_tx(&sh.full[st], G_STAGE);
                if (g.a_mn) {
                    tma_load_2d(sa, &ta, &sh.full[st], m0, k);
                    tma_load_2d(sa + G_A_STAGE / 2, &ta, &sh.full[st], m0 + 64, k);
                } else {
                    tma_load_2d(sa, &ta, &sh.full[st], k, m0);
                }
                if (g.b_mn) tma_load_2d(sb, &tb, &sh.full[st], n0, k);
                else tma_load_2d(sb, &tb, &sh.full[st], k, n0);
                pending |= 1u << st;
                pend_par = (pend_par & ~(1u << st)) | (ph << st);
            }
            if (*abort) {
                int dummy = 0;
                for (int st = 0; st < G_STAGES; ++st)
                    if (pending & (1u << st)) mbar_wait_spin(&sh.full[st], (pend_par >> st) & 1, &dummy, 100000000ull);
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && nc > 0) {
            bool ok = true;
            for (int c = 0; c < nc && ok; ++c) {
                const int st = c % G_STAGES;
                if (!mbar_wait_spin(&sh.full[st], (uint32_t)((c / G_STAGES) & 1), abort)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a0 = smem_u32(base + st * G_STAGE), b0 = a0 + G_A_STAGE;
#pragma unroll
                for (int kk = 0; kk < G_BK / 16; ++kk) {
                    const uint64_t ad = g.a_mn ? smem_desc_sw128_mn(a0 + kk * 2048, G_A_STAGE / 2)
                                               : smem_desc_sw128(a0 + kk * 32);
                    const uint64_t bd = g.b_mn ? smem_desc_sw128_mn(b0 + kk * 2048, G_B_STAGE)
                                               : smem_desc_sw128(b0 + kk * 32);
                    tc_mma_bf16(tmem, ad, bd, idesc, (c | kk) != 0);
                }
                tc_commit(&sh.empty[st]);
            }
            tc_commit(&sh.tfull);          // also when stopped: the epilogue must not hang
        }
    } else if (nc > 0) {
        const int q = warp & 3;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        if (mbar_wait_spin(&sh.tfull, 0, abort)) {
            tc_fence_after();
            const int m = m0 + q * 32 + lane;
            const bool valid = m < g.M && !*abort;
#pragma unroll 1
            for (int grp = 0; grp < G_BN / 32; ++grp) {
                float v[32];
                tmem_ld32(tmem + lane_base + grp * 32, v);
                const int n = n0 + grp * 32;
                if (!valid || n >= g.N) continue;
                const int nv = min(32, g.N - n);
                if (g.mode == GM_ADD) {
                    float *dst = g.C + (size_t)m * g.ldc + n;
                    if (nv == 32 && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            red_add_v4(dst + 4 * e, g.alpha * v[4 * e], g.alpha * v[4 * e + 1], g.alpha * v[4 * e + 2],
                                       g.alpha * v[4 * e + 3]);
                    } else {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj)
                            if (jj < nv) atomicAdd(dst + jj, g.alpha * v[jj]);
                    }
                    continue;
                }
                float x[32];
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) x[jj] = (g.mode == GM_STORE || g.mode == GM_PART) ? g.alpha * v[jj] : v[jj];
                if (g.mode == GM_RESID) {
                    const float *rr = g.R + (size_t)m * g.ldr + n;
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj)
                        if (jj < nv) x[jj] += rr[jj];
                }
                if (g.C) {
                    float *dst = g.C + (size_t)m * g.ldc + n;
                    if (g.mode == GM_PART) dst += (size_t)blockIdx.z * g.M * g.ldc;
                    if (nv == 32) {
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            reinterpret_cast<float4 *>(dst)[e] =
                                make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
                    } else {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj)
                            if (jj < nv) dst[jj] = x[jj];
                    }
                }
                if (g.Cb) {
                    uint16_t *dst = g.Cb + (size_t)m * g.ldcb + n;
                    if (g.mode == GM_ACT) {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj) x[jj] = act_fn(g.act, x[jj]);
                    }
                    if (nv == 32) {
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            reinterpret_cast<uint4 *>(dst)[e] =
                                make_uint4(pack_bf16x2(x[8 * e], x[8 * e + 1]), pack_bf16x2(x[8 * e + 2], x[8 * e + 3]),
                                           pack_bf16x2(x[8 * e + 4], x[8 * e + 5]),
                                           pack_bf16x2(x[8 * e + 6], x[8 * e + 7]));
                    } else {
#pragma unroll
                        for (int jj = 0; jj < 32; ++jj)
                            if (jj < nv) dst[jj] = f2bf(x[jj]);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, G_BN);
    }
}

}  // namespace xp
