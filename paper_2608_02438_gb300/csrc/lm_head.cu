// lm_head.cu -- the drafter's base logits s = W_lm h (Sec. 4.1, Fig. 2a: the
// target-sized LM head that produces s_k before the refiner) with Algorithm
// 1's Y^(0) = argmax_v s_k,v fused into the epilogue.
//
// GEMM view: D[v, t] = W_lm[v, :] . h[t, :], M = 128 vocabulary rows (the
// weight stream, 1.245 GB at the Qwen3-8B shape), N = NT tokens (a chunk of
// the N hidden states), K = H.  Vocabulary rows sit in TMEM lanes, so the
// stores of s are runs of 64 bytes per token and the weight stream is read
// exactly once per token chunk.  Work items are (token chunk, 128-row
// vocabulary tile), dealt round-robin over a persistent grid of G CTAs
// (G <= the number of vocabulary tiles, so every CTA meets every chunk).
//
// Roles (192 threads):
//   warp 0     TMA producer: per K-chunk of 64, a 128 x 64 box of W_lm and an
//              NT x 64 box of h (rows past V or N read as zero), into a ring
//   warp 1     TMEM allocator and tcgen05.mma issuer (one thread); two
//              accumulators of NT columns, so that the epilogue of one item
//              overlaps the MMAs of the next
//   warps 2-5  epilogue: tcgen05.ld of 32 token columns of its lane quarter,
//              rounding to bf16 (the stored s), the stores of s, and per token
//              the running argmax over the rows this warp has seen in the
//              current chunk (a 32 x 32 transpose through shared memory, so
//              that lane t reduces token t)
// Every CTA leaves one (max, id) partial per token of every chunk; the
// second kernel combines the G partials of each token (ties: smallest id).
#include "common.cuh"
#include "kernels.h"

namespace xp {

namespace {

constexpr int LM_BM = 128;
constexpr int LM_BK = 64;
constexpr int LM_EPI_WARPS = 4;
constexpr int LM_THREADS = 32 * (2 + LM_EPI_WARPS);
constexpr uint32_t LM_A_STAGE = LM_BM * LM_BK * 2;        // 16 KB of W_lm

template <int NT>
struct LmShape {
    static constexpr uint32_t B_STAGE = NT * LM_BK * 2;
    static constexpr uint32_t STAGE = LM_A_STAGE + B_STAGE;
    static constexpr int STAGES = NT <= 32 ? 8 : 4;
    static constexpr uint32_t TMEM_COLS = 2 * NT < 32 ? 32 : 2 * NT;   // NT in {32, 256}: a power of two
    static constexpr uint32_t IDESC = idesc_bf16(LM_BM, NT);
    static constexpr size_t TILE_BYTES = LM_EPI_WARPS * 32 * 33 * 4;        // per-warp transposes
    static constexpr size_t WBEST_BYTES = LM_EPI_WARPS * NT * sizeof(Partial);  // per-warp partials of a chunk
    static constexpr size_t SMEM = 1024 + (size_t)STAGES * STAGE + TILE_BYTES + WBEST_BYTES + 1024;
};

struct LmBars {
    uint64_t full[8], empty[8];
    uint64_t tfull[2], tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ void lm_epi_bar() { asm volatile("bar.sync 1, %0;" ::"n"(LM_EPI_WARPS * 32) : "memory"); }

__device__ __forceinline__ bool better(float v, int i, float bv, int bi) { return v > bv || (v == bv && i < bi); }

}  // namespace

// grid G (<= vocabulary tiles), LM_THREADS threads, LmShape<NT>::SMEM bytes.
template <int NT>
__device__ __forceinline__ void lm_head_body(const CUtensorMap &tmap_w, const CUtensorMap &tmap_h, int V, int H, int N,
                                             uint16_t *s_out, Partial *part, int32_t *status)
{
    using Sh = LmShape<NT>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    float (*tile)[32][33] = reinterpret_cast<float (*)[32][33]>(base + Sh::STAGES * Sh::STAGE);
    Partial (*wbest)[NT] = reinterpret_cast<Partial (*)[NT]>(base + Sh::STAGES * Sh::STAGE + Sh::TILE_BYTES);
    LmBars &sh = *reinterpret_cast<LmBars *>(base + Sh::STAGES * Sh::STAGE + Sh::TILE_BYTES + Sh::WBEST_BYTES);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int G = gridDim.x, r = blockIdx.x;
    const int NVT = (V + LM_BM - 1) / LM_BM, NC = (N + NT - 1) / NT, KCH = (H + LM_BK - 1) / LM_BK;
    const int items = NVT * NC;                              // item i: chunk i / NVT, tile i % NVT

    if (threadIdx.x == 0) {
        for (int i = 0; i < Sh::STAGES; ++i) { mbar_init(&sh.full[i], 1); mbar_init(&sh.empty[i], 1); }
        for (int i = 0; i < 2; ++i) { mbar_init(&sh.tfull[i], 1); mbar_init(&sh.tempty[i], LM_EPI_WARPS); }
        mbar_init(&sh.drain, 1);
        sh.abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) { tmem_alloc(&sh.tmem_base, Sh::TMEM_COLS); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem_base;
    volatile int *abort = &sh.abort;

    if (warp == 0) {
        // ------------------------------------------------------- producer
        if (lane == 0) {
            tma_prefetch_desc(&tmap_w);
            tma_prefetch_desc(&tmap_h);
            const uint64_t once = policy_evict_first();     // W_lm is read once per chunk
            int stage = 0;
            uint32_t phase = 0, pending = 0, pend_par = 0;
            bool ok = true;
            for (int it = r; it < items && ok; it += G) {
                const int chunk = it / NVT, vt = it % NVT;
                for (int kc = 0; kc < KCH; ++kc) {
                    if (!mbar_wait(&sh.empty[stage], phase ^ 1, abort)) { ok = false; break; }
                    uint8_t *dst = base + stage * Sh::STAGE;
                    mbar_expect_tx(&sh.full[stage], Sh::STAGE);
                    tma_load_2d_hint(dst, &tmap_w, &sh.full[stage], kc * LM_BK, vt * LM_BM, once);
                    tma_load_2d(dst + LM_A_STAGE, &tmap_h, &sh.full[stage], kc * LM_BK, chunk * NT);
                    pending |= 1u << stage;
                    pend_par = (pend_par & ~(1u << stage)) | (phase << stage);
                    if (++stage == Sh::STAGES) { stage = 0; phase ^= 1; }
                }
            }
            // no copy may still be landing when the CTA leaves
            int dummy = 0;
            for (int st = 0; st < Sh::STAGES; ++st)
                if (pending & (1u << st)) mbar_wait(&sh.full[st], (pend_par >> st) & 1, &dummy, 100000000ull);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            int stage = 0, t = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int it = r; it < items && ok; it += G, ++t) {
                const int buf = t & 1;
                if (!mbar_wait(&sh.tempty[buf], ((t >> 1) & 1) ^ 1, abort)) break;
                tc_fence_after();
                const uint32_t d = tmem + buf * NT;
                for (int kc = 0; kc < KCH; ++kc) {
                    if (!mbar_wait(&sh.full[stage], phase, abort)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(base + stage * Sh::STAGE), b0 = a0 + LM_A_STAGE;
#pragma unroll
                    for (int kk = 0; kk < LM_BK / 16; ++kk)
                        tc_mma_bf16(d, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + kk * 32), Sh::IDESC,
                                    (kc | kk) != 0);
                    tc_commit(&sh.empty[stage]);
                    if (++stage == Sh::STAGES) { stage = 0; phase ^= 1; }
                }
                if (ok) tc_commit(&sh.tfull[buf]);
            }
            tc_commit(&sh.drain);
            int dummy = 0;
            mbar_wait(&sh.drain, 0, &dummy, 100000000ull);
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int ew = warp - 2, q = warp & 3;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        float (*tp)[33] = tile[ew];
        float bv[NT / 32];
        int bi[NT / 32];
#pragma unroll
        for (int g = 0; g < NT / 32; ++g) { bv[g] = -INFINITY; bi[g] = 0x7fffffff; }
        int t = 0, cur_chunk = -1;
        for (int it = r;; it += G, ++t) {
            const bool more = it < items;
            const int chunk = more ? it / NVT : -1, vt = it % NVT;
            if (chunk != cur_chunk && cur_chunk >= 0) {
                // the chunk is done in this CTA: its partial per token
#pragma unroll
                for (int g = 0; g < NT / 32; ++g) wbest[ew][g * 32 + lane] = Partial{bv[g], bi[g], 0.0f, 0.0f};
                lm_epi_bar();
                for (int j = threadIdx.x - 64; j < NT; j += LM_EPI_WARPS * 32) {
                    const int tok = cur_chunk * NT + j;
                    if (tok < N) {
                        Partial a = wbest[0][j];
                        for (int w = 1; w < LM_EPI_WARPS; ++w)
                            if (better(wbest[w][j].best, wbest[w][j].idx, a.best, a.idx)) a = wbest[w][j];
                        part[(size_t)tok * G + r] = a;
                    }
                }
                lm_epi_bar();
#pragma unroll
                for (int g = 0; g < NT / 32; ++g) { bv[g] = -INFINITY; bi[g] = 0x7fffffff; }
            }
            if (!more) break;
            cur_chunk = chunk;
            const int buf = t & 1;
            const bool got = mbar_wait(&sh.tfull[buf], (t >> 1) & 1, abort);
            tc_fence_after();
            const int row = vt * LM_BM + q * 32 + lane;           // this thread's vocabulary row
#pragma unroll 1
            for (int g = 0; g < NT / 32; ++g) {
                float v[32];
                if (got) tmem_ld32(tmem + lane_base + buf * NT + g * 32, v);
                else
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = 0.0f;
                const int tok0 = chunk * NT + g * 32;
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const uint16_t b = f2bf(v[j]);
                    if (s_out && row < V && tok0 + j < N) s_out[(size_t)(tok0 + j) * V + row] = b;
                    tp[j][lane] = row < V ? bf2f(b) : -INFINITY;       // [token][row of the quarter]
                }
                __syncwarp();
                // lane j: token tok0 + j over this quarter's 32 rows (ascending ids)
                float m = -INFINITY;
                int mi = 0x7fffffff;
#pragma unroll
                for (int rr = 0; rr < 32; ++rr) {
                    const float x = tp[lane][rr];
                    if (x > m) { m = x; mi = vt * LM_BM + q * 32 + rr; }
                }
                if (better(m, mi, bv[g], bi[g])) { bv[g] = m; bi[g] = mi; }
                __syncwarp();
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.tempty[buf]);
            if (!got) break;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, Sh::TMEM_COLS);
    }
    if (threadIdx.x == 0 && sh.abort) set_status(status, ST_TIMEOUT);
    pdl_trigger();
}

// grid ceil(N / 8), 256 threads: warp w combines the G partials of token
// 8 blockIdx.x + w (ties: the smallest id).
__global__ void __launch_bounds__(256) k_lm_head_argmax(const Partial *part, int G, int N, int32_t *argmax_out)
{
    pdl_wait();
    const int tok = blockIdx.x * 8 + threadIdx.x / 32, lane = threadIdx.x % 32;
    if (tok >= N) return;
    float m = -INFINITY;
    int mi = 0x7fffffff;
    for (int c = lane; c < G; c += 32) {
        const Partial a = part[(size_t)tok * G + c];
        if (better(a.best, a.idx, m, mi)) { m = a.best; mi = a.idx; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, m, o);
        const int oi = __shfl_xor_sync(0xffffffffu, mi, o);
        if (better(om, oi, m, mi)) { m = om; mi = oi; }
    }
    if (lane == 0) argmax_out[tok] = mi;
}

__global__ void __launch_bounds__(LM_THREADS, 1)
    k_lm_head32(const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_h, int V, int H,
                int N, uint16_t *s_out, Partial *part, int32_t *status)
{
    lm_head_body<32>(tmap_w, tmap_h, V, H, N, s_out, part, status);
}

__global__ void __launch_bounds__(LM_THREADS, 1)
    k_lm_head256(const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_h, int V, int H,
                 int N, uint16_t *s_out, Partial *part, int32_t *status)
{
    lm_head_body<256>(tmap_w, tmap_h, V, H, N, s_out, part, status);
}

const size_t kLmHeadSmemBytes[2] = {LmShape<32>::SMEM, LmShape<256>::SMEM};
const int kLmHeadThreads = LM_THREADS;

}  // namespace xp
