// tcv_common.cuh -- shape constants and helpers of the small-batch Read
// (vocabulary rows as the MMA's M dimension, at most 32 token columns),
// shared by k_read_tcv and the persistent small-batch kernel.
#pragma once

#include "common.cuh"

namespace xp {

constexpr int TV_BM = 128;                    // vocabulary rows per block (MMA M)
constexpr int TV_BN = 32;                     // token columns (MMA N)
constexpr int TV_BK = 64;
constexpr int TV_KCH = RANK / TV_BK;
constexpr int TV_STAGES = 8;
constexpr int TV_NBUF = 4;
constexpr int TV_EPI_WARPS = 8;
constexpr int TV_THREADS = 32 * (2 + TV_EPI_WARPS);
constexpr uint32_t TV_A_STAGE = TV_BM * TV_BK * 2;        // 16 KB of W_r
constexpr uint32_t TV_Z_CHUNK = TV_BN * TV_BK * 2;        // 4 KB of z
constexpr uint32_t TV_Z_BYTES = TV_Z_CHUNK * TV_KCH;      // 16 KB
constexpr uint32_t TV_TMEM_COLS = TV_NBUF * TV_BN;        // 128
constexpr uint32_t TV_IDESC = idesc_bf16(TV_BM, TV_BN);

// The persistent kernel streams W_r one 128-row block (all four 64-column K
// chunks, 64 KB) per copy: a 3D tensor map (64 columns, rows, K chunk) whose
// box lands as the four 16 KB K-chunk tiles of the 2D boxes, back to back.
// Copies of 64 KB keep one issuing thread's stream well above what 16 KB
// boxes reach.
constexpr int RS_BSTAGES = TV_STAGES / TV_KCH;          // W_r blocks in flight
constexpr uint32_t RS_B_STAGE = TV_KCH * TV_A_STAGE;   // 64 KB

__device__ __forceinline__ void tma_load_3d(void *smem_dst, const CUtensorMap *map, uint64_t *bar, int x, int y, int z)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];"
        ::"r"(smem_u32(smem_dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tma_load_3d_hint(void *smem_dst, const CUtensorMap *map, uint64_t *bar, int x, int y,
                                                 int z, uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
        "%3, %4}], [%5], %6;" ::"r"(smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}

__device__ __forceinline__ void tv_epi_bar() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

__device__ __forceinline__ bool tv_epi_bar_or(bool pred)
{
    uint32_t res;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, 256, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(res)
        : "r"((uint32_t)pred)
        : "memory");
    return res != 0;
}

// s[v0 .. v0 + 31] of one token as raw bf16 pairs (zeros past V or for an
// invalid lane).
__device__ __forceinline__ void load_s_group(uint4 (&r)[4], const uint16_t *row, int v0, int V, bool valid)
{
    if (valid && v0 + GROUP <= V) {
        const uint4 *src = reinterpret_cast<const uint4 *>(row + v0);
#pragma unroll
        for (int c = 0; c < 4; ++c) r[c] = __ldg(src + c);
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

// The descriptor of the same operand layout `bytes` further on (a multiple of
// 16): only the start-address field (bits 0-13, address >> 4) moves, and it
// cannot overflow for shared-memory addresses below 256 KB.  One thread issues
// every MMA, so descriptors are formed once and advanced with one add per MMA.
__device__ __forceinline__ uint64_t smem_desc_advance(uint64_t desc, uint32_t bytes) { return desc + (bytes >> 4); }

}  // namespace xp
