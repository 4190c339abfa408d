// train_common.cuh -- device helpers of the training-step kernels
// (train_read.cu, train_gemm.cu, train_kernels.cu) on top of common.cuh:
// MN-major shared-memory descriptors, the A-from-tensor-memory MMA, TMEM
// stores and 16-column loads, a tensor-map L2 prefetch, a polling bounded
// wait and a vector reduction into global memory.
#pragma once

#include "common.cuh"

namespace xp {

// Makes this thread's ordinary shared-memory stores visible to the async proxy
// (a tcgen05.mma that reads the tile as an operand).
__device__ __forceinline__ void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Bounded wait that keeps polling with try_wait (no suspend hint): for the
// per-tile handshakes between roles, where a suspended thread wakes up
// hundreds of nanoseconds after the phase completes.
__device__ __forceinline__ bool mbar_wait_spin(uint64_t *bar, uint32_t parity, volatile int *abort,
                                               unsigned long long limit_ns = 2000000000ull)
{
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 63u) == 0) {
            if (*abort) return false;
            if (globaltimer() - t0 > limit_ns) { *abort = 1; return false; }
        }
    }
}

// L2 prefetch of the box at (x, y) of a tiled tensor map (no shared memory,
// no completion): a later TMA load of the same box then hits L2.
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap *map, int x, int y)
{
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global [%0, {%1, %2}];" ::"l"(reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y)
                 : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]^T, kind::f16: A (M rows along the TMEM
// lanes, two consecutive K elements per 32-bit column, the even one in the
// low half) read from tensor memory at column address a_tmem.
__device__ __forceinline__ void tc_mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}"
        ::"r"(d_tmem), "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Stores 32 consecutive 32-bit columns of lane (base + t) from thread t, and
// waits until the stores are done.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
          "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
          "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
          "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 32 lanes x 16 consecutive fp32 columns; thread t gets lane (base + t).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Same, with A (bit 15) and / or B (bit 16) given MN-major.
__host__ __device__ constexpr uint32_t idesc_bf16_mn(int M, int N, bool a_mn, bool b_mn)
{
    return idesc_bf16(M, N) | (a_mn ? 1u << 15 : 0u) | (b_mn ? 1u << 16 : 0u);
}

// Shared-memory matrix descriptor for an MN-major operand stored with the
// 128-byte swizzle: each 128-byte row holds 64 consecutive M (or N) elements
// of one K index, 8 consecutive K rows form a 1024-byte swizzle atom, atoms
// along K are 1024 bytes apart (stride offset) and the next 64 elements along
// M / N start `mn_stride` bytes further (leading offset).  This is the layout
// a TMA box of 64 elements (inner) x rows (outer) leaves with SWIZZLE_128B when
// the rows run along K; advancing K by 16 moves the start by 2048 bytes.
__device__ __forceinline__ uint64_t smem_desc_sw128_mn(uint32_t saddr, uint32_t mn_stride)
{
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((mn_stride >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// TMA load of a 3D box with an L2 cache policy: the readout weights viewed as
// (64 columns, rows, K chunk of 64), so that one copy brings a tile's four K
// chunks ([chunk][row][128 bytes], each chunk as a 2D box of 64 x rows would
// land).  One large copy per tile instead of four keeps the TMA unit's
// per-copy cost off the critical path.
__device__ __forceinline__ void tma_load_w3d(void *smem_dst, const CUtensorMap *map, uint64_t *bar, int row,
                                             uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
        "%3, %4}], [%5], %6;" ::"r"(smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(row), "r"(0), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}

// Adds four floats into 16-byte aligned global memory with one vector
// reduction (relaxed, GPU scope).
__device__ __forceinline__ void red_add_v4(float *dst, float a, float b, float c, float d)
{
    asm volatile("red.relaxed.gpu.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(dst), "f"(a), "f"(b), "f"(c),
                 "f"(d)
                 : "memory");
}

// Packs two floats as bf16 (round to nearest even): lo in bits 0-15.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    return (uint32_t)f2bf(lo) | ((uint32_t)f2bf(hi) << 16);
}

// The descriptor of the same operand layout `bytes` further on (a multiple of
// 16): only the start-address field (bits 0-13, address >> 4) moves, and it
// cannot overflow for shared-memory addresses below 256 KB.  One thread issues
// every MMA, so descriptors are formed once and advanced with one add per MMA.
__device__ __forceinline__ uint64_t smem_desc_advance(uint64_t desc, uint32_t bytes) { return desc + (bytes >> 4); }

}  // namespace xp
