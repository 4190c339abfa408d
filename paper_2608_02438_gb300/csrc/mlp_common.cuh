// mlp_common.cuh -- warp-level helpers of the small GEMMs (hidden
// projection, Trans) shared by the multi-kernel path and the persistent
// small-batch kernel.
#pragma once

#include "common.cuh"

namespace xp {

// Sum over the 32 lanes of v[0..31] (one value per token), scattered so that
// lane t ends with the total of token t in v[0] (recursive halving, 31 shuffles).
__device__ __forceinline__ float reduce_scatter32(float (&v)[32], int lane)
{
#pragma unroll
    for (int s = 16; s >= 1; s >>= 1) {
        const bool upper = (lane & s) != 0;
#pragma unroll
        for (int j = 0; j < s; ++j) {
            const float send = upper ? v[j] : v[j + s];
            const float keep = upper ? v[j + s] : v[j];
            v[j] = keep + __shfl_xor_sync(0xffffffffu, send, s);
        }
    }
    return v[0];
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4 &w, float (&x)[8])
{
    const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        x[2 * q] = __uint_as_float(ww[q] << 16);
        x[2 * q + 1] = __uint_as_float(ww[q] & 0xFFFF0000u);
    }
}

// D (16x8, fp32) += A (16x16, bf16, row-major) * B (16x8, bf16, column-major):
// the m16n8k16 warp-level tensor-core product (used for the small Trans GEMMs;
// the vocabulary readout uses tcgen05).
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

constexpr int COP_LD = RANK + 8;        // bf16 row strides of the A operands in
constexpr int UOP_LD = 2 * RANK + 8;    // shared memory (8-row fragments hit distinct banks)
constexpr int UOWN_LD = 64 + 8;

// Trans on tensor cores for bf16 refiners (operands are bf16 by the precision
// contract).  Tokens are the M dimension (two 16-row tiles cover up to 32),
// W_1 / W_2 rows the N dimension, features the K dimension.
// Tensor-core operand fragments of the CTA's W_1 / W_2 rows (static weights,
// fetched before the kernel waits for its predecessor): warp w owns W_1 rows
// [64 rank + 8 w, +8) and W_2 rows [32 rank + 8 (w % 4), +8) over K half w / 4.
struct MlpFrags {
    uint32_t b1[RANK / 16][2], b2[RANK / 16][2];
};

__device__ __forceinline__ void load_mlp_frags(const Params &p, int rank, MlpFrags &f)
{
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32, g = lane >> 2, tq = lane & 3;
    const uint32_t *w1row = reinterpret_cast<const uint32_t *>(static_cast<const uint16_t *>(p.W1) +
                                                               (size_t)(rank * 64 + 8 * warp + g) * RANK);
    const uint32_t *w2row = reinterpret_cast<const uint32_t *>(static_cast<const uint16_t *>(p.W2) +
                                                               (size_t)(rank * 32 + 8 * (warp & 3) + g) * 2 * RANK);
    const int khalf = warp >> 2;
#pragma unroll
    for (int ks = 0; ks < RANK / 16; ++ks) {
        f.b1[ks][0] = __ldg(w1row + ks * 8 + tq);
        f.b1[ks][1] = __ldg(w1row + ks * 8 + 4 + tq);
        const int kk = khalf * (RANK / 16) + ks;
        f.b2[ks][0] = __ldg(w2row + kk * 8 + tq);
        f.b2[ks][1] = __ldg(w2row + kk * 8 + 4 + tq);
    }
}

}  // namespace xp
