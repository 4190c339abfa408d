// kernels.h -- declarations of the kernels launched by the host code.
#pragma once

#include "common.cuh"
#include "xpress.h"

namespace xp {

// One draw of the lossless acceptance: block seq, position k (< B: the first
// rejected position, residual draw; = B: the bonus draw from p_{B+1}).
struct DrawDesc {
    int seq, k;
    float invT, lse_p, lse_q;
    int pad[3];
};

struct AcceptParams {
    int b, B, V, dtype;
    const void *target, *s;
    const int32_t *tokens;
    const float *lse, *logit_sel, *z_final, *temperature;
    const unsigned long long *seed;
    uint32_t offset;
    const void *W_r;
    int32_t *accept_len, *out_tokens;
    int32_t *status;
    Partial *rowpart;   // [b * (B + 1), chunks]
    int32_t *ticket;    // [2]: draws listed, draw CTAs done (cleared by k_acc_rows)
    DrawDesc *draws;    // [b] draws of the sampling blocks (k_acc_decide)
    unsigned long long *keys;   // [b, 2] best residual / p draw key (argmax_key), cleared by k_acc_decide
};

// refine_kernels.cu
__global__ void k_init(Params pin, Params *pdev, cudaGraphConditionalHandle handle);
__global__ void k_rowmax(const Params *pp);
__global__ void k_pre_gemm(const Params *pp, int which, int kchunk);
__global__ void k_pre_gemv(const Params *pp, int kslice);
__global__ void k_pre_mix(const Params *pp);
__global__ void k_mix_mlp(const Params *pp);
__global__ void k_read_simt(const Params *pp);
__global__ void k_reduce(const Params *pp, cudaGraphConditionalHandle handle);
__global__ void k_prof_prepare(int32_t *ctl, int32_t *act_tok, int n);
__global__ void k_build_ep(const void *W_e, const void *W_in, float *Ep, int V, int dtype);

// read_tc.cu
__global__ void k_read_tc(const Params *pp, const __grid_constant__ CUtensorMap tmap_wr,
                          const __grid_constant__ CUtensorMap tmap_z, int V);
extern const size_t kReadTcSmemBytes;
extern const int kReadTcThreads;

// read_tcv.cu (at most 32 evaluated tokens: vocabulary rows as the MMA M)
__global__ void k_read_tcv(const Params *pp, const __grid_constant__ CUtensorMap tmap_wr128,
                           const __grid_constant__ CUtensorMap tmap_z, int V, int fuse,
                           cudaGraphConditionalHandle handle);
extern const size_t kReadTcvSmemBytes;
extern const int kReadTcvThreads;
constexpr int TCV_MAX_TOKENS = 32;

// refine_small.cu (at most 32 evaluated tokens, bf16: the whole call in one
// persistent cooperative kernel of S Read CTAs + SMALL_TRANS_CTAS Trans CTAs)
__global__ void k_refine_small(const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tmap_wr128,
                               const __grid_constant__ CUtensorMap tmap_wr32, const __grid_constant__ CUtensorMap tmap_z);
__global__ void k_fold_hidden(const uint16_t *W_h, const uint16_t *W_g, const uint16_t *W_in, uint16_t *Fhl, int H);
__global__ void k_pack_L(const uint16_t *L, uint16_t *Lpk, int B);
extern const size_t kRefineSmallSmemBytes;
constexpr int SMALL_TRANS_CTAS = 8;

// trans_tc.cu (bf16, more than 32 tokens: Fuse + Mix, then Trans on tcgen05)
__global__ void k_mix_c(const Params *pp);
__global__ void k_trans_tc(const Params *pp, const __grid_constant__ CUtensorMap tmap_a,
                           const __grid_constant__ CUtensorMap tmap_b, int K, int mode);
extern const size_t kTransTcSmemBytes;

// pre_tc.cu (bf16, more than 32 tokens: the hidden projection on tcgen05)
__global__ void k_pre_tc(const Params *pp, const __grid_constant__ CUtensorMap tmap_h,
                         const __grid_constant__ CUtensorMap tmap_wh, const __grid_constant__ CUtensorMap tmap_wg,
                         int kslice);
extern const size_t kPreTcSmemBytes;

// lm_head.cu (base logits s = W_lm h and Y^(0) = argmax s; NT tokens per chunk, 32 or 256)
__global__ void k_lm_head32(const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_h, int V,
                            int H, int N, uint16_t *s_out, Partial *part, int32_t *status);
__global__ void k_lm_head256(const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_h,
                             int V, int H, int N, uint16_t *s_out, Partial *part, int32_t *status);
__global__ void k_lm_head_argmax(const Partial *part, int G, int N, int32_t *argmax_out);
extern const size_t kLmHeadSmemBytes[2];
extern const int kLmHeadThreads;

// accept_kernels.cu
__global__ void k_acc_rows(AcceptParams p, int chunks);
__global__ void k_acc_decide(AcceptParams p, int chunks);
__global__ void k_acc_draw(AcceptParams p);        // bf16 refiners (tensor-core products)
__global__ void k_acc_draw_simt(AcceptParams p);   // fp32 refiners

// fp32: c and sigma(W_1 c) of up to 32 tokens in fp32; bf16: the same as
// bf16 tensor-core operands plus this CTA's share of sigma(W_1 c)
constexpr int MIX_MLP_DYN_SMEM_MAX = (MAX_B * 3 * RANK) * 4;
inline int mix_mlp_smem(int dtype)
{
    return dtype ? (32 * (RANK + 8) + 32 * (2 * RANK + 8) + 32 * (64 + 8)) * 2 : MIX_MLP_DYN_SMEM_MAX;
}
constexpr int GEMV_SMEM = 128 * 1024;

// acceptance launch shared by xpress_accept and xpress_accept_noalloc
// (xpress_host.cu); `ws` holds the scratch laid out by accept_scratch_bytes
size_t accept_scratch_bytes(const xpress_refiner *R, int b);
int refiner_device(const xpress_refiner *R);   // the device the refiner was created on
int accept_launch(const xpress_refiner *R, const xpress_accept_in *in, int32_t *accept_len, int32_t *out_tokens,
                  void *ws, size_t ws_bytes, void *stream);
constexpr int READ_SIMT_DYN_SMEM = (32 * (RANK + 1) + 8 * 32 * 33) * 4;
inline int pre_mix_smem(int B) { return (B * 2 * RANK + RANK + 32 * (2 * RANK + 1) + B * 32) * 4; }
// k_pre_mix after k_pre_tc, whose partials already carry W_in (folded): the
// block's h and g slot values of the 32 channels, and P
inline int pre_mix_smem_folded(int B) { return 3 * B * 32 * 4; }

}  // namespace xp
