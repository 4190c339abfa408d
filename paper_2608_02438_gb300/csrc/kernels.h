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
    unsigned long long *keys;   // [b, 2] best residual / p draw key (argmax_key), cleared by k_acc_rows
    int chunks;         // vocabulary chunks per target row (k_acc_rows)
    int fused;          // 1: no k_acc_decide; every k_acc_draw CTA takes the decisions itself (b <= 8)
};
constexpr int ACCEPT_FUSED_MAX_B = 8;       // batches up to this size skip k_acc_decide

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
__global__ void k_refine_small(const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tmap_wrb,
                               const __grid_constant__ CUtensorMap tmap_wr32, const __grid_constant__ CUtensorMap tmap_z,
                               const __grid_constant__ CUtensorMap tmap_f, const __grid_constant__ CUtensorMap tmap_h);
__global__ void k_fold_hidden(const uint16_t *W_h, const uint16_t *W_g, const uint16_t *W_in, uint16_t *Fhl, int H);
__global__ void k_pack_L(const uint16_t *L, uint16_t *Lpk, int B);
extern const size_t kRefineSmallSmemBytes;
constexpr int SMALL_TRANS_CTAS = 8;
constexpr int SMALL_PC_KT = 8;              // 64-wide K tiles per precompute copy of the persistent kernel

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
__global__ void k_acc_decide(AcceptParams p);
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

// ------------------------------------------------------------ training step
// Per paired row of the training step (Sec. 4.3): row 128 j + f 64 + l is
// position 64 j + l under the teacher-forced (f = 0) or the consistency (f = 1)
// inputs.  dL/dl_v = p_v A(sgn(p_v - q_v)) - A2 [v = y*] with p, q the row's
// and its position's target softmax, A(+1) = Apos, A(-1) = Aneg,
// A(0) = (Apos + Aneg) / 2; the vocabulary passes apply the first term, the
// -A2 [v = y*] term is applied to dz and dW_r by k_train_dz.  Zero on padding
// rows.
struct alignas(16) RowCoef {
    float lse_p2, lse_q2;   // log2-domain log-sum-exp of the row's logits and of the target row
    float Apos, Aneg;
};

constexpr int TR_STATS = 0, TR_TV = 1, TR_DZ = 2;

struct TrainParams {
    int P, NR, V, B;        // positions, paired rows (multiple of 128), vocabulary, block
    int nvt, splits;        // 64-id vocabulary tiles, splits of them (k_train_tok grid.x)
    const int32_t *ystar;   // [P]
    float4 *part;           // [splits][NR] per-row partials of the statistics passes
    float *dzp;             // [splits][NR][r] dL/dz of each vocabulary split
    float *ly;              // [NR] l at y*
    const float *lse_p2;    // [NR]
    const float *lse_q2;    // [P]
    const float *lse_s2;    // [P]
    const RowCoef *coef;    // [NR]
    float *gW_r;            // [V][r] dL/dW_r, added into
    const void *W_r;
    const uint16_t *zop;    // [NR][r] the W_r operand z of every row (bf16)
    int32_t *status;
    unsigned long long wait_ns;
};

// train_read.cu
// k_train_tok_{stats, tv, dz}: the token-major kernel in its three modes
#define XP_TRAIN_TOK_ARGS                                                                                     \
    const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,                        \
        const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,               \
        const __grid_constant__ CUtensorMap tmap_t
__global__ void k_train_tok_stats(XP_TRAIN_TOK_ARGS);
__global__ void k_train_tok_tv(XP_TRAIN_TOK_ARGS);
__global__ void k_train_tok_dz(XP_TRAIN_TOK_ARGS);
#undef XP_TRAIN_TOK_ARGS
__global__ void k_train_voc(const __grid_constant__ TrainParams p, const __grid_constant__ CUtensorMap tmap_z,
                            const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_s,
                            const __grid_constant__ CUtensorMap tmap_t);
extern const size_t kTrainTokSmemBytes, kTrainVocSmemBytes;
extern const int kTrainTokThreads, kTrainVocThreads;

// train_gemm.cu: C (+)= alpha A B^T on tcgen05, A [M, K] and B [N, K] bf16 given
// K-major (rows along M / N) or MN-major (rows along K)
constexpr int GM_STORE = 0, GM_ADD = 1, GM_ACT = 2, GM_RESID = 3, GM_PART = 4;
struct GemmArgs {
    int M, N, K;
    int a_mn, b_mn;         // 1: the operand's rows run along K
    int kchunks;            // 64-wide K chunks per grid.z slice
    int mode;               // GM_STORE: C = alpha D; GM_ADD: C += alpha D (atomic);
                            // GM_ACT: C = D, Cb = bf16(sigma(D)); GM_RESID: x = R + D, C = x, Cb = bf16(x);
                            // GM_PART: slice z of C (C + z M ldc) = alpha D of K split z (summed later
                            // in a fixed order, so that the result is reproducible)
    int act;
    float alpha;
    float *C;
    int ldc;
    uint16_t *Cb;
    int ldcb;
    const float *R;
    int ldr;
};
__global__ void k_gemm(const __grid_constant__ GemmArgs g, const __grid_constant__ CUtensorMap ta,
                       const __grid_constant__ CUtensorMap tb);
extern const size_t kGemmSmemBytes;

// train_kernels.cu
struct TrainMisc {
    int b, B, P, NR, V, H, act;
    const void *h, *s, *t;                  // [P, H], [P, V], [P, V] bf16
    const int32_t *ystar, *anchor, *xhat_in;
    const uint16_t *W_e, *L;
    float a_ce, a_l1, gamma, lambda, beta;
    int nch;                                // vocabulary chunks of k_train_rows
    float4 *rpart;                          // [P][nch] max / log2-sum of s and of t
    unsigned long long *rkey;               // [P][nch] argmax key of s
    float *lse_s2, *lse_q2, *s_y;           // [P]
    int32_t *xhat;                          // [P] first argmax of s rows
    int32_t *xrow;                          // [NR] input token of each paired row
    const float *Uh, *Ug;                   // [usplits][P, r] W_h h_k, W_g h_k per K split
    int usplits;
    uint16_t *X;                            // [NR, 3r] bf16 [u_h | u_g | W_e x]
    uint16_t *Xlo;                          // [NR, 2r] bf16 [u_h - bf16(u_h) | u_g - bf16(u_g)]
    const float *a;                         // [NR, r]
    float *c;                               // [NR, r]
    uint16_t *cop;                          // [NR, r] bf16(c)
    const float4 *part;                     // [splits][NR]
    int splits;
    float *ly, *lse_p2;                     // [NR]
    RowCoef *coef;                          // [NR]
    float *A2;                              // [NR] coefficient of the -[v = y*] term
    const uint16_t *W_r, *zop;              // [V, r], [NR, r]
    float *gW_r;
    float *loss;                            // [b, 4]
    const float *dzp;                       // [splits][NR, r] per vocabulary split
    float *dz;                              // [NR, r]
    uint16_t *dzb;                          // [NR, r]
    const float *du, *tpre;                 // [NR, 2r] dL/du, W_1 c
    uint16_t *dtb;                          // [NR, 2r]
    const float *dc;                        // [NR, r]
    uint16_t *dab;                          // [NR, r]
    float *gL, *gW_e;
    const float *dX;                        // [NR, 3r]
    uint16_t *D;                            // [P, 2r] bf16 [dL/du_h | dL/du_g / B]
    int32_t *status;
};
__global__ void k_train_rows(TrainMisc m);
__global__ void k_train_rows_fin(TrainMisc m);
__global__ void k_train_fuse(TrainMisc m);
__global__ void k_train_mix(TrainMisc m);
__global__ void k_train_stats_fin(TrainMisc m);
__global__ void k_train_tv_fin(TrainMisc m);
__global__ void k_train_dz(TrainMisc m);
__global__ void k_train_dact(TrainMisc m);
__global__ void k_train_mix_bwd(TrainMisc m);
size_t train_mix_smem(int B);               // dynamic shared memory of k_train_mix / _mix_bwd
__global__ void k_train_fuse_bwd(TrainMisc m);
constexpr int TRAIN_ROW_CHUNK = 16384;      // vocabulary ids per k_train_rows item (8 warps x 32 lanes x 64)
extern const size_t kTrainRowsSmemBytes;
extern const int kTrainRowsThreads;

// acceptance launch shared by xpress_accept and xpress_accept_noalloc
// (xpress_host.cu); `ws` holds the scratch laid out by accept_scratch_bytes
size_t accept_scratch_bytes(const xpress_refiner *R, int b);
int refiner_device(const xpress_refiner *R);   // the device the refiner was created on
const xpress_weights &refiner_weights(const xpress_refiner *R);
int refiner_sms(const xpress_refiner *R);
unsigned long long refiner_wait_ns(const xpress_refiner *R);
const CUtensorMap *refiner_tmap_wr128(const xpress_refiner *R);   // W_r, boxes of 128 rows x 64
// the refiner's second stream and four events, on which the training step
// runs its weight-gradient products beside the input-gradient chain
cudaStream_t refiner_train_aux(const xpress_refiner *R, cudaEvent_t (&ev)[4]);
// 2-D bf16 tensor [outer][inner] with a row pitch of `pitch` elements,
// 128-byte swizzle, zero fill out of bounds
bool tmap_bf16(CUtensorMap *m, const void *base, uint64_t inner, uint64_t outer, uint64_t pitch, uint32_t box_inner,
               uint32_t box_outer);
// [rows][r] bf16 as (64 columns, rows, r / 64 K chunks): a box of 64 x box_rows
// x r / 64 lands as the K-chunk tiles of 2D boxes of 64 x box_rows, back to back
bool tmap_bf16_kblocks(CUtensorMap *m, const void *base, uint64_t rows, uint32_t box_rows);
int accept_launch(const xpress_refiner *R, const xpress_accept_in *in, int32_t *accept_len, int32_t *out_tokens,
                  void *ws, size_t ws_bytes, void *stream);
constexpr int READ_SIMT_DYN_SMEM = (32 * (RANK + 1) + 8 * 32 * 33) * 4;
inline int pre_mix_smem(int B) { return (B * 2 * RANK + RANK + 32 * (2 * RANK + 1) + B * 32) * 4; }
// k_pre_mix after k_pre_tc, whose partials already carry W_in (folded): the
// block's h and g slot values of the 32 channels, and P
inline int pre_mix_smem_folded(int B) { return 3 * B * 32 * 4; }

}  // namespace xp
