// train_host.cu -- xpress_train_step (include/xpress.h): workspace layout,
// tensor maps and the launch sequence of one refiner training step (Sec. 4.3).
//
// Rows of every activation follow the paired order of the Read kernels: row
// 128 j + 64 f + l is position 64 j + l under the teacher-forced (f = 0) or the
// consistency (f = 1) inputs; NR = 128 ceil(P / 64) rows, the padding rows are
// zero throughout.
#include <cudaTypedefs.h>

#include <cstdint>
#include <mutex>

#include "kernels.h"
#include "xpress.h"

using namespace xp;

namespace {

#define XT_CUDA(call)                                                                                          \
    do {                                                                                                       \
        if ((call) != cudaSuccess) {                                                                           \
            (void)cudaGetLastError();                                                                          \
            return XPRESS_ERR_CUDA;                                                                            \
        }                                                                                                      \
    } while (0)

size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

// Launch with programmatic stream serialization: the kernel may start its
// set-up while its predecessor finishes (every training kernel waits with
// griddepcontrol.wait before it touches memory).
template <typename... KArgs, typename... Args>
cudaError_t launch(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args)
{
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

struct TrainLayout {
    int P = 0, NR = 0, nch = 0, nvt = 0, splits = 1, usplits = 1;
    size_t rpart, rkey, lse_s2, lse_q2, s_y, xhat, xrow, Uh, Ug, X, Xlo, a, c, cop, t, uop, zop, part, ly, lse_p2, coef, A2,
        dzp, dz, dzb, du, dtb, dc, dab, dX, D, total;
};

// K splits of a split product of M x N x K: about one CTA per SM.
int gemm_splits(int sms, int M, int N, int K)
{
    const int tiles = ((M + 127) / 128) * ((N + 63) / 64);
    const int nk = (K + 63) / 64;
    int splits = tiles < sms ? sms / tiles : 1;
    if (splits > nk) splits = nk;
    if (splits < 1) splits = 1;
    const int kchunks = (nk + splits - 1) / splits;
    return (nk + kchunks - 1) / kchunks;          // the grid.z the product launches with
}

TrainLayout train_layout(const xpress_refiner *R, int b, int B)
{
    const xpress_weights &w = refiner_weights(R);
    TrainLayout L;
    L.P = b * B;
    L.NR = (L.P + 63) / 64 * 128;
    L.nch = (w.V + TRAIN_ROW_CHUNK - 1) / TRAIN_ROW_CHUNK;
    L.nvt = (w.V + 63) / 64;
    const int mt = L.NR / 128, sms = refiner_sms(R);
    L.splits = sms > mt ? (sms + mt / 2) / mt : 1;
    if (L.splits > L.nvt) L.splits = L.nvt;
    L.usplits = gemm_splits(sms, L.P, RANK, w.H);
    const size_t P = L.P, NR = L.NR, r = RANK;
    size_t o = 256;                                   // status word at offset 0
    auto take = [&](size_t bytes) { const size_t at = o; o += a256(bytes); return at; };
    L.rpart = take(P * L.nch * sizeof(float4));
    L.rkey = take(P * L.nch * 8);
    L.lse_s2 = take(P * 4);
    L.lse_q2 = take(P * 4);
    L.s_y = take(P * 4);
    L.xhat = take(P * 4);
    L.xrow = take(NR * 4);
    L.Uh = take((size_t)L.usplits * P * r * 4);
    L.Ug = take((size_t)L.usplits * P * r * 4);
    L.X = take(NR * 3 * r * 2);
    L.Xlo = take(NR * 2 * r * 2);
    L.a = take(NR * r * 4);
    L.c = take(NR * r * 4);
    L.cop = take(NR * r * 2);
    L.t = take(NR * 2 * r * 4);
    L.uop = take(NR * 2 * r * 2);
    L.zop = take(NR * r * 2);
    L.part = take((size_t)L.splits * NR * sizeof(float4));
    L.ly = take(NR * 4);
    L.lse_p2 = take(NR * 4);
    L.coef = take(NR * sizeof(RowCoef));
    L.A2 = take(NR * 4);
    L.dzp = take((size_t)L.splits * NR * r * 4);
    L.dz = take(NR * r * 4);
    L.dzb = take(NR * r * 2);
    L.du = take(NR * 2 * r * 4);
    L.dtb = take(NR * 2 * r * 2);
    L.dc = take(NR * r * 4);
    L.dab = take(NR * r * 2);
    L.dX = take(NR * 3 * r * 4);
    L.D = take(P * 2 * r * 2);
    L.total = o;
    return L;
}

int train_attributes()
{
    static int rc = -1;
    static std::once_flag once;
    std::call_once(once, [] {
        rc = XPRESS_OK;
        if (cudaFuncSetAttribute(k_train_tok_stats, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kTrainTokSmemBytes) != cudaSuccess ||
            cudaFuncSetAttribute(k_train_tok_tv, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTrainTokSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_train_tok_dz, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTrainTokSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_train_rows, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTrainRowsSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_train_voc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTrainVocSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_train_mix, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)train_mix_smem(MAX_B)) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_train_mix_bwd, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)train_mix_smem(MAX_B)) != cudaSuccess) {
            (void)cudaGetLastError();
            rc = XPRESS_ERR_CUDA;
        }
    });
    return rc;
}

// One operand of a product: bf16 [rows][pitch] at `base`; K-major when its rows
// run along M (or N), MN-major when they run along K.
struct Operand {
    const void *base;
    uint64_t pitch;
    bool mn;
};

// C (+)= alpha A B^T with A: M x K, B: N x K.  GM_ADD and GM_PART products
// split K over grid.z until about one CTA per SM runs (gemm_splits).
int gemm(cudaStream_t st, int sms, int M, int N, int K, Operand A, Operand B, int mode, float alpha, float *C,
         int ldc, uint16_t *Cb, int ldcb, const float *Rs, int ldr, int act)
{
    CUtensorMap ta, tb;
    const bool oka = A.mn ? tmap_bf16(&ta, A.base, (uint64_t)M, (uint64_t)K, A.pitch, 64, 64)
                          : tmap_bf16(&ta, A.base, (uint64_t)K, (uint64_t)M, A.pitch, 64, 128);
    const bool okb = B.mn ? tmap_bf16(&tb, B.base, (uint64_t)N, (uint64_t)K, B.pitch, 64, 64)
                          : tmap_bf16(&tb, B.base, (uint64_t)K, (uint64_t)N, B.pitch, 64, 64);
    if (!oka || !okb) return XPRESS_ERR_CUDA;
    GemmArgs g{};
    g.M = M;
    g.N = N;
    g.K = K;
    g.a_mn = A.mn;
    g.b_mn = B.mn;
    g.mode = mode;
    g.act = act;
    g.alpha = alpha;
    g.C = C;
    g.ldc = ldc;
    g.Cb = Cb;
    g.ldcb = ldcb;
    g.R = Rs;
    g.ldr = ldr;
    const int nk = (K + 63) / 64;
    const int splits = (mode == GM_ADD || mode == GM_PART) ? gemm_splits(sms, M, N, K) : 1;
    g.kchunks = (nk + splits - 1) / splits;
    const dim3 grid((M + 127) / 128, (N + 63) / 64, splits);
    XT_CUDA(launch(k_gemm, grid, dim3(192), kGemmSmemBytes, st, g, ta, tb));
    return XPRESS_OK;
}

}  // namespace

extern "C" {

size_t xpress_train_workspace_size(const xpress_refiner *R, int b, int B)
{
    if (!R || b < 1 || B < 1 || B > MAX_B) return 0;
    return train_layout(R, b, B).total;
}

}  // extern "C"

namespace {

// The training step; only >= 0 launches that vocabulary pass alone (0..3:
// log-sum-exp, total-variation sums, dL/dz, dL/dW_r) for profiling.
int train_run(const xpress_refiner *R, const xpress_train_in *in, const xpress_train_out *out, void *ws,
              size_t ws_bytes, void *stream, int only)
{
    if (!R || !in || !out) return XPRESS_ERR_INVALID_ARG;
    const xpress_weights &w = refiner_weights(R);
    if (w.dtype != XPRESS_BF16) return XPRESS_ERR_UNSUPPORTED;
    if (in->b < 1 || in->B != w.B || !in->h || !in->s || !in->target || !in->ystar || !in->anchor ||
        !(in->gamma > 0.0f) || !out->loss || !out->gW_e || !out->gW_h || !out->gW_g || !out->gW_in || !out->gL ||
        !out->gW1 || !out->gW2 || !out->gW_r)
        return XPRESS_ERR_INVALID_ARG;
    // h, s and target are read by bulk copies, tensor maps and 16-byte loads
    if (((reinterpret_cast<uintptr_t>(in->h) | reinterpret_cast<uintptr_t>(in->s) |
          reinterpret_cast<uintptr_t>(in->target)) & 15) != 0)
        return XPRESS_ERR_INVALID_ARG;
    if (refiner_device(R) >= 0) {
        int dev = -1;
        if (cudaGetDevice(&dev) != cudaSuccess || dev != refiner_device(R)) return XPRESS_ERR_INVALID_ARG;
    }
    const TrainLayout L = train_layout(R, in->b, in->B);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255) || ws_bytes < L.total) return XPRESS_ERR_WORKSPACE;
    if (train_attributes() != XPRESS_OK) return XPRESS_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char *W = static_cast<char *>(ws);
    const int H = w.H, V = w.V, r = RANK, P = L.P, NR = L.NR, sms = refiner_sms(R);
    auto F = [&](size_t off) { return reinterpret_cast<float *>(W + off); };
    auto U = [&](size_t off) { return reinterpret_cast<uint16_t *>(W + off); };

    TrainMisc m{};
    m.b = in->b;
    m.B = in->B;
    m.P = P;
    m.NR = NR;
    m.V = V;
    m.H = H;
    m.act = w.act;
    m.h = in->h;
    m.s = in->s;
    m.t = in->target;
    m.ystar = in->ystar;
    m.anchor = in->anchor;
    m.xhat_in = in->xhat;
    m.W_e = static_cast<const uint16_t *>(w.W_e);
    m.L = static_cast<const uint16_t *>(w.L);
    m.a_ce = in->a_ce;
    m.a_l1 = in->a_l1;
    m.gamma = in->gamma;
    m.lambda = in->lambda;
    m.beta = in->beta;
    m.nch = L.nch;
    m.rpart = reinterpret_cast<float4 *>(W + L.rpart);
    m.rkey = reinterpret_cast<unsigned long long *>(W + L.rkey);
    m.lse_s2 = F(L.lse_s2);
    m.lse_q2 = F(L.lse_q2);
    m.s_y = F(L.s_y);
    m.xhat = reinterpret_cast<int32_t *>(W + L.xhat);
    m.xrow = reinterpret_cast<int32_t *>(W + L.xrow);
    m.Uh = F(L.Uh);
    m.Ug = F(L.Ug);
    m.usplits = L.usplits;
    m.X = U(L.X);
    m.Xlo = U(L.Xlo);
    m.a = F(L.a);
    m.c = F(L.c);
    m.cop = U(L.cop);
    m.part = reinterpret_cast<const float4 *>(W + L.part);
    m.splits = L.splits;
    m.ly = F(L.ly);
    m.lse_p2 = F(L.lse_p2);
    m.coef = reinterpret_cast<RowCoef *>(W + L.coef);
    m.A2 = F(L.A2);
    m.W_r = static_cast<const uint16_t *>(w.W_r);
    m.zop = U(L.zop);
    m.gW_r = out->gW_r;
    m.loss = out->loss;
    m.dzp = F(L.dzp);
    m.dz = F(L.dz);
    m.dzb = U(L.dzb);
    m.du = F(L.du);
    m.tpre = F(L.t);
    m.dtb = U(L.dtb);
    m.dc = F(L.dc);
    m.dab = U(L.dab);
    m.gL = out->gL;
    m.gW_e = out->gW_e;
    m.dX = F(L.dX);
    m.D = U(L.D);
    m.status = reinterpret_cast<int32_t *>(W);

    TrainParams tp{};
    tp.P = P;
    tp.NR = NR;
    tp.V = V;
    tp.B = in->B;
    tp.nvt = L.nvt;
    tp.splits = L.splits;
    tp.ystar = in->ystar;
    tp.part = reinterpret_cast<float4 *>(W + L.part);
    tp.ly = F(L.ly);
    tp.lse_p2 = F(L.lse_p2);
    tp.lse_q2 = F(L.lse_q2);
    tp.lse_s2 = F(L.lse_s2);
    tp.coef = reinterpret_cast<const RowCoef *>(W + L.coef);
    tp.dzp = F(L.dzp);
    tp.gW_r = out->gW_r;
    tp.W_r = w.W_r;
    tp.zop = U(L.zop);
    tp.status = m.status;
    tp.wait_ns = refiner_wait_ns(R);

    CUtensorMap tz128, tz32, tw64, tw128, ts64, tt64, ts32, tt32;
    if (!tmap_bf16(&tz128, U(L.zop), r, NR, r, 64, 128) || !tmap_bf16(&tz32, U(L.zop), r, NR, r, 64, 32) ||
        !tmap_bf16_kblocks(&tw64, w.W_r, V, 64) || !tmap_bf16_kblocks(&tw128, w.W_r, V, 128) ||
        !tmap_bf16(&ts64, in->s, V, P, V, 64, 64) ||
        !tmap_bf16(&tt64, in->target, V, P, V, 64, 64) || !tmap_bf16(&ts32, in->s, V, P, V, 64, 32) ||
        !tmap_bf16(&tt32, in->target, V, P, V, 64, 32))
        return XPRESS_ERR_CUDA;

    const dim3 gtok(L.splits, NR / 128);
    const int nvt128 = (V + 127) / 128;
    if (only >= 0) {
        if (only == TR_STATS)
            XT_CUDA(launch(k_train_tok_stats, gtok, dim3(kTrainTokThreads), kTrainTokSmemBytes, st, tp, tz128,
                           tw128, ts64, tt64));
        else if (only == TR_TV)
            XT_CUDA(launch(k_train_tok_tv, gtok, dim3(kTrainTokThreads), kTrainTokSmemBytes, st, tp, tz128, tw64, ts64,
                           tt64));
        else if (only == TR_DZ)
            XT_CUDA(launch(k_train_tok_dz, gtok, dim3(kTrainTokThreads), kTrainTokSmemBytes, st, tp, tz128, tw64, ts64,
                           tt64));
        else
            XT_CUDA(launch(k_train_voc, dim3(nvt128 < sms ? nvt128 : sms), dim3(kTrainVocThreads), kTrainVocSmemBytes,
                           st, tp, tz32, *refiner_tmap_wr128(R), ts32, tt32));
        return XPRESS_OK;
    }

    // the status word and the padding rows' coefficients
    XT_CUDA(cudaMemsetAsync(W, 0, 4, st));
    XT_CUDA(cudaMemsetAsync(W + L.coef, 0, (size_t)NR * sizeof(RowCoef), st));
    XT_CUDA(cudaMemsetAsync(W + L.A2, 0, (size_t)NR * 4, st));

    // the drafter's rows: lse of s and of the target, s at y*, argmax s
    const int row_items = L.nch * P;
    XT_CUDA(launch(k_train_rows, dim3(row_items < sms ? row_items : sms), dim3(kTrainRowsThreads), kTrainRowsSmemBytes,
                   st, m));
    XT_CUDA(launch(k_train_rows_fin, dim3((P + 7) / 8), dim3(256), 0, st, m));

    // forward: Fuse, Mix, Trans of both input sequences
    int rc;
    const Operand h_k{in->h, (uint64_t)H, false}, h_mn{in->h, (uint64_t)H, true};
    if ((rc = gemm(st, sms, P, r, H, h_k, {w.W_h, (uint64_t)H, false}, GM_PART, 1.f, F(L.Uh), r, nullptr, 0, nullptr,
                   0, 0)))
        return rc;
    if ((rc = gemm(st, sms, P, r, H, h_k, {w.W_g, (uint64_t)H, false}, GM_PART, 1.f, F(L.Ug), r, nullptr, 0, nullptr,
                   0, 0)))
        return rc;
    XT_CUDA(launch(k_train_fuse, dim3(4 * in->b + NR / 2 - P), dim3(RANK), 0, st, m));
    if ((rc = gemm(st, sms, NR, r, 3 * r, {U(L.X), (uint64_t)3 * r, false}, {w.W_in, (uint64_t)3 * r, false}, GM_STORE,
                   1.f, F(L.a), r, nullptr, 0, nullptr, 0, 0)))
        return rc;
    // + the lo parts of u_h and u_g against W_in[:, 0:2r] (in place)
    if ((rc = gemm(st, sms, NR, r, 2 * r, {U(L.Xlo), (uint64_t)2 * r, false}, {w.W_in, (uint64_t)3 * r, false},
                   GM_RESID, 1.f, F(L.a), r, nullptr, 0, F(L.a), r, 0)))
        return rc;
    const dim3 gmix(RANK / 32, in->b), bmix(32, in->B);     // 2 sequences (both forwards of a block) per CTA
    XT_CUDA(launch(k_train_mix, gmix, bmix, train_mix_smem(in->B), st, m));
    if ((rc = gemm(st, sms, NR, 2 * r, r, {U(L.cop), (uint64_t)r, false}, {w.W1, (uint64_t)r, false}, GM_ACT, 1.f,
                   F(L.t), 2 * r, U(L.uop), 2 * r, nullptr, 0, w.act)))
        return rc;
    if ((rc = gemm(st, sms, NR, r, 2 * r, {U(L.uop), (uint64_t)2 * r, false}, {w.W2, (uint64_t)2 * r, false}, GM_RESID,
                   1.f, nullptr, 0, U(L.zop), r, F(L.c), r, 0)))
        return rc;

    // the Read passes
    const dim3 gvoc(nvt128 < sms ? nvt128 : sms);
    // W_r tiles of 128 ids (boxes of 128 rows) for the log-sum-exp pass, of 64 for the others
    XT_CUDA(launch(k_train_tok_stats, gtok, dim3(kTrainTokThreads), kTrainTokSmemBytes, st, tp, tz128, tw128,
                   ts64, tt64));
    XT_CUDA(launch(k_train_stats_fin, dim3(NR / 8), dim3(256), 0, st, m));
    XT_CUDA(launch(k_train_tok_tv, gtok, dim3(kTrainTokThreads), kTrainTokSmemBytes, st, tp, tz128, tw64, ts64,
                   tt64));
    XT_CUDA(launch(k_train_tv_fin, dim3(in->b), dim3(32), 0, st, m));
    XT_CUDA(launch(k_train_tok_dz, gtok, dim3(kTrainTokThreads), kTrainTokSmemBytes, st, tp, tz128, tw64, ts64,
                   tt64));
    XT_CUDA(launch(k_train_voc, gvoc, dim3(kTrainVocThreads), kTrainVocSmemBytes, st, tp, tz32,
                   *refiner_tmap_wr128(R), ts32, tt32));

    // backward through Trans (Eq. mlp)
    XT_CUDA(launch(k_train_dz, dim3((NR * r / 4 + 255) / 256), dim3(256), 0, st, m));
    if ((rc = gemm(st, sms, NR, 2 * r, r, {U(L.dzb), (uint64_t)r, false}, {w.W2, (uint64_t)2 * r, true}, GM_STORE, 1.f,
                   F(L.du), 2 * r, nullptr, 0, nullptr, 0, 0)))
        return rc;
    XT_CUDA(launch(k_train_dact, dim3((NR * 2 * r / 4 + 255) / 256), dim3(256), 0, st, m));
    // The weight-gradient products run on the refiner's second stream beside
    // the input-gradient chain (dz -> dc -> Mix backward -> dX -> Fuse
    // backward), each forked once its operands exist and joined at the end;
    // none of their operands is written again in the step.
    cudaEvent_t ev[4];
    const cudaStream_t aux = refiner_train_aux(R, ev);
    XT_CUDA(cudaEventRecord(ev[0], st));                        // dz and dt
    XT_CUDA(cudaStreamWaitEvent(aux, ev[0], 0));
    if ((rc = gemm(aux, sms, r, 2 * r, NR, {U(L.dzb), (uint64_t)r, true}, {U(L.uop), (uint64_t)2 * r, true}, GM_ADD,
                   1.f, out->gW2, 2 * r, nullptr, 0, nullptr, 0, 0)))
        return rc;
    if ((rc = gemm(aux, sms, 2 * r, r, NR, {U(L.dtb), (uint64_t)2 * r, true}, {U(L.cop), (uint64_t)r, true}, GM_ADD,
                   1.f, out->gW1, r, nullptr, 0, nullptr, 0, 0)))
        return rc;
    if ((rc = gemm(st, sms, NR, r, 2 * r, {U(L.dtb), (uint64_t)2 * r, false}, {w.W1, (uint64_t)r, true}, GM_RESID, 1.f,
                   F(L.dc), r, nullptr, 0, F(L.dz), r, 0)))
        return rc;

    // backward through Mix (Eq. mix) and Fuse (Eq. fuse)
    XT_CUDA(launch(k_train_mix_bwd, gmix, bmix, train_mix_smem(in->B), st, m));
    XT_CUDA(cudaEventRecord(ev[1], st));                        // dL/da
    XT_CUDA(cudaStreamWaitEvent(aux, ev[1], 0));
    if ((rc = gemm(aux, sms, r, 3 * r, NR, {U(L.dab), (uint64_t)r, true}, {U(L.X), (uint64_t)3 * r, true}, GM_ADD, 1.f,
                   out->gW_in, 3 * r, nullptr, 0, nullptr, 0, 0)))
        return rc;
    if ((rc = gemm(st, sms, NR, 3 * r, r, {U(L.dab), (uint64_t)r, false}, {w.W_in, (uint64_t)3 * r, true}, GM_STORE,
                   1.f, F(L.dX), 3 * r, nullptr, 0, nullptr, 0, 0)))
        return rc;
    XT_CUDA(launch(k_train_fuse_bwd, dim3(P), dim3(RANK), 0, st, m));
    XT_CUDA(cudaEventRecord(ev[2], st));                        // dL/du_h, dL/du_g
    XT_CUDA(cudaStreamWaitEvent(aux, ev[2], 0));
    if ((rc = gemm(aux, sms, r, H, P, {U(L.D) + r, (uint64_t)2 * r, true}, h_mn, GM_ADD, 1.f, out->gW_g, H, nullptr, 0,
                   nullptr, 0, 0)))
        return rc;
    if ((rc = gemm(st, sms, r, H, P, {U(L.D), (uint64_t)2 * r, true}, h_mn, GM_ADD, 1.f, out->gW_h, H, nullptr, 0,
                   nullptr, 0, 0)))
        return rc;
    XT_CUDA(cudaEventRecord(ev[3], aux));                       // join
    XT_CUDA(cudaStreamWaitEvent(st, ev[3], 0));
    return XPRESS_OK;
}

}  // namespace

extern "C" {

int xpress_train_step(const xpress_refiner *R, const xpress_train_in *in, const xpress_train_out *out, void *ws,
                      size_t ws_bytes, void *stream)
{
    return train_run(R, in, out, ws, ws_bytes, stream, -1);
}

int xpress_profile_train(const xpress_refiner *R, const xpress_train_in *in, const xpress_train_out *out, void *ws,
                         size_t ws_bytes, int pass, void *stream)
{
    if (pass < 0 || pass > 3) return XPRESS_ERR_INVALID_ARG;
    return train_run(R, in, out, ws, ws_bytes, stream, pass);
}

int xpress_debug_gemm(const void *A, int a_mn, const void *B, int b_mn, int M, int N, int K, float *C, int accumulate,
                      void *stream)
{
    if (!A || !B || !C || M < 1 || N < 1 || K < 1 || (a_mn && (M % 8)) || (b_mn && (N % 8)) || (!a_mn && (K % 8)) ||
        (!b_mn && (K % 8)))
        return XPRESS_ERR_INVALID_ARG;
    if (train_attributes() != XPRESS_OK) return XPRESS_ERR_CUDA;
    int dev = 0, sms = 0;
    XT_CUDA(cudaGetDevice(&dev));
    XT_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    const Operand a{A, (uint64_t)(a_mn ? M : K), a_mn != 0}, b{B, (uint64_t)(b_mn ? N : K), b_mn != 0};
    return gemm(static_cast<cudaStream_t>(stream), sms, M, N, K, a, b, accumulate ? GM_ADD : GM_STORE, 1.f, C, N,
                nullptr, 0, nullptr, 0, 0);
}

}  // extern "C"
