// xpress_host.cu -- the C ABI (include/xpress.h): argument checks, workspace
// layout, TMA descriptors, and the CUDA graph that runs Algorithm 1 with its
// iteration loop on the device (a WHILE conditional node whose condition the
// reduce kernel updates after every pass).
#include <cudaTypedefs.h>

#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>

#include "kernels.h"
#include "xpress.h"

using namespace xp;

namespace {

constexpr int XPRESS_VERSION = 2;
constexpr int CACHE_SLOTS = 8;

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}

// 2-D bf16 tensor [outer][inner], 128-byte swizzle, zero fill out of bounds.
bool make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                    uint32_t box_outer)
{
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {inner * 2};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// W_r [rows][r] bf16 viewed as (64 columns, rows, r / 64 K chunks of 64
// columns, 128 bytes apart): a box of 64 x box_rows x r / 64 lands in shared
// memory as the K-chunk tiles of 2D boxes of 64 x box_rows, back to back, with
// the same 128-byte swizzle.
bool make_tmap_bf16_kblocks(CUtensorMap *m, const void *base, uint64_t rows, uint32_t box_rows)
{
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {64, rows, RANK / 64};
    cuuint64_t strides[2] = {RANK * 2, 128};
    cuuint32_t box[3] = {64, box_rows, RANK / 64};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The folded projection Fhl [term 2][slot 2][r rows][H] bf16 as a 5D map
// (64 columns, r rows of a slot, slot, term, H / 64 K tiles of 128 bytes): a
// box of 64 x 2 x 2 x 2 x kt holds the 8 rows (term, slot, channel pair) of
// one unit over kt K tiles, landing as [K tile][row][128 bytes].
bool make_tmap_fold_k(CUtensorMap *m, const void *Fhl, uint64_t H, uint32_t kt)
{
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[5] = {64, RANK, 2, 2, H / 64};
    cuuint64_t strides[4] = {H * 2, (cuuint64_t)RANK * H * 2, (cuuint64_t)2 * RANK * H * 2, 128};
    cuuint32_t box[5] = {64, 2, 2, 2, kt};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(Fhl), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// h [N][H] bf16 as (64 columns, N rows, H / 64 K tiles): a box of
// 64 x rows x kt lands as [K tile][row][128 bytes] (rows past N zero).
bool make_tmap_rows_k(CUtensorMap *m, const void *h, uint64_t N, uint64_t H, uint32_t rows, uint32_t kt)
{
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {64, N, H / 64};
    cuuint64_t strides[2] = {H * 2, 128};
    cuuint32_t box[3] = {64, rows, kt};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(h), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct GraphEntry {
    bool used = false;
    void *ws = nullptr;
    size_t ws_bytes = 0;
    int b = 0;
    bool draft_null = false;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    cudaGraphNode_t init_node = nullptr;
    cudaGraphNode_t pre_node = nullptr;    // k_pre_tc (its h tensor map changes per call)
    cudaGraphConditionalHandle handle = 0;
    dim3 init_grid;
    uint64_t stamp = 0;
};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct Layout {
    size_t status = 0, ctl = 64, params = 256, st = 0, upart = 0, pc = 0, ynew = 0, acttok = 0, zpack = 0,
           zbuf = 0, part = 0, cbuf = 0, ubuf = 0, total = 0;
    size_t sctl = 0, cx = 0, ux = 0, pcx = 0, c0x = 0, rmax = 0, best64 = 0;
    int ksplit = 1, kchunk = 0, S = 1;
    bool gemv = false;
    bool tcv = false;
    bool small = false;      // persistent small-batch kernel
    bool pre_tc = false;     // hidden projection on tcgen05 (bf16, more than 32 tokens)
};

}  // namespace

struct xpress_refiner {
    xpress_weights w{};
    float *Ep = nullptr;
    unsigned long long *trace = nullptr;   // profiling timeline (XPRESS_TRACE=1)
    CUtensorMap tmap_wr{};                 // W_r boxes of 256 rows (k_read_tc)
    CUtensorMap tmap_wr128{};              // W_r boxes of 128 rows (k_read_tcv, the training step)
    CUtensorMap tmap_wrb{};                // W_r as (64 columns, rows, 4 K chunks): one 128-row block per box (k_refine_small)
    CUtensorMap tmap_fk{};                 // folded projection as (64 columns, rows of a slot, slot, term, K tile) (k_refine_small)
    CUtensorMap tmap_wr32{};               // W_r boxes of 32 rows (k_refine_small, partial blocks)
    CUtensorMap tmap_wh{}, tmap_wg{};      // W_h, W_g boxes of 256 rows x 64
    CUtensorMap tmap_fhi{}, tmap_flo{};    // folded projection, hi / lo term, boxes of 256 rows x 64 (k_pre_tc)
    CUtensorMap tmap_w1{}, tmap_w2{};      // W_1 [2r, r], W_2 [r, 2r], boxes of 32 rows x 64 (k_trans_tc)
    int device = 0;
    int num_sms = 0;
    unsigned long long wait_ns = 2000000000ull;   // bound on the persistent kernel's waits for other CTAs
    bool use_tc = false;
    cudaStream_t cs = nullptr;
    cudaStream_t train_aux = nullptr;      // the training step's weight-gradient products (forked, then joined)
    cudaEvent_t train_ev[4] = {};
    uint16_t *Fhl = nullptr;               // [2][2r, H] folded hidden projection, bf16 hi / lo (bf16 refiners)
    uint16_t *Lpk = nullptr;               // [B(B-1)/2, r] L's strictly lower part, channel innermost
    bool small_ok = false;                 // the small-batch kernel can run co-resident on this GPU
    void *small_ws[CACHE_SLOTS] = {};      // workspaces whose control area this refiner has cleared
    int small_ws_next = 0;
    GraphEntry cache[CACHE_SLOTS];
    uint64_t clock = 0;
};

namespace {

// k_read_tcv serves calls that evaluate at most 32 tokens (b * B <= 32)
bool use_tcv(const xpress_refiner *R, int b) { return R->use_tc && b * R->w.B <= TCV_MAX_TOKENS; }

// The persistent kernel serves the same calls unless XPRESS_SMALL=0 (the
// multi-kernel graph path then runs them).
bool use_small(const xpress_refiner *R, int b)
{
    static const bool enabled = [] {
        const char *e = std::getenv("XPRESS_SMALL");
        return !(e && e[0] == '0');
    }();
    return enabled && R->small_ok && use_tcv(R, b);
}

int read_S(const xpress_refiner *R, int b)
{
    if (R->use_tc) {
        const int rows = use_tcv(R, b) ? 128 : 256;
        const int nvt = (R->w.V + rows - 1) / rows;
        const int sms = use_small(R, b) ? R->num_sms - SMALL_TRANS_CTAS : R->num_sms;
        return nvt < sms ? nvt : sms;
    }
    const int ng = (R->w.V + GROUP - 1) / GROUP;
    return ng < 2 * R->num_sms ? ng : 2 * R->num_sms;
}

Layout make_layout(const xpress_refiner *R, int b)
{
    Layout L;
    const int B = R->w.B, N = b * B;
    const size_t esz = R->w.dtype == XPRESS_BF16 ? 2 : 4;
    size_t o = align256(L.params + sizeof(Params));
    L.sctl = o;                                    // same offset for every b
    o = align256(o + sizeof(SmallCtlArea));
    L.st = o;
    o = align256(o + (size_t)b * sizeof(SeqState));
    L.gemv = R->w.dtype == XPRESS_BF16 && N <= 32;
    if (L.gemv) {
        // the largest K-slice (multiple of 256) whose h fits in 128 KB of shared memory
        int ks = (GEMV_SMEM / (2 * N)) / 256 * 256;
        const int H256 = (R->w.H + 255) / 256 * 256;
        L.kchunk = ks < H256 ? ks : H256;
        L.ksplit = (R->w.H + L.kchunk - 1) / L.kchunk;
    } else if (R->use_tc) {
        // k_pre_tc: 128-token x 256-row tiles, split over K to about one wave
        L.pre_tc = true;
        const int tiles = 2 * ((N + 127) / 128);
        int ks = (R->num_sms + tiles / 2) / tiles;
        const int kmax = (R->w.H + 63) / 64;
        ks = ks < 1 ? 1 : (ks > kmax ? kmax : ks);
        L.kchunk = ((R->w.H + ks - 1) / ks + 63) / 64 * 64;
        L.ksplit = (R->w.H + L.kchunk - 1) / L.kchunk;
    } else {
        const int mt = (N + 63) / 64;
        const int ctas = mt * (RANK / 64) * 2;
        int ks = (2 * R->num_sms + ctas - 1) / ctas;
        const int kmax = R->w.H / 256 > 0 ? R->w.H / 256 : 1;
        ks = ks < 1 ? 1 : (ks > kmax ? kmax : ks);
        L.kchunk = ((R->w.H + ks - 1) / ks + 15) / 16 * 16;
        L.ksplit = (R->w.H + L.kchunk - 1) / L.kchunk;
    }
    L.S = read_S(R, b);
    L.small = use_small(R, b);
    int upart_ks = L.ksplit;
    L.upart = o;
    o = align256(o + (size_t)upart_ks * N * 2 * RANK * 4);
    L.pc = o;
    o = align256(o + (size_t)N * RANK * 4);
    L.ynew = o;
    o = align256(o + (size_t)N * 4);
    L.acttok = o;
    o = align256(o + (size_t)N * 4);
    L.zpack = o;
    o = align256(o + (size_t)N * RANK * esz);
    L.zbuf = o;
    o = align256(o + (size_t)N * RANK * 4);
    L.tcv = use_tcv(R, b);
    L.part = o;
    o = align256(o + (size_t)L.S * N * sizeof(RPartial));
    if (R->use_tc && !L.tcv) {
        L.cbuf = o;
        o = align256(o + (size_t)N * RANK * 4);
        L.ubuf = o;
        o = align256(o + (size_t)N * 2 * RANK * 2);
    }
    if (L.small) {
        L.cx = o;
        o = align256(o + (size_t)32 * RANK * 2);
        L.ux = o;
        o = align256(o + (size_t)32 * 2 * RANK * 2);
        L.pcx = o;
        o = align256(o + (size_t)32 * RANK * 4);
        L.c0x = o;
        o = align256(o + (size_t)32 * RANK * 4);
        L.rmax = o;
        o = align256(o + (size_t)N * RMAX_SEG * sizeof(Partial));
        L.best64 = o;
        o = align256(o + 64 * sizeof(unsigned long long));
    }
    L.total = o;
    return L;
}

Params make_params(const xpress_refiner *R, const xpress_block_in *in, const xpress_block_out *out, void *ws,
                   const Layout &L)
{
    Params P{};
    char *w = static_cast<char *>(ws);
    P.b = in->b;
    P.B = R->w.B;
    P.H = R->w.H;
    P.V = R->w.V;
    P.N = in->b * R->w.B;
    P.dtype = R->w.dtype;
    P.act = R->w.act;
    P.K_max = in->K_max;
    P.fixed_K = in->fixed_K ? 1 : 0;
    P.sequential = in->mode == XPRESS_MODE_SEQUENTIAL ? 1 : 0;
    P.offset = in->offset;
    P.S = L.S;
    P.use_graph = 1;
    P.wait_ns = R->wait_ns;
    P.trace = R->trace;
    P.ksplit = L.ksplit;
    P.h = in->h;
    P.s = in->s;
    P.draft = in->draft;
    P.anchor = in->anchor;
    P.temperature = in->temperature;
    P.seed = reinterpret_cast<const unsigned long long *>(in->seed);
    P.W_h = R->w.W_h;
    P.W_g = R->w.W_g;
    P.W_in = R->w.W_in;
    P.L = R->w.L;
    P.W1 = R->w.W1;
    P.W2 = R->w.W2;
    P.W_r = R->w.W_r;
    P.Ep = R->Ep;
    P.tokens = out->tokens;
    P.iters = out->iters;
    P.converged = out->converged;
    P.lse = out->lse;
    P.logit_sel = out->logit_sel;
    P.z_final = out->z_final;
    P.logits = out->refined_logits;
    P.traj = out->trajectory;
    P.status = reinterpret_cast<int32_t *>(w + L.status);
    P.ctl = reinterpret_cast<int32_t *>(w + L.ctl);
    P.st = reinterpret_cast<SeqState *>(w + L.st);
    P.Upart = reinterpret_cast<float *>(w + L.upart);
    P.pre_folded = L.pre_tc ? 1 : 0;
    P.Lpk = R->Lpk;                        // null for fp32 refiners
    P.Pc = reinterpret_cast<float *>(w + L.pc);
    P.Ynew = reinterpret_cast<int32_t *>(w + L.ynew);
    P.act_tok = reinterpret_cast<int32_t *>(w + L.acttok);
    P.zpack = w + L.zpack;
    P.zbuf = reinterpret_cast<float *>(w + L.zbuf);
    P.part = reinterpret_cast<RPartial *>(w + L.part);
    if (L.cbuf) {
        P.cbuf = reinterpret_cast<float *>(w + L.cbuf);
        P.ubuf = reinterpret_cast<uint16_t *>(w + L.ubuf);
    }
    if (L.small) {
        P.use_graph = 0;
        P.Fhl = R->Fhl;
        P.c0x = reinterpret_cast<float *>(w + L.c0x);
        P.cx = reinterpret_cast<uint16_t *>(w + L.cx);
        P.ux = reinterpret_cast<uint16_t *>(w + L.ux);
        P.pcx = reinterpret_cast<float *>(w + L.pcx);
        P.rmax = reinterpret_cast<Partial *>(w + L.rmax);
        P.sctl = reinterpret_cast<SmallCtlArea *>(w + L.sctl);
        P.best64 = reinterpret_cast<unsigned long long *>(w + L.best64);
    }
    return P;
}

#define XP_CUDA(call)                                                                                          \
    do {                                                                                                       \
        if ((call) != cudaSuccess) {                                                                           \
            (void)cudaGetLastError();                                                                          \
            return XPRESS_ERR_CUDA;                                                                            \
        }                                                                                                      \
    } while (0)

int set_kernel_attributes()
{
    static int rc = -1;
    static std::once_flag once;
    std::call_once(once, [] {
        rc = XPRESS_OK;
        if (cudaFuncSetAttribute(k_read_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kReadTcSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_mix_mlp, cudaFuncAttributeMaxDynamicSharedMemorySize, MIX_MLP_DYN_SMEM_MAX) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_read_simt, cudaFuncAttributeMaxDynamicSharedMemorySize, READ_SIMT_DYN_SMEM) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_pre_mix, cudaFuncAttributeMaxDynamicSharedMemorySize, pre_mix_smem(MAX_B)) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_pre_gemv, cudaFuncAttributeMaxDynamicSharedMemorySize, GEMV_SMEM) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_read_tcv, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kReadTcvSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_refine_small, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kRefineSmallSmemBytes) != cudaSuccess ||
            cudaFuncSetAttribute(k_pre_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPreTcSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_lm_head32, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kLmHeadSmemBytes[0]) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_trans_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTransTcSmemBytes) !=
                cudaSuccess ||
            cudaFuncSetAttribute(k_lm_head256, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kLmHeadSmemBytes[1]) != cudaSuccess) {
            (void)cudaGetLastError();
            rc = XPRESS_ERR_CUDA;
        }
    });
    return rc;
}

// Launch with programmatic stream serialization: the kernel may start while
// its predecessor finishes and waits for it with griddepcontrol.wait.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args... args)
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

// Arguments of a k_pre_tc launch (kept alive for cudaGraphAddKernelNode /
// cudaGraphExecKernelNodeSetParams, which read them through kernelParams).
struct PreTcArgs {
    const Params *pdev;
    CUtensorMap th;
    CUtensorMap wh, wg;
    int kslice;
    void *ptrs[5];
    bool make(const xpress_refiner *R, const Params &P, const Layout &L, Params *pd)
    {
        pdev = pd;
        wh = R->tmap_fhi;
        wg = R->tmap_flo;
        kslice = L.kchunk;
        ptrs[0] = &pdev; ptrs[1] = &th; ptrs[2] = &wh; ptrs[3] = &wg; ptrs[4] = &kslice;
        return make_tmap_bf16(&th, P.h, (uint64_t)P.H, (uint64_t)P.N, 64, 128);
    }
    cudaKernelNodeParams node(const Layout &L, int N)
    {
        cudaKernelNodeParams kp{};
        kp.func = reinterpret_cast<void *>(k_pre_tc);
        kp.gridDim = dim3((unsigned)((N + 127) / 128), 2, (unsigned)L.ksplit);
        kp.blockDim = dim3(320);
        kp.sharedMemBytes = (unsigned)kPreTcSmemBytes;
        kp.kernelParams = ptrs;
        return kp;
    }
};

void launch_pre_gemm(const Layout &L, int N, Params *pdev, cudaStream_t st)
{
    if (L.gemv) {
        k_pre_gemv<<<dim3(2 * RANK / 8, L.ksplit), 256, N * L.kchunk * 2, st>>>(pdev, L.kchunk);
    } else {
        const dim3 grid(RANK / 64, (N + 63) / 64, L.ksplit);
        k_pre_gemm<<<grid, 256, 0, st>>>(pdev, 0, L.kchunk);
        k_pre_gemm<<<grid, 256, 0, st>>>(pdev, 1, L.kchunk);
    }
}

// Tensor maps of the Trans operands on tcgen05 (graph path, bf16, more than
// 32 tokens): bf16(c) in zpack [N, r] and u in ubuf [N, 2r], boxes of 128
// token rows x 64.
bool make_trans_maps(const Params &P, CUtensorMap *tc, CUtensorMap *tu)
{
    return make_tmap_bf16(tc, P.zpack, RANK, (uint64_t)P.N, 64, 128) &&
           make_tmap_bf16(tu, P.ubuf, 2 * RANK, (uint64_t)P.N, 64, 128);
}

// Fuse + Mix and Trans of one pass: the multi-kernel tcgen05 form (bf16, more
// than 32 tokens), else k_mix_mlp.
cudaError_t launch_trans(const xpress_refiner *R, const Layout &L, const Params &P, Params *pdev, cudaStream_t st,
                         const CUtensorMap &tc, const CUtensorMap &tu)
{
    const int b = P.b;
    if (!(R->use_tc && !L.tcv))
        return launch_pdl(k_mix_mlp, dim3(8, b), dim3(256), mix_mlp_smem(P.dtype), st, (const Params *)pdev);
    const unsigned mt = (unsigned)((P.N + 127) / 128);
    cudaError_t e = launch_pdl(k_mix_c, dim3(8, b), dim3(256), 0, st, (const Params *)pdev);
    if (e == cudaSuccess)
        e = launch_pdl(k_trans_tc, dim3(mt, 2 * RANK / 32), dim3(192), kTransTcSmemBytes, st, (const Params *)pdev, tc,
                       R->tmap_w1, RANK, 1);
    if (e == cudaSuccess)
        e = launch_pdl(k_trans_tc, dim3(mt, RANK / 32), dim3(192), kTransTcSmemBytes, st, (const Params *)pdev, tu,
                       R->tmap_w2, 2 * RANK, 2);
    return e;
}

void destroy_entry(GraphEntry &e)
{
    if (e.exec) cudaGraphExecDestroy(e.exec);
    if (e.graph) cudaGraphDestroy(e.graph);
    e = GraphEntry{};
}

// Builds the per-(workspace, b) graph:
//   memset(status) -> k_init -> [k_rowmax] -> k_pre_gemm x2 -> k_pre_mix ->
//   WHILE (cond) { Trans (k_mix_mlp, or k_mix_c -> k_trans_tc x2) -> k_read_{tc,simt} -> k_reduce
//                  (updates cond) }
int build_graph(xpress_refiner *R, GraphEntry &e, const Params &P, const Layout &L, void *ws)
{
    const int b = P.b, N = P.N;
    Params *pdev = reinterpret_cast<Params *>(static_cast<char *>(ws) + L.params);
    CUtensorMap tmap_z{};
    if (R->use_tc && !make_tmap_bf16(&tmap_z, P.zpack, RANK, (uint64_t)N, 64, 32)) return XPRESS_ERR_CUDA;

    cudaGraph_t g = nullptr;
    XP_CUDA(cudaGraphCreate(&g, 0));
    e.graph = g;
    cudaMemsetParams ms{};
    ms.dst = P.status;
    ms.value = 0;
    ms.elementSize = 4;
    ms.width = 1;
    ms.height = 1;
    cudaGraphNode_t mnode = nullptr;
    XP_CUDA(cudaGraphAddMemsetNode(&mnode, g, nullptr, 0, &ms));
    e.init_grid = dim3((unsigned)((N > b ? N : b) + 255) / 256);
    XP_CUDA(cudaGraphConditionalHandleCreate(&e.handle, g, 0, cudaGraphCondAssignDefault));
    cudaGraphConditionalHandle handle = e.handle;
    {
        Params Pc = P;
        void *args[] = {&Pc, &pdev, &handle};
        cudaKernelNodeParams kp{};
        kp.func = reinterpret_cast<void *>(k_init);
        kp.gridDim = e.init_grid;
        kp.blockDim = dim3(256);
        kp.kernelParams = args;
        XP_CUDA(cudaGraphAddKernelNode(&e.init_node, g, &mnode, 1, &kp));
    }

    cudaGraphNode_t cap_dep = e.init_node;
    if (L.pre_tc) {
        PreTcArgs a;
        if (!a.make(R, P, L, pdev)) return XPRESS_ERR_CUDA;
        cudaKernelNodeParams kp = a.node(L, N);
        XP_CUDA(cudaGraphAddKernelNode(&e.pre_node, g, &e.init_node, 1, &kp));
        cap_dep = e.pre_node;
    }
    cudaStream_t cs = R->cs;
    XP_CUDA(cudaStreamBeginCaptureToGraph(cs, g, &cap_dep, nullptr, 1, cudaStreamCaptureModeThreadLocal));
    if (!P.draft) k_rowmax<<<N, 256, 0, cs>>>(pdev);
    if (!L.pre_tc) launch_pre_gemm(L, N, pdev, cs);
    k_pre_mix<<<dim3(b, RANK / 32), 256, L.pre_tc ? pre_mix_smem_folded(P.B) : pre_mix_smem(P.B), cs>>>(pdev);
    cudaStreamCaptureStatus cst;
    const cudaGraphNode_t *deps = nullptr;
    size_t ndeps = 0;
    cudaGraph_t capg = nullptr;
    if (cudaStreamGetCaptureInfo(cs, &cst, nullptr, &capg, &deps, nullptr, &ndeps) != cudaSuccess) {
        cudaGraph_t tmp;
        cudaStreamEndCapture(cs, &tmp);
        (void)cudaGetLastError();
        return XPRESS_ERR_CUDA;
    }
    cudaGraphNodeParams cp{};
    cp.type = cudaGraphNodeTypeConditional;
    cp.conditional.handle = handle;
    cp.conditional.type = cudaGraphCondTypeWhile;
    cp.conditional.size = 1;
    cudaGraphNode_t cnode = nullptr;
    const cudaError_t add_err = cudaGraphAddNode(&cnode, capg, deps, nullptr, ndeps, &cp);
    cudaError_t upd_err = cudaErrorUnknown;
    if (add_err == cudaSuccess)
        upd_err = cudaStreamUpdateCaptureDependencies(cs, &cnode, nullptr, 1, cudaStreamSetCaptureDependencies);
    cudaGraph_t outer = nullptr;
    const cudaError_t end_err = cudaStreamEndCapture(cs, &outer);
    if (add_err != cudaSuccess || upd_err != cudaSuccess || end_err != cudaSuccess) {
        (void)cudaGetLastError();
        return XPRESS_ERR_CUDA;
    }
    cudaGraph_t body = cp.conditional.phGraph_out[0];
    CUtensorMap tmap_c{}, tmap_u{};
    if (R->use_tc && !L.tcv && !make_trans_maps(P, &tmap_c, &tmap_u)) return XPRESS_ERR_CUDA;
    XP_CUDA(cudaStreamBeginCaptureToGraph(cs, body, nullptr, nullptr, 0, cudaStreamCaptureModeThreadLocal));
    XP_CUDA(launch_trans(R, L, P, pdev, cs, tmap_c, tmap_u));
    if (L.tcv) {
        // the small-batch Read kernel also ends the pass (fused reduce)
        XP_CUDA(launch_pdl(k_read_tcv, dim3(L.S), dim3(kReadTcvThreads), kReadTcvSmemBytes, cs, (const Params *)pdev,
                           R->tmap_wr128, tmap_z, R->w.V, 1, handle));
    } else {
        if (R->use_tc)
            XP_CUDA(launch_pdl(k_read_tc, dim3(L.S), dim3(kReadTcThreads), kReadTcSmemBytes, cs,
                               (const Params *)pdev, R->tmap_wr, tmap_z, R->w.V));
        else
            k_read_simt<<<L.S, 256, READ_SIMT_DYN_SMEM, cs>>>(pdev);
        XP_CUDA(launch_pdl(k_reduce, dim3(b), dim3(1024), 0, cs, (const Params *)pdev, handle));
    }
    cudaGraph_t body_out = nullptr;
    XP_CUDA(cudaStreamEndCapture(cs, &body_out));
    XP_CUDA(cudaGraphInstantiate(&e.exec, g, 0));
    return XPRESS_OK;
}

// Profiling mode (XPRESS_EAGER=1 in the environment): the same kernels
// launched one by one from the host, with a host read of the pass count after
// every pass, so that per-kernel profilers see each launch.  Not for serving.
// Per-kernel CUDA-event timer of the profiling mode (XPRESS_EAGER=2).
struct KernelTimer {
    cudaStream_t st;
    bool on;
    struct Rec { const char *name; cudaEvent_t a, b; };
    Rec recs[256];
    int n = 0;
    KernelTimer(cudaStream_t s, bool enable) : st(s), on(enable) {}
    void start(const char *name)
    {
        if (!on || n >= 256) return;
        recs[n].name = name;
        cudaEventCreate(&recs[n].a);
        cudaEventCreate(&recs[n].b);
        cudaEventRecord(recs[n].a, st);
    }
    void stop()
    {
        if (!on || n >= 256) return;
        cudaEventRecord(recs[n].b, st);
        ++n;
    }
    void report()
    {
        if (!on) return;
        cudaStreamSynchronize(st);
        std::fprintf(stderr, "xpress-timing:");
        for (int i = 0; i < n; ++i) {
            float ms = 0.0f;
            cudaEventElapsedTime(&ms, recs[i].a, recs[i].b);
            std::fprintf(stderr, " %s=%.2f", recs[i].name, 1000.0f * ms);
            cudaEventDestroy(recs[i].a);
            cudaEventDestroy(recs[i].b);
        }
        std::fprintf(stderr, "\n");
    }
};

// Profiling mode (XPRESS_EAGER=1 in the environment): the same kernels
// launched one by one from the host, with a host read of the pass count after
// every pass, so that per-kernel profilers see each launch; XPRESS_EAGER=2
// also prints CUDA-event times of every launch (microseconds) to stderr.
// Not for serving.
int run_eager(xpress_refiner *R, Params P, const Layout &L, void *ws, cudaStream_t st, bool timed)
{
    P.use_graph = 0;
    const int b = P.b, N = P.N;
    Params *pdev = reinterpret_cast<Params *>(static_cast<char *>(ws) + L.params);
    CUtensorMap tmap_z{};
    if (R->use_tc && !make_tmap_bf16(&tmap_z, P.zpack, RANK, (uint64_t)N, 64, 32)) return XPRESS_ERR_CUDA;
    KernelTimer kt(st, timed);
    XP_CUDA(cudaMemsetAsync(P.status, 0, 4, st));
    kt.start("init");
    k_init<<<((N > b ? N : b) + 255) / 256, 256, 0, st>>>(P, pdev, 0);
    kt.stop();
    if (!P.draft) {
        kt.start("rowmax");
        k_rowmax<<<N, 256, 0, st>>>(pdev);
        kt.stop();
    }
    kt.start("pre_gemm");
    if (L.pre_tc) {
        PreTcArgs a;
        if (!a.make(R, P, L, pdev)) return XPRESS_ERR_CUDA;
        k_pre_tc<<<dim3((unsigned)((N + 127) / 128), 2, (unsigned)L.ksplit), 320, kPreTcSmemBytes, st>>>(
            pdev, a.th, a.wh, a.wg, a.kslice);
    } else {
        launch_pre_gemm(L, N, pdev, st);
    }
    kt.stop();
    kt.start("pre_mix");
    k_pre_mix<<<dim3(b, RANK / 32), 256, L.pre_tc ? pre_mix_smem_folded(P.B) : pre_mix_smem(P.B), st>>>(pdev);
    kt.stop();
    CUtensorMap tmap_c{}, tmap_u{};
    if (R->use_tc && !L.tcv && !make_trans_maps(P, &tmap_c, &tmap_u)) return XPRESS_ERR_CUDA;
    for (int pass = 0; pass < P.K_max; ++pass) {
        kt.start("mix_mlp");
        XP_CUDA(launch_trans(R, L, P, pdev, st, tmap_c, tmap_u));
        kt.stop();
        kt.start("read");
        if (L.tcv)
            k_read_tcv<<<L.S, kReadTcvThreads, kReadTcvSmemBytes, st>>>(pdev, R->tmap_wr128, tmap_z, R->w.V, 1, 0);
        else if (R->use_tc)
            k_read_tc<<<L.S, kReadTcThreads, kReadTcSmemBytes, st>>>(pdev, R->tmap_wr, tmap_z, R->w.V);
        else
            k_read_simt<<<L.S, 256, READ_SIMT_DYN_SMEM, st>>>(pdev);
        kt.stop();
        if (!L.tcv) {
            kt.start("reduce");
            k_reduce<<<b, 1024, 0, st>>>(pdev, 0);
            kt.stop();
        }
        int32_t nact = 0;
        XP_CUDA(cudaMemcpyAsync(&nact, P.ctl + CTL_NACT, 4, cudaMemcpyDeviceToHost, st));
        XP_CUDA(cudaStreamSynchronize(st));
        if (nact == 0) break;
    }
    kt.report();
    XP_CUDA(cudaGetLastError());
    return XPRESS_OK;
}

void print_trace(xpress_refiner *R, cudaStream_t st);

// One call of the persistent small-batch kernel.  The control area's two
// blocks and parity word are cleared the first time this refiner meets the
// workspace; from then on each call clears the block the next call uses.
int run_small(xpress_refiner *R, const Params &P, const Layout &L, void *ws, cudaStream_t st)
{
    bool seen = false;
    for (void *s : R->small_ws) seen = seen || s == ws;
    if (!seen) {
        XP_CUDA(cudaMemsetAsync(static_cast<char *>(ws) + L.sctl, 0, sizeof(SmallCtlArea), st));
        R->small_ws[R->small_ws_next] = ws;
        R->small_ws_next = (R->small_ws_next + 1) % CACHE_SLOTS;
    }
    CUtensorMap tmap_z{}, tmap_h{};
    if (!make_tmap_bf16(&tmap_z, P.zpack, RANK, (uint64_t)P.N, 64, 32) ||
        !make_tmap_rows_k(&tmap_h, P.h, (uint64_t)P.N, (uint64_t)P.H, P.N <= 16 ? 16 : 32, SMALL_PC_KT))
        return XPRESS_ERR_CUDA;
    if (R->trace) {
        XP_CUDA(cudaMemsetAsync(R->trace, 0xFF, TRACE_SLOTS * sizeof(unsigned long long), st));
        XP_CUDA(cudaMemsetAsync(R->trace + TRACE_SLOTS, 0, TRACE_SLOTS * sizeof(unsigned long long), st));
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)(L.S + SMALL_TRANS_CTAS));
    cfg.blockDim = dim3(32 * (2 + 8));
    cfg.dynamicSmemBytes = kRefineSmallSmemBytes;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    XP_CUDA(cudaLaunchKernelEx(&cfg, k_refine_small, P, R->tmap_wrb, R->tmap_wr32, tmap_z, R->tmap_fk, tmap_h));
    if (R->trace) print_trace(R, st);
    return XPRESS_OK;
}

int eager_mode()
{
    static const int mode = [] {
        const char *e = std::getenv("XPRESS_EAGER");
        return (e && (e[0] == '1' || e[0] == '2')) ? e[0] - '0' : 0;
    }();
    return mode;
}

// Prints the device timeline of the call just launched (XPRESS_TRACE=1):
// per kernel, start and end in microseconds from the first kernel's start.
void print_trace(xpress_refiner *R, cudaStream_t st)
{
    unsigned long long h[2 * TRACE_SLOTS];
    if (cudaMemcpyAsync(h, R->trace, sizeof(h), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return;
    unsigned long long t0 = ~0ull;
    for (int i = 0; i < TRACE_SLOTS; ++i)
        if (h[i] < t0) t0 = h[i];
    static const char *pre[4] = {"init", "seed", "precompute", "pc"};
    static const char *body[3] = {"mlp", "read", "reduce"};
    std::fprintf(stderr, "xpress-trace:");
    for (int i = 0; i < TRACE_SLOTS; ++i) {
        if (h[i] == ~0ull) continue;
        char name[32];
        if (i >= 248) std::snprintf(name, sizeof(name), "transsetup%d", i - 248);
        else if (i >= 4 && i < 8) std::snprintf(name, sizeof(name), "readsetup%d", i - 4);
        else if (i >= 240 && i < 248) std::snprintf(name, sizeof(name), "end%dphase%d", (i - 240) / 4, (i - 240) % 4);
        else if (i >= 230 && i < 240) std::snprintf(name, sizeof(name), "read0phase%d", i - 230);
        else if (i >= 210) std::snprintf(name, sizeof(name), "mlp%dphase%d", (i - 210) / 8, (i - 210) % 8);
        else if (i >= 200) std::snprintf(name, sizeof(name), "readphase%d", i - 200);
        else if (i < 8) std::snprintf(name, sizeof(name), "%s", i < 4 ? pre[i] : "?");
        else std::snprintf(name, sizeof(name), "%s%d", (i - 8) % 4 < 3 ? body[(i - 8) % 4] : "?", (i - 8) / 4);
        std::fprintf(stderr, " %s=[%.1f,%.1f]", name, (h[i] - t0) / 1000.0, (h[TRACE_SLOTS + i] - t0) / 1000.0);
    }
    std::fprintf(stderr, "\n");
}

int check_ws(void *ws, size_t ws_bytes, size_t need)
{
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255) || ws_bytes < need) return XPRESS_ERR_WORKSPACE;
    return XPRESS_OK;
}

}  // namespace

extern "C" {

int xpress_version(void) { return XPRESS_VERSION; }

const char *xpress_status_string(int s)
{
    switch (s) {
    case XPRESS_OK: return "ok";
    case XPRESS_ERR_INVALID_ARG: return "invalid argument";
    case XPRESS_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case XPRESS_ERR_CUDA: return "CUDA runtime error";
    case XPRESS_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case XPRESS_ERR_TIMEOUT: return "device wait timed out";
    case XPRESS_ERR_DEVICE_CHECK: return "device bounds check failed";
    default: return "unknown status";
    }
}

int xpress_refiner_create(const xpress_weights *w, void *stream, xpress_refiner **out)
{
    if (!w || !out) return XPRESS_ERR_INVALID_ARG;
    *out = nullptr;
    if (!w->W_e || !w->W_h || !w->W_g || !w->W_in || !w->L || !w->W1 || !w->W2 || !w->W_r)
        return XPRESS_ERR_INVALID_ARG;
    if (w->r != RANK || w->B < 1 || w->B > MAX_B || w->V < GROUP || (w->V % 8) || w->H < 8 || (w->H % 8) ||
        (w->dtype != XPRESS_F32 && w->dtype != XPRESS_BF16) || w->act < 0 || w->act > 2)
        return XPRESS_ERR_UNSUPPORTED;
    if (set_kernel_attributes() != XPRESS_OK) return XPRESS_ERR_CUDA;
    xpress_refiner *R = new (std::nothrow) xpress_refiner();
    if (!R) return XPRESS_ERR_CUDA;
    R->w = *w;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int rc = XPRESS_OK;
    do {
        if (cudaGetDevice(&R->device) != cudaSuccess ||
            cudaDeviceGetAttribute(&R->num_sms, cudaDevAttrMultiProcessorCount, R->device) != cudaSuccess) {
            rc = XPRESS_ERR_CUDA;
            break;
        }
        R->use_tc = w->dtype == XPRESS_BF16;
        if (R->use_tc && (!make_tmap_bf16(&R->tmap_wr, w->W_r, RANK, (uint64_t)w->V, 64, 256) ||
                          !make_tmap_bf16(&R->tmap_wr128, w->W_r, RANK, (uint64_t)w->V, 64, 128) ||
                          !make_tmap_bf16(&R->tmap_wr32, w->W_r, RANK, (uint64_t)w->V, 64, 32) ||
                          !make_tmap_bf16_kblocks(&R->tmap_wrb, w->W_r, (uint64_t)w->V, 128) ||
                          !make_tmap_bf16(&R->tmap_wh, w->W_h, (uint64_t)w->H, RANK, 64, 256) ||
                          !make_tmap_bf16(&R->tmap_wg, w->W_g, (uint64_t)w->H, RANK, 64, 256))) {
            rc = XPRESS_ERR_CUDA;
            break;
        }
        if (const char *tr = std::getenv("XPRESS_TRACE"))
            if (tr[0] == '1' && cudaMalloc(&R->trace, 2 * TRACE_SLOTS * sizeof(unsigned long long)) != cudaSuccess) {
                rc = XPRESS_ERR_CUDA;
                break;
            }
        if (cudaMalloc(&R->Ep, (size_t)w->V * RANK * sizeof(float)) != cudaSuccess ||
            cudaStreamCreateWithFlags(&R->cs, cudaStreamNonBlocking) != cudaSuccess ||
            cudaStreamCreateWithFlags(&R->train_aux, cudaStreamNonBlocking) != cudaSuccess) {
            rc = XPRESS_ERR_CUDA;
            break;
        }
        for (auto &ev : R->train_ev)
            if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess) rc = XPRESS_ERR_CUDA;
        if (rc != XPRESS_OK) break;
        const dim3 grid(RANK / 64, (w->V + 63) / 64);
        k_build_ep<<<grid, 256, 0, st>>>(w->W_e, w->W_in, R->Ep, w->V, w->dtype);
        if (R->use_tc) {
            // persistent small-batch kernel: every CTA must be resident at once
            int coop = 0, per_sm = 0;
            if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, R->device) != cudaSuccess ||
                cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_refine_small, 32 * (2 + 8),
                                                              kRefineSmallSmemBytes) != cudaSuccess) {
                (void)cudaGetLastError();
                coop = 0;
            }
            // the folded hidden projection (both the persistent kernel and
            // k_pre_tc take it)
            if (cudaMalloc(&R->Fhl, (size_t)2 * 2 * RANK * w->H * sizeof(uint16_t)) != cudaSuccess) {
                rc = XPRESS_ERR_CUDA;
                break;
            }
            k_fold_hidden<<<dim3((w->H + 255) / 256, 2 * RANK / 8), 256, 0, st>>>(
                static_cast<const uint16_t *>(w->W_h), static_cast<const uint16_t *>(w->W_g),
                static_cast<const uint16_t *>(w->W_in), R->Fhl, w->H);
            if (!make_tmap_bf16(&R->tmap_w1, w->W1, RANK, 2 * RANK, 64, 32) ||
                !make_tmap_bf16(&R->tmap_w2, w->W2, 2 * RANK, RANK, 64, 32)) {
                rc = XPRESS_ERR_CUDA;
                break;
            }
            if (!make_tmap_bf16(&R->tmap_fhi, R->Fhl, (uint64_t)w->H, 2 * RANK, 64, 256) ||
                !make_tmap_bf16(&R->tmap_flo, R->Fhl + (size_t)2 * RANK * w->H, (uint64_t)w->H, 2 * RANK, 64, 256)) {
                rc = XPRESS_ERR_CUDA;
                break;
            }
            // L's strictly lower part, channel innermost (coalesced mixes)
            const int tri = w->B * (w->B - 1) / 2;
            if (cudaMalloc(&R->Lpk, (size_t)(tri > 0 ? tri : 1) * RANK * 2) != cudaSuccess) {
                rc = XPRESS_ERR_CUDA;
                break;
            }
            if (tri > 0)
                k_pack_L<<<(tri + 7) / 8, 256, 0, st>>>(static_cast<const uint16_t *>(w->L), R->Lpk, w->B);
            // the persistent kernel reads h and F by K tiles of 64 (H % 64 == 0)
            const bool fk = w->H % 64 == 0 && make_tmap_fold_k(&R->tmap_fk, R->Fhl, (uint64_t)w->H, SMALL_PC_KT);
            if (coop && per_sm >= 1 && R->num_sms > SMALL_TRANS_CTAS && fk) R->small_ok = true;
        }
        if (cudaGetLastError() != cudaSuccess || cudaStreamSynchronize(st) != cudaSuccess) rc = XPRESS_ERR_CUDA;
    } while (0);
    if (rc != XPRESS_OK) {
        (void)cudaGetLastError();
        xpress_refiner_destroy(R);
        return rc;
    }
    *out = R;
    return XPRESS_OK;
}

int xpress_refiner_destroy(xpress_refiner *R)
{
    if (!R) return XPRESS_ERR_INVALID_ARG;
    for (auto &e : R->cache) destroy_entry(e);
    if (R->Ep) cudaFree(R->Ep);
    if (R->Fhl) cudaFree(R->Fhl);
    if (R->Lpk) cudaFree(R->Lpk);
    if (R->cs) cudaStreamDestroy(R->cs);
    if (R->train_aux) cudaStreamDestroy(R->train_aux);
    for (auto &ev : R->train_ev)
        if (ev) cudaEventDestroy(ev);
    if (R->trace) cudaFree(R->trace);
    delete R;
    return XPRESS_OK;
}

size_t xpress_refine_workspace_size(const xpress_refiner *R, int b)
{
    if (!R || b < 1) return 0;
    return make_layout(R, b).total;
}

int xpress_refine_block(const xpress_refiner *Rc, const xpress_block_in *in, const xpress_block_out *out,
                        void *ws, size_t ws_bytes, void *stream)
{
    xpress_refiner *R = const_cast<xpress_refiner *>(Rc);
    if (!R || !in || !out) return XPRESS_ERR_INVALID_ARG;
    if (in->b < 1 || in->K_max < 1 || !in->h || !in->s || !in->anchor || !in->temperature || !in->seed ||
        !out->tokens)
        return XPRESS_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(in->s) & 15) || (reinterpret_cast<uintptr_t>(in->h) & 15))
        return XPRESS_ERR_INVALID_ARG;
    if ((in->mode != XPRESS_MODE_JACOBI && in->mode != XPRESS_MODE_SEQUENTIAL) ||
        (in->mode == XPRESS_MODE_SEQUENTIAL && in->K_max < R->w.B))
        return XPRESS_ERR_INVALID_ARG;
    const Layout L = make_layout(R, in->b);
    if (const int rc = check_ws(ws, ws_bytes, L.total)) return rc;
    Params P = make_params(R, in, out, ws, L);
    if (L.small && !eager_mode()) return run_small(R, P, L, ws, static_cast<cudaStream_t>(stream));
    if (eager_mode()) return run_eager(R, P, L, ws, static_cast<cudaStream_t>(stream), eager_mode() == 2);
    const bool draft_null = in->draft == nullptr;
    GraphEntry *hit = nullptr, *victim = &R->cache[0];
    for (auto &e : R->cache) {
        if (e.used && e.ws == ws && e.ws_bytes == ws_bytes && e.b == in->b && e.draft_null == draft_null) {
            hit = &e;
            break;
        }
        if (!e.used) victim = &e;
        else if (victim->used && e.stamp < victim->stamp) victim = &e;
    }
    if (!hit) {
        destroy_entry(*victim);
        victim->used = true;
        victim->ws = ws;
        victim->ws_bytes = ws_bytes;
        victim->b = in->b;
        victim->draft_null = draft_null;
        if (const int rc = build_graph(R, *victim, P, L, ws)) {
            destroy_entry(*victim);
            return rc;
        }
        hit = victim;
    }
    hit->stamp = ++R->clock;
    Params *pdev = reinterpret_cast<Params *>(static_cast<char *>(ws) + L.params);
    cudaGraphConditionalHandle handle = hit->handle;
    void *args[] = {&P, &pdev, &handle};
    cudaKernelNodeParams kp{};
    kp.func = reinterpret_cast<void *>(k_init);
    kp.gridDim = hit->init_grid;
    kp.blockDim = dim3(256);
    kp.kernelParams = args;
    XP_CUDA(cudaGraphExecKernelNodeSetParams(hit->exec, hit->init_node, &kp));
    if (L.pre_tc) {
        PreTcArgs a;
        if (!a.make(R, P, L, pdev)) return XPRESS_ERR_CUDA;
        cudaKernelNodeParams pk = a.node(L, P.N);
        XP_CUDA(cudaGraphExecKernelNodeSetParams(hit->exec, hit->pre_node, &pk));
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (R->trace) {
        XP_CUDA(cudaMemsetAsync(R->trace, 0xFF, TRACE_SLOTS * sizeof(unsigned long long), st));
        XP_CUDA(cudaMemsetAsync(R->trace + TRACE_SLOTS, 0, TRACE_SLOTS * sizeof(unsigned long long), st));
    }
    XP_CUDA(cudaGraphLaunch(hit->exec, st));
    if (R->trace) print_trace(R, st);
    return XPRESS_OK;
}

// ------------------------------------------------------------------ accept

namespace {
struct AcceptLayout {
    size_t status = 0, rowpart = 256, ticket = 0, draws = 0, keys = 0, total = 0;
    int chunks = 1, row_ctas = 1, draw_ctas = 1;
};

AcceptLayout accept_layout(const xpress_refiner *R, int b)
{
    AcceptLayout A;
    const int rows = b * (R->w.B + 1);
    // chunks per target row: enough items to spread a small batch over the
    // SMs, and chunks of at most 32768 ids so that a large batch's items
    // balance over the persistent grid
    int c = (2 * R->num_sms + rows - 1) / rows;
    const int cv = (R->w.V + 32767) / 32768;
    c = c > cv ? c : cv;
    A.chunks = c < 1 ? 1 : (c > 64 ? 64 : c);
    const int items = rows * A.chunks;
    A.row_ctas = items < 4 * R->num_sms ? items : 4 * R->num_sms;
    A.draw_ctas = 2 * R->num_sms;                 // two CTAs of k_acc_draw fit on an SM
    size_t o = A.rowpart + align256((size_t)rows * A.chunks * sizeof(Partial));
    A.ticket = o;
    o += 256;
    A.draws = o;
    o += align256((size_t)b * sizeof(DrawDesc));
    A.keys = o;
    o += align256((size_t)b * 2 * sizeof(unsigned long long));
    A.total = o;
    return A;
}
}  // namespace

}  // extern "C"

namespace xp {

int refiner_device(const xpress_refiner *R) { return R ? R->device : -1; }
const xpress_weights &refiner_weights(const xpress_refiner *R) { return R->w; }
int refiner_sms(const xpress_refiner *R) { return R->num_sms; }
unsigned long long refiner_wait_ns(const xpress_refiner *R) { return R->wait_ns; }
const CUtensorMap *refiner_tmap_wr128(const xpress_refiner *R) { return &R->tmap_wr128; }
cudaStream_t refiner_train_aux(const xpress_refiner *R, cudaEvent_t (&ev)[4])
{
    for (int i = 0; i < 4; ++i) ev[i] = R->train_ev[i];
    return R->train_aux;
}

bool tmap_bf16_kblocks(CUtensorMap *m, const void *base, uint64_t rows, uint32_t box_rows)
{
    return make_tmap_bf16_kblocks(m, base, rows, box_rows);
}

bool tmap_bf16(CUtensorMap *m, const void *base, uint64_t inner, uint64_t outer, uint64_t pitch, uint32_t box_inner,
               uint32_t box_outer)
{
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {pitch * 2};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t accept_scratch_bytes(const xpress_refiner *R, int b)
{
    if (!R || b < 1) return 0;
    return accept_layout(R, b).total;
}

int accept_launch(const xpress_refiner *R, const xpress_accept_in *in, int32_t *accept_len, int32_t *out_tokens,
                  void *ws, size_t ws_bytes, void *stream)
{
    if (!R || !in || !accept_len || !out_tokens) return XPRESS_ERR_INVALID_ARG;
    if (in->b < 1 || !in->target || !in->tokens || !in->temperature || !in->seed || !in->s || !in->lse ||
        !in->logit_sel || !in->z_final)
        return XPRESS_ERR_INVALID_ARG;
    const AcceptLayout A = accept_layout(R, in->b);
    if (const int rc = check_ws(ws, ws_bytes, A.total)) return rc;
    char *w = static_cast<char *>(ws);
    AcceptParams P{};
    P.b = in->b;
    P.B = R->w.B;
    P.V = R->w.V;
    P.dtype = R->w.dtype;
    P.target = in->target;
    P.s = in->s;
    P.tokens = in->tokens;
    P.lse = in->lse;
    P.logit_sel = in->logit_sel;
    P.z_final = in->z_final;
    P.temperature = in->temperature;
    P.seed = reinterpret_cast<const unsigned long long *>(in->seed);
    P.offset = in->offset;
    P.W_r = R->w.W_r;
    P.accept_len = accept_len;
    P.out_tokens = out_tokens;
    P.status = reinterpret_cast<int32_t *>(w + A.status);
    P.rowpart = reinterpret_cast<Partial *>(w + A.rowpart);
    P.ticket = reinterpret_cast<int32_t *>(w + A.ticket);
    P.draws = reinterpret_cast<DrawDesc *>(w + A.draws);
    P.keys = reinterpret_cast<unsigned long long *>(w + A.keys);
    P.chunks = A.chunks;
    P.fused = in->b <= ACCEPT_FUSED_MAX_B;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // each is chained to its predecessor with programmatic dependent launch
    // (k_acc_rows clears the status word, the draw counters and keys); small
    // batches skip k_acc_decide (the draw kernel's CTAs decide)
    XP_CUDA(launch_pdl(k_acc_rows, dim3(A.row_ctas), dim3(256), 0, st, P, A.chunks));
    if (!P.fused) XP_CUDA(launch_pdl(k_acc_decide, dim3(in->b), dim3(32), 0, st, P));
    XP_CUDA(launch_pdl(R->w.dtype == XPRESS_BF16 ? k_acc_draw : k_acc_draw_simt, dim3(A.draw_ctas), dim3(256), 0, st,
                       P));
    XP_CUDA(cudaGetLastError());
    return XPRESS_OK;
}

}  // namespace xp

extern "C" {


size_t xpress_accept_workspace_size(const xpress_refiner *R, int b)
{
    if (!R || b < 1) return 0;
    return accept_layout(R, b).total;
}

int xpress_accept(const xpress_refiner *R, const xpress_accept_in *in, int32_t *accept_len, int32_t *out_tokens,
                  void *ws, size_t ws_bytes, void *stream)
{
    return xp::accept_launch(R, in, accept_len, out_tokens, ws, ws_bytes, stream);
}

int xpress_get_device_status(void *ws, void *stream, int32_t *status_out)
{
    if (!ws || !status_out) return XPRESS_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int32_t v = 0;
    XP_CUDA(cudaStreamSynchronize(st));
    XP_CUDA(cudaMemcpy(&v, ws, 4, cudaMemcpyDeviceToHost));
    XP_CUDA(cudaMemset(ws, 0, 4));
    *status_out = (v & ST_TIMEOUT) ? XPRESS_ERR_TIMEOUT : (v & ST_BOUNDS) ? XPRESS_ERR_DEVICE_CHECK : XPRESS_OK;
    return XPRESS_OK;
}

int xpress_profile_read_prepare(const xpress_refiner *R, void *ws, int b, int n_tokens, void *stream)
{
    if (!R || b < 1 || n_tokens < 1 || n_tokens > b * R->w.B) return XPRESS_ERR_INVALID_ARG;
    const Layout L = make_layout(R, b);
    if (const int rc = check_ws(ws, L.total, L.total)) return rc;
    char *w = static_cast<char *>(ws);
    k_prof_prepare<<<(n_tokens + 255) / 256, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<int32_t *>(w + L.ctl), reinterpret_cast<int32_t *>(w + L.acttok), n_tokens);
    XP_CUDA(cudaGetLastError());
    return XPRESS_OK;
}

int xpress_profile_read(const xpress_refiner *R, void *ws, int b, void *stream)
{
    if (!R || b < 1) return XPRESS_ERR_INVALID_ARG;
    const Layout L = make_layout(R, b);
    if (const int rc = check_ws(ws, L.total, L.total)) return rc;
    char *w = static_cast<char *>(ws);
    const Params *pdev = reinterpret_cast<const Params *>(w + L.params);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (R->use_tc) {
        CUtensorMap tmap_z{};
        if (!make_tmap_bf16(&tmap_z, w + L.zpack, RANK, (uint64_t)b * R->w.B, 64, 32)) return XPRESS_ERR_CUDA;
        if (L.tcv)
            k_read_tcv<<<L.S, kReadTcvThreads, kReadTcvSmemBytes, st>>>(pdev, R->tmap_wr128, tmap_z, R->w.V, 0, 0);
        else
            k_read_tc<<<L.S, kReadTcThreads, kReadTcSmemBytes, st>>>(pdev, R->tmap_wr, tmap_z, R->w.V);
    } else {
        k_read_simt<<<L.S, 256, READ_SIMT_DYN_SMEM, st>>>(pdev);
    }
    XP_CUDA(cudaGetLastError());
    return XPRESS_OK;
}

int xpress_set_wait_limit(xpress_refiner *R, uint64_t limit_ns)
{
    if (!R || limit_ns > 60000000000ull) return XPRESS_ERR_INVALID_ARG;
    R->wait_ns = limit_ns;
    return XPRESS_OK;
}

int xpress_get_pass_count(void *ws, void *stream, int32_t *passes_out)
{
    if (!ws || !passes_out) return XPRESS_ERR_INVALID_ARG;
    XP_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    XP_CUDA(cudaMemcpy(passes_out, static_cast<char *>(ws) + 64 + CTL_PASS * 4, 4, cudaMemcpyDeviceToHost));
    return XPRESS_OK;
}

}  // extern "C"

// ------------------------------------------------------------------ base logits

namespace {
int lm_grid(int V)
{
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                  cudaSuccess) {
        (void)cudaGetLastError();
        return 0;
    }
    const int nvt = (V + 127) / 128;
    return nvt < sms ? nvt : sms;
}
}  // namespace

extern "C" {

size_t xpress_lm_head_workspace_size(int V, int N)
{
    if (V < 1 || N < 1) return 0;
    const int G = lm_grid(V);
    if (G < 1) return 0;
    return 256 + align256((size_t)N * G * sizeof(Partial));
}

int xpress_lm_head(const void *W_lm, int V, int H, const void *h, int N, void *s_out, int32_t *argmax_out,
                   void *ws, size_t ws_bytes, void *stream)
{
    if (!W_lm || !h || (!s_out && !argmax_out) || V < 1 || N < 1 || H < 8 || (H % 8)) return XPRESS_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(W_lm) & 15) || (reinterpret_cast<uintptr_t>(h) & 15))
        return XPRESS_ERR_INVALID_ARG;
    const int G = lm_grid(V);
    if (G < 1) return XPRESS_ERR_CUDA;
    if (const int rc = check_ws(ws, ws_bytes, 256 + align256((size_t)N * G * sizeof(Partial)))) return rc;
    if (set_kernel_attributes() != XPRESS_OK) return XPRESS_ERR_CUDA;
    const bool wide = N > 32;                       // token chunks of 256, else one chunk of 32
    CUtensorMap tw{}, th{};
    if (!make_tmap_bf16(&tw, W_lm, (uint64_t)H, (uint64_t)V, 64, 128) ||
        !make_tmap_bf16(&th, h, (uint64_t)H, (uint64_t)N, 64, wide ? 256 : 32))
        return XPRESS_ERR_CUDA;
    char *w = static_cast<char *>(ws);
    int32_t *status = reinterpret_cast<int32_t *>(w);
    Partial *part = reinterpret_cast<Partial *>(w + 256);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    XP_CUDA(cudaMemsetAsync(status, 0, 4, st));
    if (wide)
        k_lm_head256<<<G, kLmHeadThreads, kLmHeadSmemBytes[1], st>>>(tw, th, V, H, N,
                                                                        static_cast<uint16_t *>(s_out), part, status);
    else
        k_lm_head32<<<G, kLmHeadThreads, kLmHeadSmemBytes[0], st>>>(tw, th, V, H, N, static_cast<uint16_t *>(s_out),
                                                                       part, status);
    XP_CUDA(cudaGetLastError());
    if (argmax_out) XP_CUDA(launch_pdl(k_lm_head_argmax, dim3((unsigned)((N + 7) / 8)), dim3(256), 0, st,
                                       (const Partial *)part, G, N, argmax_out));
    return XPRESS_OK;
}

}  // extern "C"
