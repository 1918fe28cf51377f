// Internal launch interface between the C ABI (qx_api.cu) and the kernels.
#pragma once

#include <atomic>

#include <algorithm>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "qx_common.cuh"

namespace qx {

struct QuantArgs {
    const __half *W;
    int64_t n, k;
    int bits, g, kind, lloyd_iters;
    int G;       // groups per row
    int zbytes;  // zero-point bytes per row
    uint8_t *codes;
    __half *scales;
    uint8_t *zeros;
    __half *luts;
    uint32_t *status;
};

struct DequantArgs {
    const uint8_t *codes;
    const __half *scales;
    const uint8_t *zeros;
    const __half *luts;
    int64_t n, k;
    int bits, g, kind, G, zbytes;
    __half *W;
};

constexpr int kMaxGemvMats = 8;     // matrices of one group (one phase)
constexpr int kMaxGemvPhases = 4;   // groups of one fused launch (qx_gemv_fused)
constexpr int kMaxGemvTotal = 16;   // matrices of one launch over all its phases
constexpr int kMaxGemvCtas = 256;

// One matrix of a (multi-matrix) decode launch.  The fields after log2g are
// filled by plan_gemv().
struct GemvMat {
    const uint8_t *codes;
    const __half *scales;
    const uint8_t *zeros;
    const __half *luts;
    const __half *x;  // [batch][k]
    void *y;          // [batch][n]
    int64_t n, k;
    int G, zbytes, log2g;
    int nks;         // 1024-weight slices per row
    int nlb;         // LUT boxes (32 rows x 8 groups) per slice
    int nrb;         // 32-row blocks
    int rb_off;      // first row-block of this matrix in its phase's list
    int st_off;      // first stage (row block x slice) of this matrix in its phase's list
};

// A decode launch: one phase (qx_gemv_multi), or several phases run one after
// another by one persistent grid (qx_gemv_fused), each phase's x read only
// after every CTA has finished the phase before it.
struct GemvMulti {
    // scalars first: the kernel's set-up reads them before anything else
    int count, bits, kind, batch, y_f32;   // count: matrices over all phases
    int nphase;
    int phase_first[kMaxGemvPhases + 1];   // first matrix of each phase; [nphase] = count
    int grid, ring, rb_slots, stage_bytes, red_bytes, tab_bytes, smem_bytes;
    int64_t total_bytes;
    uint32_t *status;
    uint32_t *phase_ctr;                   // nphase counters (nphase > 1): zero between launches
    // Row blocks split between two CTAs (allowed when split_part is set; the
    // plan sets has_split when it uses that): the CTA with the block's later
    // slices stores their fp32 sums to split_part [CTA][16][32] and raises
    // split_flag[CTA] (zero between launches); the CTA with the earlier slices
    // adds them to its own and writes y
    float *split_part;
    uint32_t *split_flag;
    int has_split;
    uint64_t wait_limit_ns;
    GemvMat mat[kMaxGemvTotal];
    // per phase, the first stage (row block x 1024-weight slice) of every CTA
    // in the phase's list, byte-balanced on the host; at whole row blocks
    // unless split_part is set.  cta_st[p][grid] = the phase's stages
    int32_t cta_st[kMaxGemvPhases][kMaxGemvCtas + 1];
    CUtensorMap tm_codes[kMaxGemvTotal];  // packed codes, 32-row x 128-byte boxes
    CUtensorMap tm_luts[kMaxGemvTotal];   // LUTs, 32-row x 128-byte boxes (LUT kind)
};

struct GemmArgs {
    const uint8_t *codes;
    const __half *scales;
    const uint8_t *zeros;
    const __half *luts;
    int64_t n, k, m;
    int bits, kind, log2g, G, zbytes;
    const __half *X;  // [m][k]
    __half *Y;        // [m][n]
    uint32_t *status;
    uint64_t wait_limit_ns;
    // packed-code ring (filled by launch_gemm): slots of one 128-weight
    // superblock of a 128-row W tile
    int pslots, pslot_bytes, lut_box;
    int smem_bytes;
    // token tile (16 or 256) and the number of k splits of every tile (from
    // plan_gemm); with splits > 1, ws_cnt [tiles][4] counts the row quarters
    // that have stored their fp32 partial tiles to ws_part [units][bn][128]
    int bn, splits;
    float *ws_part;
    uint32_t *ws_cnt;
    // launched with programmatic dependent launch: the weight-side roles start
    // while the previous kernel runs; X is read and Y / the workspace written
    // only after it has finished
    int pdl;
};

// A split-k workspace starts with a fixed region of counters (one word per
// row quarter of a tile, so at most 4096 tiles split), which every completed
// call leaves zero whatever the shapes of earlier calls; the fp32 partial
// tiles follow it.
constexpr size_t kSplitCounterBytes = 65536;

// Tiling of one prefill/decode matmul on the tensor cores.
struct GemmPlan {
    int bn;            // tokens per tile: 16 for m <= 16, else 256
    int splits;        // k splits per tile (1: no workspace)
    int64_t tiles;     // token tiles x 128-row W tiles
    int64_t units;     // tiles x splits
    size_t ws_bytes;   // workspace the split needs (0 when splits == 1)
};

// allow_split = false: one CTA per tile (qx_gemm); true: k is split when the
// tile grid leaves SMs idle (qx_gemm_splitk).
GemmPlan plan_gemm(int64_t n, int64_t k, int64_t m, int num_sms, bool allow_split);

// W.A8 decode (uniform weights, int8 per-token activations).
struct GemvA8Args {
    const uint8_t *codes;
    const __half *scales;
    const uint8_t *zeros;
    int64_t n, k;
    int bits, G, zbytes, log2g;
    const int8_t *q;          // [batch][k]
    const float *act_scales;  // [batch]
    int batch;
    void *y;                  // [batch][n]
    int y_f32;
};
cudaError_t launch_quantize_act(const __half *x, int batch, int64_t k, int8_t *q, float *scales, cudaStream_t st);
cudaError_t launch_dequant_act(const int8_t *q, const float *scales, int64_t m, int64_t k, __half *xh, int num_sms,
                              cudaStream_t st);
cudaError_t launch_gemv_a8(const GemvA8Args &a, cudaStream_t st);

// Exact sum of (W - W_hat)^2 2^48 over `count` fp16 elements (a multiple of 8,
// 16-byte aligned): per-block partials (2 words per block, sq_error_blocks of
// them) and the total in out[0] (low word), out[1].
int sq_error_blocks(int num_sms);
cudaError_t launch_sq_error(const __half *W, const __half *W_hat, int64_t count, unsigned long long *partials,
                            unsigned long long *out, int num_sms, cudaStream_t st);

// Size of the file-scope scratch that qx_gemm_splitk_noalloc uses in place of
// a workspace, and its device address on the current device (looked up once
// per device with cudaGetSymbolAddress).
constexpr size_t kNoAllocScratchBytes = (size_t)4 << 20;
cudaError_t noalloc_scratch(void **ptr);

// Raise a kernel's dynamic shared-memory limit to the 227 KB maximum (and the
// preferred carveout to all shared memory) once per device: a driver call per
// launch would cost host time on every decode step.  `ready` holds one bit per
// device (devices 0..63; others set the attributes every time).
inline cudaError_t ensure_kernel_attrs(const void *kern, std::atomic<uint64_t> &ready, bool carveout) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = (dev >= 0 && dev < 64) ? (1ull << dev) : 0ull;
    if (bit != 0 && (ready.load(std::memory_order_acquire) & bit) != 0) return cudaSuccess;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e == cudaSuccess && carveout) e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e == cudaSuccess && bit != 0) ready.fetch_or(bit, std::memory_order_acq_rel);
    return e;
}

// Q4X shared-codebook matrices: groups of 64 weights with an fp16 scale and a
// 2-bit book index (four per byte), 4-bit codes in the 4-bit layout, and four
// codebooks of 16 fp16 levels per matrix.
constexpr int kQ4xGroup = 64;

struct Q4xMat {
    const uint8_t *codes;     // [n][k/2]
    const __half *scales;     // [n][G]
    const uint8_t *books;     // [n][bbytes]
    const __half *codebooks;  // [4][16]
    int64_t n, k;
    int G, bbytes;            // G = k/64, bbytes = ceil(G/4)
};

struct Q4xQuantArgs {
    const __half *W;  // [n][k]
    int64_t n, k;
    int G, bbytes, iters;
    uint8_t *codes;
    __half *scales;
    uint8_t *books;
    __half *codebooks;
    void *ws;  // q4x_workspace_bytes(n, k), 256-byte aligned
    uint32_t *status;
};

// Decode matmul over up to eight Q4X matrices in one launch: y[i] = x[i] W_i^T.
constexpr int kMaxQ4xMats = 8;
struct Q4xGemvMulti {
    int count, batch, y_f32;
    Q4xMat mat[kMaxQ4xMats];
    const __half *x[kMaxQ4xMats];  // [batch][k_i]
    void *y[kMaxQ4xMats];          // [batch][n_i]
    int64_t row_off[kMaxQ4xMats + 1];  // first row of matrix i in the launch's row list
};

size_t q4x_workspace_bytes(int64_t n, int64_t k);
cudaError_t launch_q4x_quantize(const Q4xQuantArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_q4x_dequant(const Q4xMat &m, __half *W, int num_sms, cudaStream_t st);
cudaError_t launch_q4x_gemv(const Q4xGemvMulti &a, int num_sms, cudaStream_t st);

// One CTA whose bounded mbarrier wait runs out (nothing arrives): records
// kStatusTimeout in *status after limit_ns and returns.
cudaError_t launch_wait_selftest(uint64_t limit_ns, uint32_t *status, cudaStream_t st);

cudaError_t launch_quantize(const QuantArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_dequant(const DequantArgs &a, int num_sms, cudaStream_t st);
bool plan_gemv(GemvMulti &a, int num_sms);
cudaError_t launch_gemv_multi(GemvMulti &a, cudaStream_t st, bool pdl);
cudaError_t launch_gemm(const GemmArgs &a, int num_sms, cudaStream_t st);

// Copies of a decode step done by a kernel (qx_copy.cu): src and dst are
// device-accessible addresses (a pinned host buffer's mapped device address
// on the host side); `bytes` each.  pdl: launched with programmatic dependent
// launch, so that it waits for the previous kernel in the stream inside the
// kernel rather than before it starts.
constexpr int kMaxCopies = 16;
struct CopyList {
    int n;
    const uint8_t *src[kMaxCopies];
    uint8_t *dst[kMaxCopies];
    int64_t bytes[kMaxCopies];
};
cudaError_t launch_copies(const CopyList &c, int num_sms, bool pdl, cudaStream_t st);

// cuTensorMapEncodeTiled, fetched once through the runtime's driver entry
// point (null if the driver does not provide it).
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_fn();

}  // namespace qx
