// Internal launch interface between the C ABI (qx_api.cu) and the kernels.
#pragma once

#include <algorithm>
#include <cstdint>
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

constexpr int kMaxGemvMats = 8;

// One matrix of a (multi-matrix) decode launch.  The geometry fields after
// log2g are filled by plan_gemv().
struct GemvMat {
    const uint8_t *codes;
    const __half *scales;
    const uint8_t *zeros;
    const __half *luts;
    const __half *x;  // [batch][k]
    void *y;          // [batch][n]
    int64_t n, k;
    int G, zbytes, log2g;
    int CB, LB, SB, ZB, row_bytes, RB;
    int64_t byte_off;
};

constexpr int kMaxGemvCtas = 1024;

struct GemvMulti {
    GemvMat mat[kMaxGemvMats];
    // first row of every CTA in the concatenation of all matrices' rows
    // (byte-balanced slices computed on the host); cta_row[grid] = total rows
    int64_t cta_row[kMaxGemvCtas + 1];
    int64_t row_off[kMaxGemvMats + 1];  // first concatenated row of each matrix
    int count, bits, kind, batch, y_f32;
    int grid, stages, stage_bytes, x_smem_bytes, smem_bytes;
    int64_t total_bytes;
    uint32_t *status;
    uint64_t wait_limit_ns;
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
};

cudaError_t launch_quantize(const QuantArgs &a, int num_sms, cudaStream_t st);
cudaError_t launch_dequant(const DequantArgs &a, int num_sms, cudaStream_t st);
bool plan_gemv(GemvMulti &a, int num_sms);
cudaError_t launch_gemv_multi(const GemvMulti &a, cudaStream_t st, bool pdl);
cudaError_t launch_gemm(const GemmArgs &a, int num_sms, cudaStream_t st);

}  // namespace qx
