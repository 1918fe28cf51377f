// Decode matmul y[b][n] = sum_k w_hat[n][k] x[b][k] on CUDA cores.
//
// Decoding reads every weight once per token, so it is bound by HBM bandwidth
// and by the cost of unpacking the codes (paper Section 2.4).  Per 32-weight
// unit a lane issues one 16-byte coalesced code load (4-bit) or three (one per
// plane of a 128-weight 3-bit superblock), turns the codes into fp16 with the
// magic-number / byte-permute primitives, and multiplies them with x staged in
// shared memory using packed half2 FMAs.  The uniform scale is folded out of
// the inner loop: a unit contributes s * sum (q - z) x, accumulated in fp32.
// The LUT family contributes sum LUT[q] x.  Each 32-weight partial sum is a
// half2 FMA chain of 16 products, promoted to fp32 before it joins the row
// total; rows are finished by an fp32 warp-shuffle reduction.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float dot16(const __half2 (&w)[16], const __half *xs) {
    const uint4 *xv = reinterpret_cast<const uint4 *>(xs);
    __half2 acc = __float2half2_rn(0.0f);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint4 v = xv[q];
        acc = __hfma2(w[4 * q + 0], u2h2(v.x), acc);
        acc = __hfma2(w[4 * q + 1], u2h2(v.y), acc);
        acc = __hfma2(w[4 * q + 2], u2h2(v.z), acc);
        acc = __hfma2(w[4 * q + 3], u2h2(v.w), acc);
    }
    const float2 f = __half22float2(acc);
    return f.x + f.y;
}

template <int BITS, int KIND, int BMAX, int R>
__global__ void __launch_bounds__(kThreads) gemv_kernel(GemvArgs a) {
    extern __shared__ __align__(16) uint8_t smem_x[];
    __half *sx = reinterpret_cast<__half *>(smem_x);
    const int nb = a.batch;
    const int64_t K = a.k;
    {   // stage x [nb][K] into shared memory
        const uint4 *src = reinterpret_cast<const uint4 *>(a.x);
        uint4 *dst = reinterpret_cast<uint4 *>(sx);
        const int64_t vecs = (int64_t)nb * K / 8;
        for (int64_t i = threadIdx.x; i < vecs; i += blockDim.x) dst[i] = src[i];
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int warps = blockDim.x >> 5;
    const int64_t tiles = (a.n + R - 1) / R;
    const int G = a.G;
    for (int64_t tile = (int64_t)blockIdx.x * warps + warp; tile < tiles;
         tile += (int64_t)gridDim.x * warps) {
        float acc[R][BMAX];
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int b = 0; b < BMAX; ++b) acc[r][b] = 0.0f;
        if (BITS == 4) {
            const int64_t units = K / 32;
            for (int64_t j = lane; j < units; j += 32) {
                const int grp = (int)((32 * j) >> a.log2g);
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int64_t row = tile * R + r;
                    if (row >= a.n) break;
                    const uint4 c = ldg_nc_v4(a.codes + row * (K / 2) + 16 * j);
                    const uint32_t z = zero_nibble(a.zeros + row * a.zbytes, grp);
                    const float s = __half2float(a.scales[row * G + grp]);
                    const __half2 zl = zlo_of(z), zh = zhi_of(z);
                    __half2 w[16];
                    const uint32_t wd[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
                    for (int t = 0; t < 4; ++t) {
                        __half2 o[4];
                        unpack4_qz(wd[t], zl, zh, o);
#pragma unroll
                        for (int p = 0; p < 4; ++p) w[4 * t + p] = o[p];
                    }
#pragma unroll
                    for (int b = 0; b < BMAX; ++b)
                        if (b < nb) acc[r][b] += s * dot16(w, sx + b * K + 32 * j);
                }
            }
        } else {
            const int64_t units = K / 128;
            const int64_t plane = K >> 3;
            for (int64_t j = lane; j < units; j += 32) {
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int64_t row = tile * R + r;
                    if (row >= a.n) break;
                    const uint8_t *rc = a.codes + row * (3 * K / 8) + 16 * j;
                    const uint4 pa = ldg_nc_v4(rc);
                    const uint4 pb = ldg_nc_v4(rc + plane);
                    const uint4 pc = ldg_nc_v4(rc + 2 * plane);
                    const uint32_t A[4] = {pa.x, pa.y, pa.z, pa.w};
                    const uint32_t Bw[4] = {pb.x, pb.y, pb.z, pb.w};
                    const uint32_t C[4] = {pc.x, pc.y, pc.z, pc.w};
                    Table8 tab;
                    float s = 1.0f;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int64_t k0 = 128 * j + 32 * i;
                        const int grp = (int)(k0 >> a.log2g);
                        if (i == 0 || a.log2g < 7) {
                            if (KIND == 1) {
                                const uint4 l = ldg_nc_v4(a.luts + ((int64_t)row * G + grp) * 8);
                                tab = make_table8(l.x, l.y, l.z, l.w);
                            } else {
                                tab = table8_offsets(zero_nibble(a.zeros + row * a.zbytes, grp));
                                s = __half2float(a.scales[row * G + grp]);
                            }
                        }
                        __half2 w[16];
                        lookup_triple(tab, A[i], Bw[i], C[i], w);
#pragma unroll
                        for (int b = 0; b < BMAX; ++b)
                            if (b < nb) acc[r][b] += s * dot16(w, sx + b * K + k0);
                    }
                }
            }
        }
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int64_t row = tile * R + r;
#pragma unroll
            for (int b = 0; b < BMAX; ++b) {
                const float v = warp_sum(acc[r][b]);
                if (lane == 0 && row < a.n && b < nb) {
                    if (a.y_f32)
                        reinterpret_cast<float *>(a.y)[(int64_t)b * a.n + row] = v;
                    else
                        reinterpret_cast<__half *>(a.y)[(int64_t)b * a.n + row] = __float2half_rn(v);
                }
            }
        }
    }
}

template <int BITS, int KIND, int BMAX, int R>
cudaError_t launch_one(const GemvArgs &a, int num_sms, cudaStream_t st) {
    const size_t smem = (size_t)a.batch * a.k * sizeof(__half);
    auto kern = gemv_kernel<BITS, KIND, BMAX, R>;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    const int64_t tiles = (a.n + R - 1) / R;
    const int warps = kThreads / 32;
    int per_sm = 1;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem);
    per_sm = std::max(per_sm, 1);
    const int64_t blocks = std::min<int64_t>((tiles + warps - 1) / warps, (int64_t)num_sms * per_sm);
    kern<<<(unsigned)blocks, kThreads, smem, st>>>(a);
    return cudaGetLastError();
}

template <int BITS, int KIND>
cudaError_t launch_bits(const GemvArgs &a, int num_sms, cudaStream_t st) {
    if (a.batch <= 1) return launch_one<BITS, KIND, 1, 2>(a, num_sms, st);
    if (a.batch <= 2) return launch_one<BITS, KIND, 2, 2>(a, num_sms, st);
    if (a.batch <= 4) return launch_one<BITS, KIND, 4, 1>(a, num_sms, st);
    if (a.batch <= 8) return launch_one<BITS, KIND, 8, 1>(a, num_sms, st);
    return launch_one<BITS, KIND, 16, 1>(a, num_sms, st);
}

}  // namespace

// Batches whose staged activations exceed the shared-memory budget are split
// into chunks that each stream the weights once.
cudaError_t launch_gemv(const GemvArgs &a0, int num_sms, cudaStream_t st) {
    const int64_t budget = 200 * 1024;
    int chunk = a0.batch;
    while (chunk > 1 && (int64_t)chunk * a0.k * 2 > budget) chunk = (chunk + 1) / 2;
    for (int b0 = 0; b0 < a0.batch; b0 += chunk) {
        GemvArgs a = a0;
        a.batch = std::min(chunk, a0.batch - b0);
        a.x = a0.x + (int64_t)b0 * a0.k;
        const int esz = a0.y_f32 ? 4 : 2;
        a.y = reinterpret_cast<uint8_t *>(a0.y) + (int64_t)b0 * a0.n * esz;
        cudaError_t e;
        if (a.bits == 4)
            e = launch_bits<4, 0>(a, num_sms, st);
        else if (a.kind == 1)
            e = launch_bits<3, 1>(a, num_sms, st);
        else
            e = launch_bits<3, 0>(a, num_sms, st);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace qx
