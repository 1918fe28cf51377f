// Exact squared Frobenius error between a weight matrix and its dequantized
// image, the measure by which a recipe is chosen per matrix (paper Sections
// 2.2-2.3: uniform or non-uniform per matrix by the error norm).
//
// fp16 values are integer multiples of 2^-24 (|w| <= 65504 < 2^16), so
// (w - w_hat) 2^24 is an integer below 2^41 and its square fits in 128 bits;
// sums of up to 2^36 of them stay below 2^118.  Every partial sum is an exact
// integer, so the result does not depend on the order of the additions.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kErrThreads = 256;

using u128 = unsigned __int128;

__device__ __forceinline__ long long scaled24(__half h) {
    return (long long)((double)__half2float(h) * 16777216.0);  // exact
}

__device__ __forceinline__ u128 sq_diff8(uint4 a, uint4 b) {
    const __half *ha = reinterpret_cast<const __half *>(&a);
    const __half *hb = reinterpret_cast<const __half *>(&b);
    u128 s = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const long long d = scaled24(ha[j]) - scaled24(hb[j]);
        const unsigned long long ad = (unsigned long long)(d < 0 ? -d : d);
        s += (u128)ad * ad;
    }
    return s;
}

// Per-block partial sums (two words each, low first) of (W - W_hat)^2 2^48.
__global__ void __launch_bounds__(kErrThreads) sq_err_kernel(const uint4 *W, const uint4 *Wh, int64_t nvec,
                                                             unsigned long long *partials) {
    __shared__ u128 red[kErrThreads];
    u128 acc = 0;
    for (int64_t i = (int64_t)blockIdx.x * kErrThreads + threadIdx.x; i < nvec; i += (int64_t)gridDim.x * kErrThreads)
        acc += sq_diff8(W[i], Wh[i]);
    red[threadIdx.x] = acc;
    __syncthreads();
    for (int s = kErrThreads / 2; s > 0; s >>= 1) {
        if ((int)threadIdx.x < s) red[threadIdx.x] += red[threadIdx.x + s];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        partials[2 * blockIdx.x] = (unsigned long long)red[0];
        partials[2 * blockIdx.x + 1] = (unsigned long long)(red[0] >> 64);
    }
}

__global__ void sum_partials_kernel(const unsigned long long *partials, int blocks, unsigned long long *out) {
    if (threadIdx.x != 0) return;
    u128 s = 0;
    for (int b = 0; b < blocks; ++b) s += ((u128)partials[2 * b + 1] << 64) | partials[2 * b];
    out[0] = (unsigned long long)s;
    out[1] = (unsigned long long)(s >> 64);
}

}  // namespace

int sq_error_blocks(int num_sms) { return 4 * (num_sms > 0 ? num_sms : 1); }

cudaError_t launch_sq_error(const __half *W, const __half *W_hat, int64_t count, unsigned long long *partials,
                            unsigned long long *out, int num_sms, cudaStream_t st) {
    const int blocks = sq_error_blocks(num_sms);
    sq_err_kernel<<<blocks, kErrThreads, 0, st>>>(reinterpret_cast<const uint4 *>(W),
                                                  reinterpret_cast<const uint4 *>(W_hat), count / 8, partials);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    sum_partials_kernel<<<1, 32, 0, st>>>(partials, blocks, out);
    return cudaGetLastError();
}

}  // namespace qx
