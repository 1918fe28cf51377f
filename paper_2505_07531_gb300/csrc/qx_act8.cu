// W.A8 decode: 8-bit per-token activations against uniform 3/4-bit weights
// with integer dot products (paper Table 2: "8-bit RTN per-token quantization
// for the activation tensors"; Table 1: W3A8).
//
//   activations, per token b:  s_b = fp32(max|x_b| / 127),
//                              q = clamp(rint(x / s_b), -127, 127) (int8)
//   matmul:  y[b][n] = s_b * sum_g s_g * sum_{k in g} (q_w - z) q[b][k]
//
// The group sums are exact 32-bit integers from dp4a (four int8 products per
// instruction); the scales are applied in fp32.  One warp per weight row;
// lane l takes the 32-weight units l, l + 32, ... of the row, so a warp's code
// loads are contiguous.  Non-uniform (LUT) weights have no integer form.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kActThreads = 1024;
constexpr int kA8Warps = 8;  // rows per block

__global__ void __launch_bounds__(kActThreads) quantize_act_kernel(const __half *x, int64_t k, int8_t *q,
                                                                   float *scales) {
    __shared__ float red[kActThreads / 32];
    const __half *xr = x + (int64_t)blockIdx.x * k;
    float m = 0.0f;
    for (int64_t i = threadIdx.x; i < k; i += kActThreads) m = fmaxf(m, fabsf(__half2float(xr[i])));
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x < 32) {
        m = red[threadIdx.x];
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (threadIdx.x == 0) red[0] = m;
    }
    __syncthreads();
    const float s = __fdiv_rn(red[0], 127.0f);  // IEEE division
    int8_t *qr = q + (int64_t)blockIdx.x * k;
    for (int64_t i = threadIdx.x; i < k; i += kActThreads) {
        float v = 0.0f;
        if (s > 0.0f) v = fminf(fmaxf(rintf(__fdiv_rn(__half2float(xr[i]), s)), -127.0f), 127.0f);
        qr[i] = (int8_t)(int)v;
    }
    if (threadIdx.x == 0) scales[blockIdx.x] = s;
}

// W.A8 prefill: the tensor cores take fp16 operands, so the int8 activations
// enter the matmul as x_hat = fp16(fp32(s_b q)), one IEEE fp32 product then a
// round to nearest even.  One thread per 16 codes: a 16-byte load, two
// 16-byte stores.
constexpr int kDqThreads = 256;

__global__ void __launch_bounds__(kDqThreads) dequant_act_kernel(const int8_t *q, const float *scales, int64_t m,
                                                                 int64_t k, __half *xh) {
    const int64_t vpr = k / 16, total = m * vpr;
    for (int64_t i = (int64_t)blockIdx.x * kDqThreads + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * kDqThreads) {
        const float s = scales[i / vpr];
        const uint4 v = reinterpret_cast<const uint4 *>(q)[i];
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
        uint32_t o[8];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int c0 = (int)(int8_t)((w[t] >> (16 * e)) & 0xffu);
                const int c1 = (int)(int8_t)((w[t] >> (16 * e + 8)) & 0xffu);
                const uint32_t h0 = __half_as_ushort(__float2half_rn(__fmul_rn(s, (float)c0)));
                const uint32_t h1 = __half_as_ushort(__float2half_rn(__fmul_rn(s, (float)c1)));
                o[2 * t + e] = h0 | (h1 << 16);
            }
        }
        uint4 *dst = reinterpret_cast<uint4 *>(xh) + 2 * i;
        dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
        dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
    }
}

__device__ __forceinline__ uint32_t prmt_b(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// 32 signed bytes (q_w - z) of one 3-bit unit (words A, B, C of its
// superblock), in natural k order, 4 per word.
__device__ __forceinline__ void offsets3(uint32_t A, uint32_t B, uint32_t C, uint32_t z, uint32_t (&o)[8]) {
    // byte table of (j - z) mod 256, j = 0..7, as two words (entries 0-3, 4-7);
    // byte-wise subtraction, as a borrow must not cross bytes
    const uint32_t zz = z * 0x01010101u;
    const uint32_t lo = __vsub4(0x03020100u, zz), hi = __vsub4(0x07060504u, zz);
    const uint32_t m = 0x77777777u;
    const uint32_t a = A & m, b = B & m, c = C & m;
    const uint32_t e = ((A >> 3) & 0x11111111u) | ((B >> 2) & 0x22222222u) | ((C >> 1) & 0x44444444u);
    o[0] = prmt_b(lo, hi, a);
    o[1] = prmt_b(lo, hi, a >> 16);
    o[2] = prmt_b(lo, hi, b);
    o[3] = prmt_b(lo, hi, b >> 16);
    o[4] = prmt_b(lo, hi, c);
    o[5] = prmt_b(lo, hi, c >> 16);
    o[6] = prmt_b(lo, hi, e);
    o[7] = prmt_b(lo, hi, e >> 16);
}

template <int BITS, int NB>
__global__ void __launch_bounds__(32 * kA8Warps) gemv_a8_kernel(GemvA8Args a) {
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * kA8Warps + (threadIdx.x >> 5);
    if (row >= a.n) return;
    const int units = (int)(a.k / 32);
    float acc[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) acc[b] = 0.0f;
    const uint8_t *zrow = a.zeros + row * a.zbytes;
    const __half *srow = a.scales + row * a.G;
    for (int u = lane; u < units; u += 32) {
        const int grp = (32 * u) >> a.log2g;
        const float sg = __half2float(srow[grp]);
        const uint32_t z = (zrow[grp >> 1] >> ((grp & 1) * 4)) & 15u;
        uint32_t o[8];  // 32 weights as bytes in natural k order, 4 per word
        bool signed_off = true;
        if (BITS == 3) {
            const uint8_t *c = a.codes + row * (a.k * 3 / 8);
            const int64_t off = 16 * (u >> 2) + 4 * (u & 3);
            const uint32_t A = __ldg(reinterpret_cast<const uint32_t *>(c + off));
            const uint32_t B = __ldg(reinterpret_cast<const uint32_t *>(c + a.k / 8 + off));
            const uint32_t C = __ldg(reinterpret_cast<const uint32_t *>(c + a.k / 4 + off));
            offsets3(A, B, C, z, o);  // (q - z), signed bytes
        } else {
            const uint4 w = __ldg(reinterpret_cast<const uint4 *>(a.codes + row * (a.k / 2) + 16 * (int64_t)u));
            const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                // nibble j/2 + 4 (j % 2) holds k = 8t + j: low nibbles give j = 0,4,1,5,
                // high nibbles j = 2,6,3,7; put them back in k order
                const uint32_t lo = ws[t] & 0x0F0F0F0Fu, hi = (ws[t] >> 4) & 0x0F0F0F0Fu;
                o[2 * t] = prmt_b(lo, hi, 0x6420u);
                o[2 * t + 1] = prmt_b(lo, hi, 0x7531u);
            }
            signed_off = false;  // codes 0..15; the zero-point enters as z * sum(q_x)
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            if (b >= a.batch) break;
            const int4 *xq = reinterpret_cast<const int4 *>(a.q + (int64_t)b * a.k + 32 * (int64_t)u);
            const int4 x0 = __ldg(xq), x1 = __ldg(xq + 1);
            const int xs[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
            int dot = 0;
            if (signed_off) {
#pragma unroll
                for (int i = 0; i < 8; ++i) dot = __dp4a((int)o[i], xs[i], dot);
            } else {
                int sx = 0;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    dot = __dp4a((int)o[i], xs[i], dot);      // codes 0..15 x signed activations
                    sx = __dp4a(0x01010101, xs[i], sx);      // sum of the unit's activations
                }
                dot -= (int)z * sx;
            }
            acc[b] = fmaf(sg, (float)dot, acc[b]);
        }
    }
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        float v = acc[b];
        for (int o2 = 16; o2 > 0; o2 >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o2);
        acc[b] = v;
    }
    if (lane == 0) {
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            if (b >= a.batch) break;
            const float y = acc[b] * a.act_scales[b];
            if (a.y_f32)
                reinterpret_cast<float *>(a.y)[(int64_t)b * a.n + row] = y;
            else
                reinterpret_cast<__half *>(a.y)[(int64_t)b * a.n + row] = __float2half_rn(y);
        }
    }
}

template <int BITS>
cudaError_t launch_a8_bits(const GemvA8Args &a, cudaStream_t st) {
    const unsigned grid = (unsigned)((a.n + kA8Warps - 1) / kA8Warps);
    const int nb = a.batch;
    if (nb <= 1) gemv_a8_kernel<BITS, 1><<<grid, 32 * kA8Warps, 0, st>>>(a);
    else if (nb <= 2) gemv_a8_kernel<BITS, 2><<<grid, 32 * kA8Warps, 0, st>>>(a);
    else if (nb <= 4) gemv_a8_kernel<BITS, 4><<<grid, 32 * kA8Warps, 0, st>>>(a);
    else if (nb <= 8) gemv_a8_kernel<BITS, 8><<<grid, 32 * kA8Warps, 0, st>>>(a);
    else gemv_a8_kernel<BITS, 16><<<grid, 32 * kA8Warps, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_quantize_act(const __half *x, int batch, int64_t k, int8_t *q, float *scales, cudaStream_t st) {
    quantize_act_kernel<<<batch, kActThreads, 0, st>>>(x, k, q, scales);
    return cudaGetLastError();
}

cudaError_t launch_dequant_act(const int8_t *q, const float *scales, int64_t m, int64_t k, __half *xh, int num_sms,
                              cudaStream_t st) {
    const int64_t need = (m * (k / 16) + kDqThreads - 1) / kDqThreads;
    const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(need, (int64_t)num_sms * 8));
    dequant_act_kernel<<<grid, kDqThreads, 0, st>>>(q, scales, m, k, xh);
    return cudaGetLastError();
}

cudaError_t launch_gemv_a8(const GemvA8Args &a, cudaStream_t st) {
    return a.bits == 3 ? launch_a8_bits<3>(a, st) : launch_a8_bits<4>(a, st);
}

}  // namespace qx
