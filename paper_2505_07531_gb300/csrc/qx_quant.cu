// Quantize (fp16 W -> packed codes + scales/zeros or LUTs) and dequantize
// (packed -> fp16 W_hat) kernels.  Both must agree bit for bit with the CPU
// oracle, so the arithmetic below follows the definitions exactly:
//   uniform (paper Section 2.2 equally spaced points, Section 3.2 RTN on a group,
//   asymmetric scale + minimum):
//     lo = min(0, min w), hi = max(0, max w)
//     s16 = fp16_rn(fp32(hi - lo) / (2^b - 1)), s = float(s16)
//     s16 == 0 -> z = 0, q = 0; else z = clamp(rint(-lo/s)), q = clamp(rint(w/s) + z)
//   non-uniform (Section 2.2, Fig. 2a: a per-group codebook where the mass is),
//   fit by Lloyd-Max with quantile initialisation, float64 nearest-level
//   assignment (ties to the lowest index), exact cell sums, one float64 division
//   per level, early stop when an assignment repeats, ascending sort, one
//   float64 -> fp16 rounding, final nearest-entry codes.
// IEEE operations are spelled out (__fdiv_rn, __fsub_rn, rintf, __ddiv_rn) so
// that no contraction or approximate division can change a result.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kWarp = 32;

__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ uint16_t f64_to_f16_bits(double x) {
    // One IEEE rounding, round to nearest even, straight from float64.
    uint16_t h;
    asm("cvt.rn.f16.f64 %0, %1;" : "=h"(h) : "d"(x));
    return h;
}

__device__ __forceinline__ double f16_bits_to_f64(uint16_t b) {
    return (double)__half2float(__ushort_as_half(b));  // exact
}

// Pack the codes of one group (held in shared memory, one byte per code) into
// the layout of include/qx.h.  `k0` is the group's first column; every lane
// of the warp calls this.
__device__ void pack_group(const uint8_t *sc, int g, int bits, int64_t k0, int64_t k,
                           uint8_t *row_codes, int lane) {
    if (bits == 4) {
        for (int t = lane; t < g / 8; t += kWarp) {
            const uint8_t *c = sc + 8 * t;
            uint32_t w = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) w |= (uint32_t)c[j] << (4 * (j / 2 + 4 * (j % 2)));
            reinterpret_cast<uint32_t *>(row_codes + (k0 >> 1))[t] = w;
        }
    } else {
        const int triples = g / 32;
        for (int t = lane; t < 3 * triples; t += kWarp) {
            const int tri = t / 3, plane = t % 3;
            const uint8_t *c = sc + 32 * tri;
            const int64_t kk = k0 + 32 * tri;
            const int64_t s = kk >> 7;
            const int i = (int)((kk & 127) >> 5);
            uint32_t w = 0;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                w |= (uint32_t)(c[8 * plane + u] & 7u) << (4 * u);
                w |= (uint32_t)((c[24 + u] >> plane) & 1u) << (4 * u + 3);
            }
            uint8_t *dst = row_codes + plane * (k >> 3) + 16 * s + 4 * i;
            *reinterpret_cast<uint32_t *>(dst) = w;
        }
    }
}

// ------------------------------------------------------------ uniform quantize
// One warp per pair of groups of a row (the two groups share a zero-point byte).
__global__ void __launch_bounds__(256) quantize_uniform_kernel(QuantArgs a) {
    extern __shared__ uint8_t smem_codes[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int warps = blockDim.x >> 5;
    const int g = a.g;
    const int E = g / kWarp;  // weights per lane per group (1..8)
    uint8_t *sc = smem_codes + warp * g;
    const int pairs_per_row = (a.G + 1) / 2;
    const int64_t total = (int64_t)a.n * pairs_per_row;
    const float qmax = (float)((1 << a.bits) - 1);
    for (int64_t task = (int64_t)blockIdx.x * warps + warp; task < total;
         task += (int64_t)gridDim.x * warps) {
        const int64_t row = task / pairs_per_row;
        const int pair = (int)(task % pairs_per_row);
        uint32_t zbyte = 0;
        for (int h = 0; h < 2; ++h) {
            const int grp = 2 * pair + h;
            if (grp >= a.G) break;
            const int64_t k0 = (int64_t)grp * g;
            const __half *src = a.W + row * a.k + k0 + lane * E;
            float w[8];
            bool finite = true;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                if (e < E) {
                    w[e] = __half2float(src[e]);
                    finite &= isfinite(w[e]);
                }
            }
            if (!finite) atomicOr(a.status, kStatusNonfinite);
            float lo = 0.0f, hi = 0.0f;  // range widened to contain 0
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                if (e < E) {
                    lo = fminf(lo, w[e]);
                    hi = fmaxf(hi, w[e]);
                }
            }
            lo = warp_min(lo);
            hi = warp_max(hi);
            const __half s16 = __float2half_rn(__fdiv_rn(__fsub_rn(hi, lo), qmax));
            const float s = __half2float(s16);
            float z = 0.0f;
            if (s != 0.0f) z = fminf(fmaxf(rintf(__fdiv_rn(-lo, s)), 0.0f), qmax);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                if (e < E) {
                    float q = 0.0f;
                    if (s != 0.0f) q = fminf(fmaxf(__fadd_rn(rintf(__fdiv_rn(w[e], s)), z), 0.0f), qmax);
                    sc[lane * E + e] = (uint8_t)q;
                }
            }
            __syncwarp();
            pack_group(sc, g, a.bits, k0, a.k, a.codes + row * (a.k * a.bits / 8), lane);
            __syncwarp();
            if (lane == 0) a.scales[row * a.G + grp] = s16;
            zbyte |= (uint32_t)z << (4 * h);
        }
        if (lane == 0) a.zeros[row * a.zbytes + pair] = (uint8_t)zbyte;
    }
}

// ------------------------------------------------------------- LUT quantize
// One warp per group.  Lloyd-Max on 2^b levels in float64 (exact int64 sums).
template <int L>
__global__ void __launch_bounds__(256) quantize_lut_kernel(QuantArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int warps = blockDim.x >> 5;
    const int g = a.g;
    const int E = g / kWarp;
    // per warp: g doubles of sorted values + g code bytes
    double *sorted = reinterpret_cast<double *>(smem_raw) + (size_t)warp * g;
    uint8_t *sc = smem_raw + (size_t)warps * g * sizeof(double) + (size_t)warp * g;
    const int64_t total = (int64_t)a.n * a.G;
    const double two_m24 = 5.9604644775390625e-08;  // 2^-24
    for (int64_t task = (int64_t)blockIdx.x * warps + warp; task < total;
         task += (int64_t)gridDim.x * warps) {
        const int64_t row = task / a.G;
        const int grp = (int)(task % a.G);
        const int64_t k0 = (int64_t)grp * g;
        const __half *src = a.W + row * a.k + k0 + lane * E;
        double w[8];
        long long wi[8];
        bool finite = true;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (e < E) {
                const float f = __half2float(src[e]);
                finite &= isfinite(f);
                w[e] = (double)f;
                wi[e] = (long long)(w[e] * 16777216.0);  // exact: fp16 = m * 2^-24
            }
        }
        if (!finite) atomicOr(a.status, kStatusNonfinite);
        // rank of every element: (# smaller) + (# equal with lower index)
        int rank[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) rank[e] = 0;
        for (int src_lane = 0; src_lane < kWarp; ++src_lane) {
#pragma unroll
            for (int f = 0; f < 8; ++f) {
                if (f < E) {
                    const double v = __shfl_sync(0xffffffffu, w[f], src_lane);
                    const int j = src_lane * E + f;
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        if (e < E) {
                            const int i = lane * E + e;
                            rank[e] += (v < w[e]) || (v == w[e] && j < i);
                        }
                    }
                }
            }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e)
            if (e < E) sorted[rank[e]] = w[e];
        __syncwarp();
        // number of distinct values
        int distinct_local = 0;
        for (int p = lane; p < g; p += kWarp) distinct_local += (p == 0) || (sorted[p] != sorted[p - 1]);
        const int distinct = warp_sum_i(distinct_local);
        double c[L];
        if (distinct <= L) {
            // the LUT is the distinct values, ascending, padded by the largest
            int cnt = 0;
            double last = sorted[0];
#pragma unroll
            for (int j = 0; j < L; ++j) c[j] = 0.0;
            for (int p = 0; p < g; ++p) {
                const double v = sorted[p];
                if (p == 0 || v != last) {
#pragma unroll
                    for (int j = 0; j < L; ++j)
                        if (j == cnt) c[j] = v;
                    ++cnt;
                    last = v;
                }
            }
#pragma unroll
            for (int j = 0; j < L; ++j)
                if (j >= cnt) c[j] = last;
        } else {
#pragma unroll
            for (int j = 0; j < L; ++j) c[j] = sorted[((2 * j + 1) * g) / (2 * L)];
            int prev[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) prev[e] = -1;
            for (int it = 0; it < a.lloyd_iters; ++it) {
                int asg[8];
                bool changed = false;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    if (e < E) {
                        int best = 0;
                        double bd = fabs(w[e] - c[0]);
#pragma unroll
                        for (int j = 1; j < L; ++j) {
                            const double d = fabs(w[e] - c[j]);
                            if (d < bd) {
                                bd = d;
                                best = j;
                            }
                        }
                        asg[e] = best;
                        changed |= (best != prev[e]);
                        prev[e] = best;
                    }
                }
                if (it > 0 && !__any_sync(0xffffffffu, changed)) break;
#pragma unroll
                for (int j = 0; j < L; ++j) {
                    long long s = 0;
                    int nj = 0;
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        if (e < E && asg[e] == j) {
                            s += wi[e];
                            ++nj;
                        }
                    }
                    s = warp_sum_ll(s);
                    nj = warp_sum_i(nj);
                    if (nj > 0) c[j] = __ddiv_rn((double)s * two_m24, (double)nj);
                }
            }
            // ascending sort of the levels (insertion sort, stable)
#pragma unroll
            for (int i = 1; i < L; ++i) {
#pragma unroll
                for (int j = i; j > 0; --j) {
                    if (c[j] < c[j - 1]) {
                        const double t = c[j];
                        c[j] = c[j - 1];
                        c[j - 1] = t;
                    }
                }
            }
        }
        uint16_t lut[L];
        double lutd[L];
#pragma unroll
        for (int j = 0; j < L; ++j) {
            lut[j] = f64_to_f16_bits(c[j]);
            lutd[j] = f16_bits_to_f64(lut[j]);
        }
        // final codes: nearest LUT entry, ties to the lowest index
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (e < E) {
                int best = 0;
                double bd = fabs(w[e] - lutd[0]);
#pragma unroll
                for (int j = 1; j < L; ++j) {
                    const double d = fabs(w[e] - lutd[j]);
                    if (d < bd) {
                        bd = d;
                        best = j;
                    }
                }
                sc[lane * E + e] = (uint8_t)best;
            }
        }
        __syncwarp();
        pack_group(sc, g, a.bits, k0, a.k, a.codes + row * (a.k * a.bits / 8), lane);
        if (lane < L / 2) {
            reinterpret_cast<uint32_t *>(a.luts + (row * a.G + grp) * L)[lane] =
                (uint32_t)lut[2 * lane] | ((uint32_t)lut[2 * lane + 1] << 16);
        }
        __syncwarp();
    }
}

// ------------------------------------------------------------------ dequant
// One thread per 32-code unit (a 16-byte chunk of 4-bit codes, or one triple of
// 3-bit words).  Uniform 4-bit goes through the magic-number unpack, 3-bit
// through the byte-permute table, so this kernel also checks, bit for bit,
// the unpack primitives the matmul kernels use.
__global__ void __launch_bounds__(256) dequant_kernel(DequantArgs a) {
    const int64_t units_per_row = a.k / 32;
    const int64_t total = a.n * units_per_row;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int64_t row = u / units_per_row;
        const int64_t j = u % units_per_row;
        const int64_t k0 = 32 * j;
        const int grp = (int)(k0 / a.g);
        __half2 v[16];
        if (a.bits == 4) {
            const uint4 c = *reinterpret_cast<const uint4 *>(a.codes + row * (a.k / 2) + 16 * j);
            const uint32_t z = zero_nibble(a.zeros + row * a.zbytes, grp);
            const __half s = a.scales[row * a.G + grp];
            const __half2 s2 = __halves2half2(s, s);
            const __half2 zl = zlo_of(z), zh = zhi_of(z);
            const uint32_t wds[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                __half2 o[4];
                unpack4_qz(wds[t], zl, zh, o);
#pragma unroll
                for (int p = 0; p < 4; ++p) v[4 * t + p] = __hmul2(o[p], s2);
            }
        } else {
            const uint8_t *rc = a.codes + row * (3 * a.k / 8);
            const int64_t s = k0 >> 7;
            const int i = (int)((k0 & 127) >> 5);
            const int64_t plane = a.k >> 3;
            const uint32_t A = *reinterpret_cast<const uint32_t *>(rc + 16 * s + 4 * i);
            const uint32_t B = *reinterpret_cast<const uint32_t *>(rc + plane + 16 * s + 4 * i);
            const uint32_t C = *reinterpret_cast<const uint32_t *>(rc + 2 * plane + 16 * s + 4 * i);
            Table8 t;
            if (a.kind == 1) {
                const uint4 l = *reinterpret_cast<const uint4 *>(a.luts + (row * a.G + grp) * 8);
                t = make_table8(l.x, l.y, l.z, l.w);
                lookup_triple(t, A, B, C, v);
            } else {
                const uint32_t z = zero_nibble(a.zeros + row * a.zbytes, grp);
                const __half sc = a.scales[row * a.G + grp];
                const __half2 s2 = __halves2half2(sc, sc);
                t = table8_offsets(z);
                lookup_triple(t, A, B, C, v);
#pragma unroll
                for (int p = 0; p < 16; ++p) v[p] = __hmul2(v[p], s2);
            }
        }
        uint4 *dst = reinterpret_cast<uint4 *>(a.W + row * a.k + k0);
#pragma unroll
        for (int q = 0; q < 4; ++q)
            dst[q] = make_uint4(h22u(v[4 * q]), h22u(v[4 * q + 1]), h22u(v[4 * q + 2]), h22u(v[4 * q + 3]));
    }
}

}  // namespace

cudaError_t launch_quantize(const QuantArgs &a, int num_sms, cudaStream_t st) {
    const int threads = 256, warps = threads / 32;
    if (a.kind == 0) {
        const int64_t tasks = a.n * ((a.G + 1) / 2);
        const int64_t blocks = std::min<int64_t>((tasks + warps - 1) / warps, (int64_t)num_sms * 16);
        const size_t smem = (size_t)warps * a.g;
        quantize_uniform_kernel<<<(unsigned)blocks, threads, smem, st>>>(a);
    } else {
        const int64_t tasks = a.n * a.G;
        const int64_t blocks = std::min<int64_t>((tasks + warps - 1) / warps, (int64_t)num_sms * 16);
        const size_t smem = (size_t)warps * a.g * (sizeof(double) + 1);
        quantize_lut_kernel<8><<<(unsigned)blocks, threads, smem, st>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_dequant(const DequantArgs &a, int num_sms, cudaStream_t st) {
    const int threads = 256;
    const int64_t units = a.n * (a.k / 32);
    const int64_t blocks = std::min<int64_t>((units + threads - 1) / threads, (int64_t)num_sms * 32);
    dequant_kernel<<<(unsigned)blocks, threads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace qx
