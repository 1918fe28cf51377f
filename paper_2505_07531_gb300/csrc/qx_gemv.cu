// Decode matmul y[b][n] = sum_k w_hat[n][k] x[b][k] on CUDA cores, fed by TMA.
//
// Decoding reads every weight once per token: it is bound by HBM bandwidth
// and by the cost of unpacking the codes (paper Section 2.4).  To keep HBM
// busy every SM needs tens of kilobytes of loads in flight from its first
// cycle, and the launch itself must be amortised over as many bytes as
// possible, so the kernel is built around the Blackwell bulk-copy engine and
// serves several matrices in one launch:
//
//   * one persistent CTA per SM owns a byte-balanced slice of the rows of all
//     matrices of the call, taken in order (a slice may span matrices);
//   * a producer warp streams whole rows of packed codes (and LUTs) into a
//     ring of up to 8 shared-memory stages with cp.async.bulk, completing on
//     mbarriers; the small uniform scales and zero-points are copied by its
//     lanes.  Weight copies are issued before the programmatic-dependent-launch
//     wait, so they overlap the tail of the previous kernel;
//   * sixteen consumer warps decode 32-weight units out of shared memory with
//     the magic-number / byte-permute primitives and multiply them with x,
//     which is staged once per CTA in a padded (bank-conflict-free) layout and
//     reused across a group of rows held in registers;
//   * per 32-weight unit the products form two half2 FMA chains of 8, promoted
//     to fp32; a warp-shuffle reduction per row group feeds fp32 shared-memory
//     row accumulators, and the producer writes finished rows to y.
// The uniform scale is folded out of the inner loop (a unit contributes
// s * sum (q - z) x); the LUT family contributes sum LUT[q] x.  Every wait is
// bounded in time and reports QX_ERR_TIMEOUT through the device status word.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kConsumerWarps = 16;
constexpr int kThreads = 32 * (1 + kConsumerWarps);
constexpr int kMaxStages = 8;
constexpr int kMaxRB = 16;
constexpr int kSmemBudget = 210 * 1024;
constexpr int kStageTarget = 24 * 1024;
constexpr int kHeader = 1024;  // barriers, flags, stage descriptors
constexpr int kAccBytes = kMaxStages * kMaxRB * 4 * 4;

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(b)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: false after `limit_ns`, or once another warp has raised the
// abort flag (when `abort_flag` is not null).
__device__ __noinline__ bool mbar_wait(uint64_t *b, uint32_t parity, uint64_t limit_ns,
                                       volatile uint32_t *abort_flag) {
    if (mbar_try_wait(b, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(b, parity)) return true;
        if ((i & 15u) == 0) {
            if (abort_flag != nullptr && *abort_flag) return false;
            if (globaltimer_ns() - t0 > limit_ns) return false;
            __nanosleep(64);
        }
    }
}

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void consumer_bar() {
    asm volatile("bar.sync 1, %0;" ::"n"(32 * kConsumerWarps) : "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float dot16(const __half2 (&w)[16], const __half2 (&x)[16]) {
    __half2 a0 = __hmul2(w[0], x[0]);
    __half2 a1 = __hmul2(w[1], x[1]);
#pragma unroll
    for (int i = 2; i < 16; i += 2) {
        a0 = __hfma2(w[i], x[i], a0);
        a1 = __hfma2(w[i + 1], x[i + 1], a1);
    }
    const float2 f0 = __half22float2(a0);
    const float2 f1 = __half22float2(a1);
    return (f0.x + f0.y) + (f1.x + f1.y);
}

// x is kept in shared memory with every 32-value unit padded to 80 bytes, so
// that lanes reading consecutive units hit distinct banks.
__device__ __forceinline__ int64_t xpad(int64_t k) { return (k >> 5) * 40 + (k & 31); }

__device__ __forceinline__ void load_x16(const __half *unit, __half2 (&x)[16]) {
    const uint4 *v = reinterpret_cast<const uint4 *>(unit);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint4 t = v[q];
        x[4 * q + 0] = u2h2(t.x);
        x[4 * q + 1] = u2h2(t.y);
        x[4 * q + 2] = u2h2(t.z);
        x[4 * q + 3] = u2h2(t.w);
    }
}

struct StageDesc {
    int mat;
    int rb;
    int64_t row0;
};

// Rows [first, end) of matrix `m` owned by this CTA: those whose starting byte
// (in the concatenation of all matrices' rows) falls in the CTA's byte range.
__device__ __forceinline__ void cta_rows(const GemvMulti &a, int m, int64_t &first, int64_t &end) {
    const int64_t lo = (int64_t)blockIdx.x * a.total_bytes / gridDim.x;
    const int64_t hi = (int64_t)(blockIdx.x + 1) * a.total_bytes / gridDim.x;
    const int64_t off = a.mat[m].byte_off, rb = a.mat[m].row_bytes, n = a.mat[m].n;
    const int64_t f = lo <= off ? 0 : (lo - off + rb - 1) / rb;
    const int64_t e = hi <= off ? 0 : (hi - off + rb - 1) / rb;
    first = f < n ? f : n;
    end = e < n ? e : n;
}

template <int BITS, int KIND, int BMAX, int RSUB>
__global__ void __launch_bounds__(kThreads, 1) gemv_kernel(const __grid_constant__ GemvMulti a) {
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    uint64_t *empty = full + kMaxStages;
    volatile uint32_t *abort_flag = reinterpret_cast<volatile uint32_t *>(empty + kMaxStages);
    StageDesc *desc = reinterpret_cast<StageDesc *>(smem + 256);
    float *acc = reinterpret_cast<float *>(smem + kHeader);
    __half *xs = reinterpret_cast<__half *>(smem + kHeader + kAccBytes);
    uint8_t *stages = smem + kHeader + kAccBytes + a.x_smem_bytes;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int nb = a.batch;

    if (threadIdx.x == 0) {
        for (int i = 0; i < a.stages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], kConsumerWarps);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    for (int i = threadIdx.x; i < kMaxStages * kMaxRB * BMAX; i += blockDim.x) acc[i] = 0.0f;
    __syncthreads();
    // let the next kernel in the stream begin its own weight prefetch early;
    // it still waits for this grid's completion before touching activations
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        int sq = 0;
        bool ok = true;
        bool waited_dep = false;
        for (int m = 0; m < a.count && ok; ++m) {
            int64_t first, end;
            cta_rows(a, m, first, end);
            const GemvMat &M = a.mat[m];
            for (int64_t r0 = first; r0 < end && ok; r0 += M.RB, ++sq) {
                const int st = sq % a.stages;
                const uint32_t ph = (uint32_t)(sq / a.stages) & 1u;
                bool got = true;
                if (lane == 0) got = mbar_wait(&empty[st], ph ^ 1u, a.wait_limit_ns, abort_flag);
                if (!__shfl_sync(0xffffffffu, got, 0)) {
                    ok = false;
                    break;
                }
                if (sq >= a.stages) {  // retire the rows that last used this stage
                    if (!waited_dep) {
                        asm volatile("griddepcontrol.wait;" ::: "memory");
                        waited_dep = true;
                    }
                    const StageDesc d = desc[st];
                    __syncwarp();  // every lane holds d before lane 0 overwrites desc[st] below
                    const GemvMat &P = a.mat[d.mat];
                    float *pacc = acc + st * kMaxRB * BMAX;
                    for (int i = lane; i < d.rb * nb; i += 32) {
                        const int r = i / nb, b = i % nb;
                        const float v = pacc[r * BMAX + b];
                        pacc[r * BMAX + b] = 0.0f;
                        if (a.y_f32)
                            reinterpret_cast<float *>(P.y)[(int64_t)b * P.n + d.row0 + r] = v;
                        else
                            reinterpret_cast<__half *>(P.y)[(int64_t)b * P.n + d.row0 + r] = __float2half_rn(v);
                    }
                }
                const int rb = (int)((end - r0) < M.RB ? (end - r0) : M.RB);
                uint8_t *sbase = stages + (size_t)st * a.stage_bytes;
                if (KIND == 0) {  // scales and zero-points: lane copies (rows not 16-byte aligned)
                    __half *ss = reinterpret_cast<__half *>(sbase + M.RB * M.CB);
                    uint8_t *sz = sbase + M.RB * M.CB + M.RB * M.SB;
                    const __half *gs = M.scales + r0 * M.G;
                    const uint8_t *gz = M.zeros + r0 * M.zbytes;
                    for (int i = lane; i < rb * M.G; i += 32) ss[i] = gs[i];
                    for (int i = lane; i < rb * M.zbytes; i += 32) sz[i] = gz[i];
                }
                if (lane == 0) {
                    desc[st].mat = m;
                    desc[st].rb = rb;
                    desc[st].row0 = r0;
                }
                __syncwarp();
                if (lane == 0) {
                    const uint32_t cbytes = (uint32_t)(rb * M.CB);
                    const uint32_t lbytes = (uint32_t)(rb * M.LB);
                    mbar_arrive_expect_tx(&full[st], cbytes + lbytes);
                    bulk_g2s(sbase, M.codes + r0 * M.CB, cbytes, &full[st]);
                    if (KIND == 1) bulk_g2s(sbase + M.RB * M.CB, M.luts + r0 * M.G * 8, lbytes, &full[st]);
                }
            }
        }
        if (!waited_dep) asm volatile("griddepcontrol.wait;" ::: "memory");
        // retire the last stages (after an abort: let in-flight copies land)
        for (int q = (sq - a.stages > 0 ? sq - a.stages : 0); q < sq; ++q) {
            const int st = q % a.stages;
            const uint32_t ph = (uint32_t)(q / a.stages) & 1u;
            bool got = ok;
            if (lane == 0 && ok) got = mbar_wait(&empty[st], ph, a.wait_limit_ns, abort_flag);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (!got) {
                ok = false;
                if (lane == 0) mbar_wait(&full[st], ph, a.wait_limit_ns, nullptr);
                __syncwarp();
                continue;
            }
            const StageDesc d = desc[st];
            __syncwarp();
            const GemvMat &P = a.mat[d.mat];
            const float *pacc = acc + st * kMaxRB * BMAX;
            for (int i = lane; i < d.rb * nb; i += 32) {
                const int r = i / nb, b = i % nb;
                const float v = pacc[r * BMAX + b];
                if (a.y_f32)
                    reinterpret_cast<float *>(P.y)[(int64_t)b * P.n + d.row0 + r] = v;
                else
                    reinterpret_cast<__half *>(P.y)[(int64_t)b * P.n + d.row0 + r] = __float2half_rn(v);
            }
        }
        if (!ok && lane == 0) {
            *abort_flag = 1u;
            atomicOr(a.status, kStatusTimeout);
        }
    } else {
        // ------------------------------------------------------------ consumers
        const int cw = warp - 1;
        const int ct = threadIdx.x - 32;
        asm volatile("griddepcontrol.wait;" ::: "memory");
        {   // stage the x of every matrix this CTA touches, padded
            int64_t xoff = 0;
            for (int m = 0; m < a.count; ++m) {
                int64_t first, end;
                cta_rows(a, m, first, end);
                if (first >= end) continue;
                const GemvMat &M = a.mat[m];
                const int64_t vecs = (int64_t)nb * M.k / 8;
                for (int64_t i = ct; i < vecs; i += 32 * kConsumerWarps) {
                    const int64_t e = 8 * i, b = e / M.k, kk = e % M.k;
                    *reinterpret_cast<uint4 *>(xs + xoff + b * (M.k / 32) * 40 + xpad(kk)) =
                        *reinterpret_cast<const uint4 *>(M.x + e);
                }
                xoff += (int64_t)nb * (M.k / 32) * 40;
            }
        }
        consumer_bar();
        bool ok = true;
        int sq = 0;
        int64_t xoff = 0;
        for (int m = 0; m < a.count && ok; ++m) {
            int64_t first, end;
            cta_rows(a, m, first, end);
            if (first >= end) continue;
            const GemvMat &M = a.mat[m];
            const int64_t K = M.k;
            const int64_t U = K / 32;  // 32-weight units per row
            const int chunks_per_sg = (int)((U + 31) / 32);
            const __half *xm = xs + xoff;
            const int64_t xstride = (K / 32) * 40;
            for (int64_t r0 = first; r0 < end; r0 += M.RB, ++sq) {
                const int st = sq % a.stages;
                const uint32_t ph = (uint32_t)(sq / a.stages) & 1u;
                ok = mbar_wait(&full[st], ph, a.wait_limit_ns, abort_flag);
                if (!__all_sync(0xffffffffu, ok)) {
                    ok = false;
                    break;
                }
                const int rb = (int)((end - r0) < M.RB ? (end - r0) : M.RB);
                const uint8_t *sbase = stages + (size_t)st * a.stage_bytes;
                float *sacc = acc + st * kMaxRB * BMAX;
                const int nsg = (rb + RSUB - 1) / RSUB;
                const int nchunks = nsg * chunks_per_sg;
                const int rot = (int)(((int64_t)sq * nchunks) % kConsumerWarps);
                for (int c = (cw - rot + kConsumerWarps) % kConsumerWarps; c < nchunks; c += kConsumerWarps) {
                    const int sg = c / chunks_per_sg;
                    const int64_t u = (int64_t)(c % chunks_per_sg) * 32 + lane;
                    float p[RSUB][BMAX];
#pragma unroll
                    for (int r = 0; r < RSUB; ++r)
#pragma unroll
                        for (int b = 0; b < BMAX; ++b) p[r][b] = 0.0f;
                    if (u < U) {
                        const int grp = (int)((32 * u) >> M.log2g);
                        __half2 xv[BMAX][16];
#pragma unroll
                        for (int b = 0; b < BMAX; ++b)
                            if (b < nb) load_x16(xm + b * xstride + 40 * u, xv[b]);
#pragma unroll
                        for (int r = 0; r < RSUB; ++r) {
                            const int rl = sg * RSUB + r;
                            if (rl >= rb) break;
                            const uint8_t *rc = sbase + rl * M.CB;
                            __half2 w[16];
                            float s = 1.0f;
                            if (BITS == 4) {
                                const uint4 cw4 = *reinterpret_cast<const uint4 *>(rc + 16 * u);
                                const __half *ss = reinterpret_cast<const __half *>(sbase + M.RB * M.CB);
                                const uint8_t *sz = sbase + M.RB * M.CB + M.RB * M.SB;
                                s = __half2float(ss[rl * M.G + grp]);
                                const uint32_t z = (sz[rl * M.zbytes + (grp >> 1)] >> ((grp & 1) * 4)) & 15u;
                                const __half2 zl = zlo_of(z), zh = zhi_of(z);
                                const uint32_t wd[4] = {cw4.x, cw4.y, cw4.z, cw4.w};
#pragma unroll
                                for (int t = 0; t < 4; ++t) {
                                    __half2 o[4];
                                    unpack4_qz(wd[t], zl, zh, o);
#pragma unroll
                                    for (int q = 0; q < 4; ++q) w[4 * t + q] = o[q];
                                }
                            } else {
                                const int64_t off = 4 * u;  // word u of each plane
                                const uint32_t A = *reinterpret_cast<const uint32_t *>(rc + off);
                                const uint32_t B = *reinterpret_cast<const uint32_t *>(rc + (K >> 3) + off);
                                const uint32_t C = *reinterpret_cast<const uint32_t *>(rc + 2 * (K >> 3) + off);
                                Table8 tab;
                                if (KIND == 1) {
                                    const uint4 l = *reinterpret_cast<const uint4 *>(sbase + M.RB * M.CB +
                                                                                      (rl * M.G + grp) * 16);
                                    tab = make_table8(l.x, l.y, l.z, l.w);
                                } else {
                                    const __half *ss = reinterpret_cast<const __half *>(sbase + M.RB * M.CB);
                                    const uint8_t *sz = sbase + M.RB * M.CB + M.RB * M.SB;
                                    s = __half2float(ss[rl * M.G + grp]);
                                    tab = table8_offsets((sz[rl * M.zbytes + (grp >> 1)] >> ((grp & 1) * 4)) & 15u);
                                }
                                lookup_triple(tab, A, B, C, w);
                            }
#pragma unroll
                            for (int b = 0; b < BMAX; ++b)
                                if (b < nb) p[r][b] = s * dot16(w, xv[b]);
                        }
                    }
#pragma unroll
                    for (int r = 0; r < RSUB; ++r) {
#pragma unroll
                        for (int b = 0; b < BMAX; ++b) {
                            const float v = warp_sum(p[r][b]);
                            const int rl = sg * RSUB + r;
                            if (lane == 0 && rl < rb && b < nb) atomicAdd(&sacc[rl * BMAX + b], v);
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[st]);
            }
            xoff += (int64_t)nb * xstride;
        }
        if (!ok && lane == 0) {
            *abort_flag = 1u;
            atomicOr(a.status, kStatusTimeout);
        }
    }
    __syncthreads();
}

template <int BITS, int KIND, int BMAX, int RSUB>
cudaError_t launch_one(const GemvMulti &a, cudaStream_t st, bool pdl) {
    auto kern = gemv_kernel<BITS, KIND, BMAX, RSUB>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, a.smem_bytes);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)a.grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = (size_t)a.smem_bytes;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

}  // namespace

// Host-side plan: per-matrix stage geometry, the byte-balanced CTA slices and
// the shared-memory budget (x of every matrix a CTA touches + the ring).
// Returns false if the matrices cannot share one launch.
bool plan_gemv(GemvMulti &a, int num_sms) {
    int max_stage = 0;
    int64_t total = 0;
    for (int m = 0; m < a.count; ++m) {
        GemvMat &M = a.mat[m];
        M.CB = (int)(M.k * a.bits / 8);
        M.LB = a.kind == 1 ? M.G * 16 : 0;
        M.SB = a.kind == 0 ? ((M.G * 2 + 15) / 16) * 16 : 0;
        M.ZB = a.kind == 0 ? ((M.zbytes + 15) / 16) * 16 : 0;
        M.row_bytes = M.CB + M.LB + M.SB + M.ZB;
        M.RB = std::max(1, std::min(kMaxRB, kStageTarget / M.row_bytes));
        M.byte_off = total;
        total += M.n * M.row_bytes;
        max_stage = std::max(max_stage, M.RB * M.row_bytes);
    }
    a.total_bytes = total;
    int64_t rows = 0;
    for (int m = 0; m < a.count; ++m) rows += a.mat[m].n;
    a.grid = (int)std::min<int64_t>(num_sms, rows);
    // x bytes per CTA: simulate the slices
    int64_t xmax = 0;
    for (int c = 0; c < a.grid; ++c) {
        const int64_t lo = (int64_t)c * total / a.grid, hi = (int64_t)(c + 1) * total / a.grid;
        int64_t xb = 0;
        for (int m = 0; m < a.count; ++m) {
            const GemvMat &M = a.mat[m];
            const int64_t f = lo <= M.byte_off ? 0 : (lo - M.byte_off + M.row_bytes - 1) / M.row_bytes;
            const int64_t e = hi <= M.byte_off ? 0 : (hi - M.byte_off + M.row_bytes - 1) / M.row_bytes;
            if (std::min(f, M.n) < std::min(e, M.n)) xb += (int64_t)a.batch * (M.k / 32) * 80;
        }
        xmax = std::max(xmax, xb);
    }
    a.x_smem_bytes = (int)((xmax + 127) / 128 * 128);
    a.stage_bytes = (max_stage + 127) / 128 * 128;
    const int fixed = kHeader + kAccBytes + a.x_smem_bytes;
    a.stages = std::min(kMaxStages, (kSmemBudget - fixed) / a.stage_bytes);
    a.smem_bytes = fixed + a.stages * a.stage_bytes;
    return a.stages >= 2;
}

cudaError_t launch_gemv_multi(const GemvMulti &a, cudaStream_t st, bool pdl) {
    if (a.bits == 4) {
        if (a.batch <= 1) return launch_one<4, 0, 1, 4>(a, st, pdl);
        if (a.batch <= 2) return launch_one<4, 0, 2, 2>(a, st, pdl);
        return launch_one<4, 0, 4, 1>(a, st, pdl);
    }
    if (a.kind == 1) {
        if (a.batch <= 1) return launch_one<3, 1, 1, 4>(a, st, pdl);
        if (a.batch <= 2) return launch_one<3, 1, 2, 2>(a, st, pdl);
        return launch_one<3, 1, 4, 1>(a, st, pdl);
    }
    if (a.batch <= 1) return launch_one<3, 0, 1, 4>(a, st, pdl);
    if (a.batch <= 2) return launch_one<3, 0, 2, 2>(a, st, pdl);
    return launch_one<3, 0, 4, 1>(a, st, pdl);
}

}  // namespace qx
