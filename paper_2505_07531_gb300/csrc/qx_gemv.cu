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

constexpr int kMaxStages = 8;
constexpr int kMaxRB = 16;
constexpr int kSmemBudget = 210 * 1024;
constexpr int kStageTarget = 24 * 1024;
constexpr int kHeader = 2048;  // barriers, flags, stage descriptors, matrix table
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

// try_wait with a suspend-time hint: a thread whose phase is not complete
// sleeps in hardware (up to the hint) instead of spinning on issue slots.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(b)), "r"(parity), "r"(100000u)
        : "memory");
    return ok != 0;
}

// Bounded wait: false after `limit_ns`, or once another warp has raised the
// abort flag (when `abort_flag` is not null).
__device__ __noinline__ bool mbar_wait(uint64_t *b, uint32_t parity, uint64_t limit_ns,
                                       volatile uint32_t *abort_flag) {
    if (mbar_try_wait(b, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        if (mbar_try_wait_sleep(b, parity)) return true;
        if (abort_flag != nullptr && *abort_flag) return false;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

// Shared-memory loads with 32-bit shared-window addresses.  The ring's
// contents change between barrier phases, so these are volatile: they are
// neither merged nor moved across the (volatile) barrier waits.
__device__ __forceinline__ uint32_t lds32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds8(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u8 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds16(uint32_t a) {
    uint16_t v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}

template <int CW>
__device__ __forceinline__ void consumer_bar() {
    asm volatile("bar.sync 1, %0;" ::"n"(32 * CW) : "memory");
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

__device__ __forceinline__ void load_x16(uint32_t unit, __half2 (&x)[16]) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint4 t = lds128(unit + 16 * q);
        x[4 * q + 0] = u2h2(t.x);
        x[4 * q + 1] = u2h2(t.y);
        x[4 * q + 2] = u2h2(t.z);
        x[4 * q + 3] = u2h2(t.w);
    }
}

// Per-matrix fields and this CTA's row range, copied once from the (large)
// parameter block into shared memory: the loops then never index the
// parameter space with a runtime matrix number.
struct MatS {
    const uint8_t *codes;
    const __half *scales;
    const uint8_t *zeros;
    const __half *luts;
    const __half *x;
    void *y;
    int64_t n, first, end;
    int k, CB, LB, SB, RB, G, zbytes, log2g;
};

struct StageDesc {
    int mat;
    int rb;
    int64_t row0;
};

// Rows [first, end) of matrix `m` owned by this CTA (slices precomputed on
// the host, so the kernel does no 64-bit division).
__device__ __forceinline__ void cta_rows(const GemvMulti &a, int m, int64_t &first, int64_t &end) {
    const int64_t lo = a.cta_row[blockIdx.x], hi = a.cta_row[blockIdx.x + 1];
    const int64_t o = a.row_off[m], n = a.mat[m].n;
    const int64_t f = lo - o, e = hi - o;
    first = f < 0 ? 0 : (f > n ? n : f);
    end = e < 0 ? 0 : (e > n ? n : e);
}

// 12 consumer warps + 1 producer: registers are reserved per four warps, so
// 13 warps cost 16 warp slots and leave 128 registers per thread.
constexpr int kConsumerWarps = 12;
constexpr int kGroupWarps = 4;  // consumer warps that share one stage
constexpr int kThreads = 32 * (1 + kConsumerWarps);

template <int BITS, int KIND, int BMAX>
__global__ void __launch_bounds__(kThreads, 1) gemv_kernel(const __grid_constant__ GemvMulti a) {
    constexpr int NG = kConsumerWarps / kGroupWarps;  // consumer groups
    constexpr int RMAX = 8 / BMAX;                    // rows accumulated per pass
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    uint64_t *empty = full + kMaxStages;
    volatile uint32_t *abort_flag = reinterpret_cast<volatile uint32_t *>(empty + kMaxStages);
    StageDesc *desc = reinterpret_cast<StageDesc *>(smem + 256);
    MatS *mats = reinterpret_cast<MatS *>(smem + 512);
    float *acc = reinterpret_cast<float *>(smem + kHeader);
    __half *xs = reinterpret_cast<__half *>(smem + kHeader + kAccBytes);
    uint8_t *stages = smem + kHeader + kAccBytes + a.x_smem_bytes;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int nb = a.batch;
    const int count = a.count, nring = a.stages, stage_bytes = a.stage_bytes;

    if (threadIdx.x == 0) {
        for (int i = 0; i < nring; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], kGroupWarps);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x < count) {  // per-matrix fields -> shared memory, once
        const int m = threadIdx.x;
        const GemvMat &M = a.mat[m];
        MatS &S = mats[m];
        S.codes = M.codes;
        S.scales = M.scales;
        S.zeros = M.zeros;
        S.luts = M.luts;
        S.x = M.x;
        S.y = M.y;
        S.n = M.n;
        cta_rows(a, m, S.first, S.end);
        S.k = (int)M.k;
        S.CB = M.CB;
        S.LB = M.LB;
        S.SB = M.SB;
        S.RB = M.RB;
        S.G = M.G;
        S.zbytes = M.zbytes;
        S.log2g = M.log2g;
    }
    for (int i = threadIdx.x; i < kMaxStages * kMaxRB * BMAX; i += blockDim.x) acc[i] = 0.0f;
    __syncthreads();
    // let the next kernel in the stream begin its own weight prefetch early;
    // it still waits for this grid's completion before touching activations
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        int sq = 0, st = 0;
        uint32_t ph = 0;
        bool ok = true;
        bool waited_dep = false;
        for (int m = 0; m < count && ok; ++m) {
            const MatS &M = mats[m];
            const int64_t first = M.first, end = M.end;
            const int RB = M.RB, CB = M.CB, LB = M.LB, G = M.G;
            const uint8_t *codes = M.codes;
            const __half *luts = M.luts;
            for (int64_t r0 = first; r0 < end && ok; r0 += RB) {
                bool got = true;
                if (lane == 0 && sq >= nring) got = mbar_wait(&empty[st], ph ^ 1u, a.wait_limit_ns, abort_flag);
                if (!__shfl_sync(0xffffffffu, got, 0)) {
                    ok = false;
                    break;
                }
                if (sq >= nring) {  // retire the rows that last used this stage
                    if (!waited_dep) {
                        asm volatile("griddepcontrol.wait;" ::: "memory");
                        waited_dep = true;
                    }
                    const StageDesc d = desc[st];
                    __syncwarp();  // every lane holds d before lane 0 overwrites desc[st] below
                    const MatS &P = mats[d.mat];
                    float *pacc = acc + st * kMaxRB * BMAX;
                    for (int i = lane; i < d.rb * nb; i += 32) {
                        const int r = i / nb, b = i - r * nb;
                        const float v = pacc[r * BMAX + b];
                        pacc[r * BMAX + b] = 0.0f;
                        if (a.y_f32)
                            reinterpret_cast<float *>(P.y)[(int64_t)b * P.n + d.row0 + r] = v;
                        else
                            reinterpret_cast<__half *>(P.y)[(int64_t)b * P.n + d.row0 + r] = __float2half_rn(v);
                    }
                }
                const int rb = (int)((end - r0) < RB ? (end - r0) : RB);
                uint8_t *sbase = stages + st * stage_bytes;
                if (KIND == 0) {  // scales and zero-points: lane copies (rows not 16-byte aligned)
                    __half *ss = reinterpret_cast<__half *>(sbase + RB * CB);
                    uint8_t *sz = sbase + RB * CB + RB * M.SB;
                    const __half *gs = M.scales + r0 * G;
                    const uint8_t *gz = M.zeros + r0 * M.zbytes;
                    for (int i = lane; i < rb * G; i += 32) ss[i] = gs[i];
                    for (int i = lane; i < rb * M.zbytes; i += 32) sz[i] = gz[i];
                }
                if (lane == 0) {
                    desc[st].mat = m;
                    desc[st].rb = rb;
                    desc[st].row0 = r0;
                }
                __syncwarp();
                if (lane == 0) {
                    const uint32_t cbytes = (uint32_t)(rb * CB);
                    const uint32_t lbytes = (uint32_t)(rb * LB);
                    mbar_arrive_expect_tx(&full[st], cbytes + lbytes);
                    bulk_g2s(sbase, codes + r0 * CB, cbytes, &full[st]);
                    if (KIND == 1) bulk_g2s(sbase + RB * CB, luts + r0 * G * 8, lbytes, &full[st]);
                }
                ++sq;
                if (++st == nring) {
                    st = 0;
                    ph ^= 1u;
                }
            }
        }
        if (!waited_dep) asm volatile("griddepcontrol.wait;" ::: "memory");
        // retire the last stages (after an abort: let in-flight copies land)
        for (int q = (sq - nring > 0 ? sq - nring : 0); q < sq; ++q) {
            const int qs = q % nring;
            const uint32_t qp = (uint32_t)(q / nring) & 1u;
            bool got = ok;
            if (lane == 0 && ok) got = mbar_wait(&empty[qs], qp, a.wait_limit_ns, abort_flag);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (!got) {
                ok = false;
                if (lane == 0) mbar_wait(&full[qs], qp, a.wait_limit_ns, nullptr);
                __syncwarp();
                continue;
            }
            const StageDesc d = desc[qs];
            __syncwarp();
            const MatS &P = mats[d.mat];
            const float *pacc = acc + qs * kMaxRB * BMAX;
            for (int i = lane; i < d.rb * nb; i += 32) {
                const int r = i / nb, b = i - r * nb;
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
        const int grp_id = cw / kGroupWarps;  // stages sq with sq % NG == grp_id
        const int j = cw % kGroupWarps;       // warp within the group
        const int ct = threadIdx.x - 32;
        asm volatile("griddepcontrol.wait;" ::: "memory");
        {   // stage the x of every matrix this CTA touches, padded
            int xoff = 0;
            for (int m = 0; m < count; ++m) {
                const MatS &M = mats[m];
                if (M.first >= M.end) continue;
                const int K = M.k;
                const int vecs = nb * K / 8;
                const __half *xg = M.x;
                for (int i = ct; i < vecs; i += 32 * kConsumerWarps) {
                    const int e = 8 * i, b = e / K, kk = e - b * K;
                    *reinterpret_cast<uint4 *>(xs + xoff + b * (K / 32) * 40 + xpad(kk)) =
                        *reinterpret_cast<const uint4 *>(xg + e);
                }
                xoff += nb * (K / 32) * 40;
            }
        }
        consumer_bar<kConsumerWarps>();
        bool ok = true;
        int sq = 0, st = 0;
        uint32_t ph = 0;
        uint32_t xm = smem_u32(xs);  // shared address of this matrix's padded x
        const uint32_t stages_s = smem_u32(stages);
        for (int m = 0; m < count && ok; ++m) {
            const MatS &M = mats[m];
            const int64_t first = M.first, end = M.end;
            if (first >= end) continue;
            // per-matrix constants in 32-bit registers (k <= 32768, a stage < 64 KB)
            const int K = M.k;
            const int CB = M.CB, RB = M.RB, G = M.G;
            const int SBb = M.SB, ZBb = M.zbytes, log2g = M.log2g;
            const int U = K >> 5;      // 32-weight units per row
            const int plane = K >> 3;  // bytes per 3-bit plane
            const int nuc = (U + 31) >> 5;  // unit-chunks (32 units, one per lane) per row
            const uint32_t xstride = (uint32_t)U * 80u;  // bytes per batch row of padded x
            // split of a stage among the group's warps: unit-chunks when there
            // are enough of them, otherwise unit-chunks x interleaved rows
            int uc0, ucstep, rfirst, rmask;
            bool idle = false;
            if (nuc >= kGroupWarps) {
                uc0 = j;
                ucstep = kGroupWarps;
                rfirst = 0;
                rmask = 0;
            } else {
                const int rsplit = nuc == 1 ? 4 : (nuc == 2 ? 2 : 1);
                uc0 = j % nuc;
                ucstep = nuc;
                rfirst = j / nuc;
                rmask = rsplit - 1;
                idle = j >= nuc * rsplit;
            }
            for (int64_t r0 = first; r0 < end && ok; r0 += RB) {
                const int mysq = sq;
                const int myst = st;
                const uint32_t myph = ph;
                ++sq;
                if (++st == nring) {
                    st = 0;
                    ph ^= 1u;
                }
                if (mysq % NG != grp_id) continue;  // another group's stage
                ok = mbar_wait(&full[myst], myph, a.wait_limit_ns, abort_flag);
                if (!__all_sync(0xffffffffu, ok)) {
                    ok = false;
                    break;
                }
                const int rb = (int)((end - r0) < RB ? (end - r0) : RB);
                const uint32_t sb = stages_s + (uint32_t)(myst * stage_bytes);
                const uint32_t meta = sb + (uint32_t)(RB * CB);
                float *sacc = acc + myst * (kMaxRB * BMAX);
                if (!idle) {
                    for (int rp = 0; rp < rb; rp += RMAX) {
                        float p[RMAX][BMAX];
#pragma unroll
                        for (int r = 0; r < RMAX; ++r)
#pragma unroll
                            for (int b = 0; b < BMAX; ++b) p[r][b] = 0.0f;
                        for (int uc = uc0; uc < nuc; uc += ucstep) {
                            const int u = uc * 32 + lane;
                            if (u >= U) continue;
                            const int grp = (32 * u) >> log2g;
                            __half2 xv[BMAX][16];
#pragma unroll
                            for (int b = 0; b < BMAX; ++b)
                                if (b < nb) load_x16(xm + (uint32_t)b * xstride + 80u * (uint32_t)u, xv[b]);
#pragma unroll
                            for (int ri = 0; ri < RMAX; ++ri) {
                                const int rl = rp + ri;
                                if (rl < rb && (rl & rmask) == rfirst) {
                                    const uint32_t rc = sb + (uint32_t)(rl * CB);
                                    __half2 w[16];
                                    float s = 1.0f;
                                    if (BITS == 4) {
                                        const uint4 cw4 = lds128(rc + 16u * (uint32_t)u);
                                        s = __half2float(__ushort_as_half((unsigned short)lds16(meta + 2u * (uint32_t)(rl * G + grp))));
                                        const uint32_t z = (lds8(meta + (uint32_t)(RB * SBb + rl * ZBb + (grp >> 1))) >> ((grp & 1) * 4)) & 15u;
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
                                        const uint32_t cp = rc + 4u * (uint32_t)u;  // word u of each plane
                                        const uint32_t A = lds32(cp);
                                        const uint32_t B = lds32(cp + (uint32_t)plane);
                                        const uint32_t C = lds32(cp + 2u * (uint32_t)plane);
                                        Table8 tab;
                                        if (KIND == 1) {
                                            const uint4 l = lds128(meta + 16u * (uint32_t)(rl * G + grp));
                                            tab = make_table8(l.x, l.y, l.z, l.w);
                                        } else {
                                            s = __half2float(__ushort_as_half((unsigned short)lds16(meta + 2u * (uint32_t)(rl * G + grp))));
                                            tab = table8_offsets((lds8(meta + (uint32_t)(RB * SBb + rl * ZBb + (grp >> 1))) >> ((grp & 1) * 4)) & 15u);
                                        }
                                        lookup_triple(tab, A, B, C, w);
                                    }
#pragma unroll
                                    for (int b = 0; b < BMAX; ++b)
                                        if (b < nb) p[ri][b] += s * dot16(w, xv[b]);
                                }
                            }
                        }
#pragma unroll
                        for (int ri = 0; ri < RMAX; ++ri) {
                            const int rl = rp + ri;
                            if (rl < rb && (rl & rmask) == rfirst) {
#pragma unroll
                                for (int b = 0; b < BMAX; ++b) {
                                    if (b < nb) {
                                        const float v = warp_sum(p[ri][b]);
                                        if (lane == 0) atomicAdd(&sacc[rl * BMAX + b], v);
                                    }
                                }
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[myst]);
            }
            xm += (uint32_t)nb * xstride;
        }
        if (!ok && lane == 0) {
            *abort_flag = 1u;
            atomicOr(a.status, kStatusTimeout);
        }
    }
    __syncthreads();
}

template <int BITS, int KIND, int BMAX>
cudaError_t launch_one(const GemvMulti &a, cudaStream_t st, bool pdl) {
    auto kern = gemv_kernel<BITS, KIND, BMAX>;
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
    for (int m = 0; m < a.count; ++m) {
        a.row_off[m] = rows;
        rows += a.mat[m].n;
    }
    a.row_off[a.count] = rows;
    a.grid = (int)std::min<int64_t>(std::min(num_sms, kMaxGemvCtas), rows);
    // CTA c owns the rows whose first byte lies in [c * total / grid, (c+1) * total / grid)
    for (int c = 0; c <= a.grid; ++c) {
        const int64_t b = (int64_t)((__int128)c * total / a.grid);
        int64_t r = rows;
        for (int m = 0; m < a.count; ++m) {
            const GemvMat &M = a.mat[m];
            if (b < M.byte_off + M.n * M.row_bytes) {
                const int64_t lr = b <= M.byte_off ? 0 : (b - M.byte_off + M.row_bytes - 1) / M.row_bytes;
                r = a.row_off[m] + std::min(lr, M.n);
                break;
            }
        }
        a.cta_row[c] = r;
    }
    // x bytes per CTA: simulate the slices
    int64_t xmax = 0;
    for (int c = 0; c < a.grid; ++c) {
        int64_t xb = 0;
        for (int m = 0; m < a.count; ++m) {
            const int64_t f = std::max(a.cta_row[c], a.row_off[m]);
            const int64_t e = std::min(a.cta_row[c + 1], a.row_off[m + 1]);
            if (f < e) xb += (int64_t)a.batch * (a.mat[m].k / 32) * 80;
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
        if (a.batch <= 1) return launch_one<4, 0, 1>(a, st, pdl);
        if (a.batch <= 2) return launch_one<4, 0, 2>(a, st, pdl);
        return launch_one<4, 0, 4>(a, st, pdl);
    }
    if (a.kind == 1) {
        if (a.batch <= 1) return launch_one<3, 1, 1>(a, st, pdl);
        if (a.batch <= 2) return launch_one<3, 1, 2>(a, st, pdl);
        return launch_one<3, 1, 4>(a, st, pdl);
    }
    if (a.batch <= 1) return launch_one<3, 0, 1>(a, st, pdl);
    if (a.batch <= 2) return launch_one<3, 0, 2>(a, st, pdl);
    return launch_one<3, 0, 4>(a, st, pdl);
}

}  // namespace qx
