// Q4X shared-codebook format (paper Section 3.2, Fig. 3a/3b; Table 2
// "Q4X W4A8G64"): groups of 64 weights, each with an fp16 scale s, a 2-bit
// index naming one of four codebooks, and a 4-bit code per weight; the four
// codebooks of 16 levels are learned per matrix.
//
// The paper gives the pieces, not the arithmetic.  The readings this file
// implements (bit-exact with the CPU oracle) are:
//   1. s = max |w| of the group (an fp16 value; s = 0: a dead group, book 0,
//      codes 0, no part in learning).
//   2. U = rint(fp64(w) / fp64(s) * 2^20), exact integers, |U| <= 2^20.
//   3. A 32-bin histogram of U per group, bin = min(31, (U + 2^20) >> 16).
//   4. "Four histograms that represent all": k-means with 4 centres over the
//      live groups' histograms.  The centres start as the histograms of the
//      groups at ranks floor((2j+1) L / 8) of the order by (sum U^2, position);
//      squared distances are summed in float64 in bin order, ties go to the
//      lower centre; a centre becomes the exact integer sum of its members'
//      histograms over their count (one float64 division per bin); the
//      iteration stops when an assignment repeats, after at most `iters`.
//   5. "Reduce each to 16 samples": the 16-level Lloyd-Max quantizer of the
//      book's values U (at most 16 distinct values: those, padded with the
//      largest; none: the uniform levels ((2j+1)/16 - 1) 2^20; else quantile
//      start, float64 nearest level with ties to the lower, exact integer cell
//      sums, one float64 division, stop when an assignment repeats), sorted;
//      codebook entry = fp16(level / 2^20), one rounding.
//   6. Codes: the nearest of the 16 candidates fp16(fp32(s) fp32(CB[b][j]))
//      (ties to the lower j); dequantization w_hat = fp16(fp32(s) fp32(CB[b][q])).
//
// GPU form of the learner.  Every reduction is an integer reduction (atomics
// on integers commute), and every float64 step is one IEEE operation in the
// oracle's order, so the result does not depend on thread timing:
//   * the k-means start is a 10-pass radix select (8-bit digits) of the four
//     ranks over the 80-bit keys (sum U^2 in bits 32..79, group index in bits
//     0..31), which orders the groups exactly as the (sum U^2, position) sort;
//   * the Lloyd-Max step of a book runs on the histogram of its values over
//     all 2^21 + 1 integers U: the nearest level, the cell sums and the
//     repeat test depend only on a value and its count, and quantiles are
//     prefix sums of the histogram;
//   * the iteration loops are launched `iters` times and stop on the device:
//     a kernel whose stage has converged returns at once, so the host never
//     waits on the device.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kOne = 1 << 20;            // fixed-point unit of the normalised values U
constexpr int kNV = 2 * kOne + 1;        // integers U = -2^20 .. 2^20
constexpr int kBins = 32;                // histogram bins per group
constexpr int kBooks = 4;
constexpr int kLevels = 16;
constexpr int kSelectPasses = 10;        // 80-bit keys, 8-bit digits
constexpr int kThreads = 256;

// Learner state at the start of the workspace (zero-filled by the call).
struct Q4xState {
    unsigned long long live;                      // L, live groups
    unsigned long long rank[kBooks];              // remaining rank of each select target
    unsigned long long key_hi[kBooks];            // selected key digits, sum U^2 part
    unsigned long long key_lo[kBooks];            // selected key digits, group-index part
    unsigned long long km_sum[kBooks][kBins];     // member histogram sums of an iteration
    unsigned long long km_cnt[kBooks];
    double centre[kBooks][kBins];
    unsigned long long book_n[kBooks];            // values per book
    unsigned long long distinct[kBooks];          // distinct values per book
    unsigned long long cell_sum[kBooks][kLevels]; // int64 cell sums (two's complement)
    unsigned long long cell_cnt[kBooks][kLevels];
    double level[kBooks][kLevels];
    unsigned int km_changed, km_done;
    int km_final;                                 // 0: no k-means step ran; else 1 + buffer
    unsigned int error;                           // an internal consistency check failed
    unsigned int ll_changed[kBooks], ll_done[kBooks];
};
static_assert(sizeof(Q4xState) <= 4096, "learner state fits its region");

constexpr size_t round256(size_t b) { return (b + 255) & ~(size_t)255; }

// Workspace regions; the first three are zero-filled by every call.
struct Q4xLayout {
    size_t state, select_hist, value_hist, value_assign, group_hist, group_m2, assign, total, zeroed;
    explicit Q4xLayout(int64_t groups) {
        state = 0;
        select_hist = 4096;
        value_hist = select_hist + round256(sizeof(uint32_t) * kSelectPasses * kBooks * 256);
        value_assign = value_hist + round256(sizeof(uint32_t) * (size_t)kBooks * kNV);
        zeroed = value_assign;
        group_hist = value_assign + round256((size_t)kBooks * kNV);
        group_m2 = group_hist + round256((size_t)groups * kBins);
        assign = group_m2 + round256((size_t)groups * 8);
        total = assign + round256((size_t)groups * 2);
    }
};

// fp16 value as an exact integer multiple of 2^-24 (finite or not: only the
// bit pattern is read, so no input can take an index out of range).
__device__ __forceinline__ long long f16_fixed24(uint32_t h) {
    const uint32_t e = (h >> 10) & 31u, m = h & 1023u;
    const long long mag = e ? (long long)(m | 1024u) << (e - 1) : (long long)m;
    return (h & 0x8000u) ? -mag : mag;
}

__device__ __forceinline__ double f16_bits_to_f64(uint32_t b) {
    return (double)__half2float(__ushort_as_half((unsigned short)b));  // exact
}

__device__ __forceinline__ uint16_t f64_to_f16_bits(double x) {
    uint16_t h;
    asm("cvt.rn.f16.f64 %0, %1;" : "=h"(h) : "d"(x));  // one rounding from float64
    return h;
}

// U = rint(fp64(w) / fp64(s) * 2^20) for a live group (s > 0), clamped so
// that a value can always index the value histogram.
__device__ __forceinline__ int normalised(uint32_t wbits, double s) {
    const double q = __dmul_rn(__ddiv_rn(f16_bits_to_f64(wbits), s), (double)kOne);
    long long u = __double2ll_rn(q);
    u = u < -kOne ? -kOne : (u > kOne ? kOne : u);
    return (int)u;
}

__device__ __forceinline__ int warp_max_i(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ long long warp_sum_ll(long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ uint32_t book_of(const uint8_t *a0, const uint8_t *a1, int final_buf, int64_t gi) {
    if (final_buf == 1) return a0[gi] & 3u;
    if (final_buf == 2) return a1[gi] & 3u;
    return 0u;
}

// ---------------------------------------------------------------- steps 1-3
// One warp per group (lane l holds weights 2l, 2l+1): the scale, the live
// count, the 32-bin histogram and sum U^2.  A group holding NaN or Inf raises
// the non-finite status and is written as a dead group.
__global__ void __launch_bounds__(kThreads) q4x_stats_kernel(const __half *W, int64_t k, int G, int64_t groups,
                                                             __half *scales, uint8_t *ghist, long long *gm2,
                                                             Q4xState *st, uint32_t *status) {
    __shared__ uint32_t hist[kThreads / 32][kBins];
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const int64_t nwarps = (int64_t)gridDim.x * (kThreads / 32);
    for (int64_t gi = (int64_t)blockIdx.x * (kThreads / 32) + wib; gi < groups; gi += nwarps) {
        const int64_t row = gi / G, j = gi % G;
        const uint32_t pair = reinterpret_cast<const uint32_t *>(W + row * k + 64 * j)[lane];
        const uint32_t m0 = pair & 0x7FFFu, m1 = (pair >> 16) & 0x7FFFu;
        const bool bad = __any_sync(0xffffffffu, m0 >= 0x7C00u || m1 >= 0x7C00u);
        int smax = warp_max_i((int)max(m0, m1));  // |fp16| bit patterns order like their values
        if (bad) {
            smax = 0;
            if (lane == 0) atomicOr(status, kStatusNonfinite);
        }
        if (lane == 0) scales[gi] = __ushort_as_half((unsigned short)smax);
        if (smax == 0) continue;  // dead: no histogram, no part in learning
        if (lane == 0) atomicAdd(&st->live, 1ull);
        const double s = f16_bits_to_f64((uint32_t)smax);
        const int u0 = normalised(pair & 0xFFFFu, s), u1 = normalised(pair >> 16, s);
        hist[wib][lane] = 0;
        __syncwarp();
        atomicAdd(&hist[wib][min(31, (u0 + kOne) >> 16)], 1u);
        atomicAdd(&hist[wib][min(31, (u1 + kOne) >> 16)], 1u);
        __syncwarp();
        ghist[gi * kBins + lane] = (uint8_t)hist[wib][lane];
        const long long m2 = warp_sum_ll((long long)u0 * u0 + (long long)u1 * u1);
        if (lane == 0) gm2[gi] = m2;
        __syncwarp();  // the histogram row is reused by the warp's next group
    }
}

// ---------------------------------------------------------------- step 4 start
// Digit p (0 = most significant) of the 80-bit key (hi = sum U^2 < 2^48 in
// bits 32..79, lo = group index in bits 0..31), and whether the key's digits
// above p equal the ones selected so far.
__device__ __forceinline__ uint32_t key_digit(unsigned long long hi, unsigned long long lo, int p) {
    return p < 6 ? (uint32_t)(hi >> (40 - 8 * p)) & 255u : (uint32_t)(lo >> (72 - 8 * p)) & 255u;
}

__device__ __forceinline__ bool key_prefix_match(unsigned long long hi, unsigned long long lo, unsigned long long phi,
                                                 unsigned long long plo, int p) {
    if (p == 0) return true;
    if (p <= 6) return (hi >> (48 - 8 * p)) == (phi >> (48 - 8 * p));
    return hi == phi && (lo >> (32 - 8 * (p - 6))) == (plo >> (32 - 8 * (p - 6)));
}

// Pass p of the radix select: the digit histogram of the live keys that match
// each target's selected prefix.
__global__ void __launch_bounds__(kThreads) q4x_select_hist_kernel(const __half *scales, const long long *gm2,
                                                                   int64_t groups, const Q4xState *st,
                                                                   uint32_t *hist_p, int p) {
    __shared__ uint32_t h[kBooks][256];
    __shared__ unsigned long long phi[kBooks], plo[kBooks];
    if (st->live == 0) return;
    for (int i = threadIdx.x; i < kBooks * 256; i += kThreads) h[i / 256][i % 256] = 0;
    if (threadIdx.x < kBooks) {
        phi[threadIdx.x] = st->key_hi[threadIdx.x];
        plo[threadIdx.x] = st->key_lo[threadIdx.x];
    }
    __syncthreads();
    const unsigned short *sb = reinterpret_cast<const unsigned short *>(scales);
    for (int64_t gi = (int64_t)blockIdx.x * kThreads + threadIdx.x; gi < groups; gi += (int64_t)gridDim.x * kThreads) {
        if (sb[gi] == 0) continue;
        const unsigned long long hi = (unsigned long long)gm2[gi], lo = (unsigned long long)gi;
        const uint32_t d = key_digit(hi, lo, p);
#pragma unroll
        for (int t = 0; t < kBooks; ++t)
            if (key_prefix_match(hi, lo, phi[t], plo[t], p)) atomicAdd(&h[t][d], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < kBooks * 256; i += kThreads)
        if (h[i / 256][i % 256] != 0) atomicAdd(&hist_p[i], h[i / 256][i % 256]);
}

// Pass p, one warp per target: the digit whose cumulative count first exceeds
// the target's remaining rank.  Pass 0 sets the ranks floor((2t+1) L / 8).
__global__ void __launch_bounds__(32 * kBooks) q4x_select_pick_kernel(Q4xState *st, const uint32_t *hist_p, int p) {
    const int t = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const unsigned long long L = st->live;
    if (L == 0) return;
    const unsigned long long r = p == 0 ? ((2ull * t + 1ull) * L) / 8ull : st->rank[t];
    uint32_t c[8];
    unsigned long long sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        c[i] = hist_p[t * 256 + 8 * lane + i];
        sum += c[i];
    }
    unsigned long long incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
    }
    const unsigned long long excl = incl - sum;
    const bool mine = excl <= r && r < incl;
    const uint32_t who = __ballot_sync(0xffffffffu, mine);
    if (who == 0) {  // cannot happen when the histograms are consistent
        if (lane == 0) atomicOr(&st->error, 1u);
        return;
    }
    if (mine) {
        unsigned long long acc = excl;
        int d = 8 * lane;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            if (r < acc + c[i]) {
                d = 8 * lane + i;
                break;
            }
            acc += c[i];
        }
        st->rank[t] = r - acc;
        if (p < 6)
            st->key_hi[t] |= (unsigned long long)d << (40 - 8 * p);
        else
            st->key_lo[t] |= (unsigned long long)d << (72 - 8 * p);
    }
}

// The starting centres: the histograms of the selected groups.
__global__ void q4x_km_init_kernel(const uint8_t *ghist, int64_t groups, Q4xState *st) {
    if (st->live == 0) return;
    const int t = threadIdx.x >> 5, b = threadIdx.x & 31;
    unsigned long long gi = st->key_lo[t];
    if (gi >= (unsigned long long)groups) {
        if (b == 0) atomicOr(&st->error, 2u);
        gi = 0;
    }
    st->centre[t][b] = (double)ghist[gi * kBins + b];
}

// ---------------------------------------------------------------- step 4 iteration
// Iteration t: thread per live group, nearest centre (float64, bins in order,
// ties to the lower), written to a_cur; the members' histograms are summed for
// the update in integers.  A change against a_prev (t > 0) is flagged.
__global__ void __launch_bounds__(kThreads) q4x_km_assign_kernel(const __half *scales, const uint8_t *ghist,
                                                                 int64_t groups, Q4xState *st, uint8_t *a_cur,
                                                                 const uint8_t *a_prev, int t) {
    __shared__ double C[kBooks][kBins];
    __shared__ uint32_t sum[kBooks][kBins];
    __shared__ uint32_t cnt[kBooks];
    __shared__ int changed;
    if (st->km_done != 0 || st->live == 0) return;
    for (int i = threadIdx.x; i < kBooks * kBins; i += kThreads) {
        C[i / kBins][i % kBins] = st->centre[i / kBins][i % kBins];
        sum[i / kBins][i % kBins] = 0;
    }
    if (threadIdx.x < kBooks) cnt[threadIdx.x] = 0;
    if (threadIdx.x == 0) changed = 0;
    __syncthreads();
    const unsigned short *sb = reinterpret_cast<const unsigned short *>(scales);
    for (int64_t gi = (int64_t)blockIdx.x * kThreads + threadIdx.x; gi < groups; gi += (int64_t)gridDim.x * kThreads) {
        if (sb[gi] == 0) continue;
        const uint4 *hp = reinterpret_cast<const uint4 *>(ghist + gi * kBins);
        const uint4 h0 = hp[0], h1 = hp[1];
        const uint32_t hw[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
        double D[kBooks] = {0.0, 0.0, 0.0, 0.0};
#pragma unroll
        for (int b = 0; b < kBins; ++b) {
            const double h = (double)((hw[b >> 2] >> (8 * (b & 3))) & 255u);
#pragma unroll
            for (int c = 0; c < kBooks; ++c) {
                const double d = __dsub_rn(h, C[c][b]);
                D[c] = __dadd_rn(D[c], __dmul_rn(d, d));
            }
        }
        int best = 0;
#pragma unroll
        for (int c = 1; c < kBooks; ++c)
            if (D[c] < D[best]) best = c;
        if (t > 0 && a_prev[gi] != best) changed = 1;
        a_cur[gi] = (uint8_t)best;
#pragma unroll
        for (int b = 0; b < kBins; ++b) {
            const uint32_t h = (hw[b >> 2] >> (8 * (b & 3))) & 255u;
            if (h != 0) atomicAdd(&sum[best][b], h);
        }
        atomicAdd(&cnt[best], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < kBooks * kBins; i += kThreads)
        if (sum[i / kBins][i % kBins] != 0) atomicAdd(&st->km_sum[i / kBins][i % kBins], (unsigned long long)sum[i / kBins][i % kBins]);
    if (threadIdx.x < kBooks && cnt[threadIdx.x] != 0) atomicAdd(&st->km_cnt[threadIdx.x], (unsigned long long)cnt[threadIdx.x]);
    if (threadIdx.x == 0 && changed) atomicOr(&st->km_changed, 1u);
}

// Iteration t, one block of 4 x 32 threads: stop if the assignment repeated,
// else move every centre with members to their mean and clear the sums.
__global__ void q4x_km_update_kernel(Q4xState *st, int t) {
    __shared__ int stop;
    if (st->km_done != 0 || st->live == 0) return;
    if (threadIdx.x == 0) stop = (t > 0 && st->km_changed == 0);
    __syncthreads();
    if (stop) {
        if (threadIdx.x == 0) {
            st->km_done = 1;
            st->km_final = 1 + (t & 1);  // equal to the previous assignment
        }
        return;
    }
    const int c = threadIdx.x >> 5, b = threadIdx.x & 31;
    const unsigned long long n = st->km_cnt[c];
    if (n != 0) st->centre[c][b] = __ddiv_rn((double)st->km_sum[c][b], (double)n);
    __syncthreads();  // every thread has read its count before it is cleared
    st->km_sum[c][b] = 0;
    if (b == 0) st->km_cnt[c] = 0;
    if (threadIdx.x == 0) {
        st->km_changed = 0;
        st->km_final = 1 + (t & 1);
    }
}

// ---------------------------------------------------------------- step 5 data
// One warp per live group: its 64 values U counted in its book's histogram.
__global__ void __launch_bounds__(kThreads) q4x_value_hist_kernel(const __half *W, int64_t k, int G, int64_t groups,
                                                                  const __half *scales, const uint8_t *a0,
                                                                  const uint8_t *a1, Q4xState *st, uint32_t *vh) {
    const int lane = threadIdx.x & 31;
    const int final_buf = st->km_final;
    const int64_t nwarps = (int64_t)gridDim.x * (kThreads / 32);
    const unsigned short *sb = reinterpret_cast<const unsigned short *>(scales);
    for (int64_t gi = (int64_t)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); gi < groups; gi += nwarps) {
        const uint32_t sbits = sb[gi];
        if (sbits == 0) continue;
        const int64_t row = gi / G, j = gi % G;
        const uint32_t pair = reinterpret_cast<const uint32_t *>(W + row * k + 64 * j)[lane];
        const double s = f16_bits_to_f64(sbits);
        const uint32_t b = book_of(a0, a1, final_buf, gi);
        uint32_t *h = vh + (size_t)b * kNV + kOne;
        atomicAdd(h + normalised(pair & 0xFFFFu, s), 1u);
        atomicAdd(h + normalised(pair >> 16, s), 1u);
        if (lane == 0) atomicAdd(&st->book_n[b], 64ull);
    }
}

// Distinct values per book (non-zero histogram entries).
__global__ void __launch_bounds__(kThreads) q4x_distinct_kernel(const uint32_t *vh, Q4xState *st) {
    __shared__ uint32_t cnt[kBooks];
    if (threadIdx.x < kBooks) cnt[threadIdx.x] = 0;
    __syncthreads();
    const int64_t total = (int64_t)kBooks * kNV;
    for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < total; i += (int64_t)gridDim.x * kThreads)
        if (vh[i] != 0) atomicAdd(&cnt[i / kNV], 1u);
    __syncthreads();
    if (threadIdx.x < kBooks && cnt[threadIdx.x] != 0) atomicAdd(&st->distinct[threadIdx.x], (unsigned long long)cnt[threadIdx.x]);
}

// Exclusive prefix sum over the block (1024 threads); every thread gets its
// own offset and the block total.
template <typename T>
__device__ T block_exclusive_scan(T v, T *warp_tot, T &total) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    T incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const T u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += u;
    }
    if (lane == 31) warp_tot[w] = incl;
    __syncthreads();
    if (w == 0) {
        T x = warp_tot[lane];
        T xi = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const T u = __shfl_up_sync(0xffffffffu, xi, o);
            if (lane >= o) xi += u;
        }
        warp_tot[lane] = xi - x;  // exclusive offset of warp `lane`
        if (lane == 31) warp_tot[32] = xi;
    }
    __syncthreads();
    const T r = warp_tot[w] + incl - v;
    total = warp_tot[32];
    __syncthreads();  // warp_tot may be reused by the caller
    return r;
}

constexpr int kSetupThreads = 1024;
constexpr int kSetupChunk = (kNV + kSetupThreads - 1) / kSetupThreads;

// Block b (1024 threads): the starting levels of book b.  No values: the
// uniform levels; at most 16 distinct values: those, padded with the largest
// (final); else the quantiles floor((2j+1) N / 32) of the book's values.
__global__ void __launch_bounds__(kSetupThreads) q4x_lloyd_setup_kernel(const uint32_t *vh, Q4xState *st) {
    __shared__ unsigned long long wt[33];
    const int b = blockIdx.x;
    const unsigned long long N = st->book_n[b];
    if (N == 0) {
        if (threadIdx.x < kLevels) st->level[b][threadIdx.x] = ((2.0 * threadIdx.x + 1.0) / kLevels - 1.0) * kOne;
        if (threadIdx.x == 0) st->ll_done[b] = 1;
        return;
    }
    const uint32_t *h = vh + (size_t)b * kNV;
    const int lo = threadIdx.x * kSetupChunk, hi = min(kNV, lo + kSetupChunk);
    const bool few = st->distinct[b] <= (unsigned long long)kLevels;
    unsigned long long mine = 0;
    for (int v = lo; v < hi; ++v) mine += few ? (h[v] != 0) : h[v];
    unsigned long long total = 0;
    const unsigned long long off = block_exclusive_scan<unsigned long long>(mine, wt, total);
    if (few) {
        unsigned long long o = off;
        for (int v = lo; v < hi && o < kLevels; ++v)
            if (h[v] != 0) st->level[b][o++] = (double)(v - kOne);
        __syncthreads();
        if (threadIdx.x == 0) {
            int D = (int)min(total, (unsigned long long)kLevels);
            if (D == 0) {  // N > 0 implies a non-zero entry: flag the inconsistency
                atomicOr(&st->error, 4u);
                st->level[b][0] = 0.0;
                D = 1;
            }
            for (int i = D; i < kLevels; ++i) st->level[b][i] = st->level[b][D - 1];
            st->ll_done[b] = 1;
        }
        return;
    }
    for (int j = 0; j < kLevels; ++j) {
        const unsigned long long r = ((2ull * j + 1ull) * N) / (2ull * kLevels);
        if (off <= r && r < off + mine) {
            unsigned long long acc = off;
            for (int v = lo; v < hi; ++v) {
                acc += h[v];
                if (acc > r) {
                    st->level[b][j] = (double)(v - kOne);
                    break;
                }
            }
        }
    }
}

// ---------------------------------------------------------------- step 5 iteration
constexpr int kLloydBlocks = 128;  // blocks per book

// Iteration t over the values of book blockIdx.y: nearest level (float64
// |U - c_j|, ties to the lower), exact cell sums of count x U, and a flag when
// a value's level differs from iteration t - 1 (va holds the last levels).
__global__ void __launch_bounds__(kThreads) q4x_lloyd_assign_kernel(const uint32_t *vh, uint8_t *va, Q4xState *st,
                                                                    int t) {
    __shared__ double c[kLevels];
    __shared__ unsigned long long sum[kLevels], cnt[kLevels];
    __shared__ int changed;
    const int b = blockIdx.y;
    if (st->ll_done[b] != 0) return;
    if (threadIdx.x < kLevels) {
        c[threadIdx.x] = st->level[b][threadIdx.x];
        sum[threadIdx.x] = 0;
        cnt[threadIdx.x] = 0;
    }
    if (threadIdx.x == 0) changed = 0;
    __syncthreads();
    const uint32_t *h = vh + (size_t)b * kNV;
    uint8_t *a = va + (size_t)b * kNV;
    for (int v = blockIdx.x * kThreads + threadIdx.x; v < kNV; v += gridDim.x * kThreads) {
        const uint32_t n = h[v];
        if (n == 0) continue;
        const long long u = (long long)v - kOne;
        const double x = (double)u;
        int best = 0;
        double bd = fabs(__dsub_rn(x, c[0]));
#pragma unroll
        for (int j = 1; j < kLevels; ++j) {
            const double d = fabs(__dsub_rn(x, c[j]));
            if (d < bd) {
                bd = d;
                best = j;
            }
        }
        if (t > 0 && a[v] != best) changed = 1;
        a[v] = (uint8_t)best;
        atomicAdd(&sum[best], (unsigned long long)(u * (long long)n));  // two's complement: exact int64 sum
        atomicAdd(&cnt[best], (unsigned long long)n);
    }
    __syncthreads();
    if (threadIdx.x < kLevels && cnt[threadIdx.x] != 0) {
        atomicAdd(&st->cell_sum[b][threadIdx.x], sum[threadIdx.x]);
        atomicAdd(&st->cell_cnt[b][threadIdx.x], cnt[threadIdx.x]);
    }
    if (threadIdx.x == 0 && changed) atomicOr(&st->ll_changed[b], 1u);
}

// Iteration t, one block of 4 x 16 threads: a book whose assignment repeated
// stops; else every level with values moves to its cell mean.
__global__ void q4x_lloyd_update_kernel(Q4xState *st, int t) {
    __shared__ int stop[kBooks];
    const int b = threadIdx.x / kLevels, j = threadIdx.x % kLevels;
    if (j == 0) stop[b] = st->ll_done[b] != 0 ? 2 : ((t > 0 && st->ll_changed[b] == 0) ? 1 : 0);
    __syncthreads();
    if (stop[b] == 2) return;
    if (stop[b] == 1) {
        if (j == 0) st->ll_done[b] = 1;
        return;
    }
    const unsigned long long n = st->cell_cnt[b][j];
    if (n != 0) st->level[b][j] = __ddiv_rn((double)(long long)st->cell_sum[b][j], (double)n);
    st->cell_sum[b][j] = 0;
    st->cell_cnt[b][j] = 0;
    if (j == 0) st->ll_changed[b] = 0;
}

// The codebooks: each book's levels sorted ascending, fp16(level / 2^20).
__global__ void q4x_codebook_kernel(const Q4xState *st, __half *codebooks) {
    const int b = threadIdx.x;
    if (b >= kBooks) return;
    double v[kLevels];
    for (int j = 0; j < kLevels; ++j) v[j] = st->level[b][j];
    for (int i = 1; i < kLevels; ++i) {  // insertion sort: equal levels are equal values
        const double x = v[i];
        int j = i - 1;
        while (j >= 0 && v[j] > x) {
            v[j + 1] = v[j];
            --j;
        }
        v[j + 1] = x;
    }
    for (int j = 0; j < kLevels; ++j)
        codebooks[b * kLevels + j] = __ushort_as_half(f64_to_f16_bits(__dmul_rn(v[j], 1.0 / kOne)));
}

// ---------------------------------------------------------------- step 6
// One warp per four groups of a row (groups 4m .. 4m+3, one packed book byte):
// lane l codes the eight weights 8(l % 8) .. 8(l % 8) + 7 of group 4m + l / 8
// against its 16 candidates, compared exactly as integers of 2^-24.
__global__ void __launch_bounds__(kThreads) q4x_codes_kernel(const __half *W, int64_t n, int64_t k, int G,
                                                             int bbytes, const __half *scales, const uint8_t *a0,
                                                             const uint8_t *a1, const Q4xState *st,
                                                             const __half *codebooks, uint8_t *codes,
                                                             uint8_t *books) {
    __shared__ float cb[kBooks * kLevels];
    if (threadIdx.x < kBooks * kLevels) cb[threadIdx.x] = __half2float(codebooks[threadIdx.x]);
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int final_buf = st->km_final;
    const int64_t units = n * bbytes;
    const int64_t nwarps = (int64_t)gridDim.x * (kThreads / 32);
    const unsigned short *sb = reinterpret_cast<const unsigned short *>(scales);
    for (int64_t wu = (int64_t)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); wu < units; wu += nwarps) {
        const int64_t row = wu / bbytes;
        const int m = (int)(wu % bbytes);
        const int j = 4 * m + (lane >> 3);
        uint32_t book = 0;
        if (j < G) {
            const int64_t gi = row * G + j;
            const uint32_t sbits = sb[gi];
            book = sbits != 0 ? book_of(a0, a1, final_buf, gi) : 0u;
            const float s = __half2float(__ushort_as_half((unsigned short)sbits));
            long long cand[kLevels];
#pragma unroll
            for (int i = 0; i < kLevels; ++i)  // exact fp32 product, one rounding to fp16
                cand[i] = f16_fixed24(__half_as_ushort(__float2half_rn(__fmul_rn(s, cb[book * kLevels + i]))));
            const int64_t off = row * k + 64 * (int64_t)j + 8 * (lane & 7);
            const uint4 wv = *reinterpret_cast<const uint4 *>(W + off);
            const uint32_t ww[4] = {wv.x, wv.y, wv.z, wv.w};
            uint32_t word = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const long long x = f16_fixed24((ww[e >> 1] >> (16 * (e & 1))) & 0xFFFFu);
                int q = 0;
                long long bd = llabs(x - cand[0]);
#pragma unroll
                for (int i = 1; i < kLevels; ++i) {
                    const long long d = llabs(x - cand[i]);
                    if (d < bd) {
                        bd = d;
                        q = i;
                    }
                }
                word |= (uint32_t)q << (4 * (e / 2 + 4 * (e % 2)));
            }
            reinterpret_cast<uint32_t *>(codes)[off >> 3] = word;
        }
        uint32_t byte = 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) byte |= (__shfl_sync(0xffffffffu, book, 8 * q) & 3u) << (2 * q);
        if (lane == 0) books[row * bbytes + m] = (uint8_t)byte;
    }
}

// ---------------------------------------------------------------- step 7
__device__ __forceinline__ uint32_t book_index(const uint8_t *books_row, int j) {
    return (books_row[j >> 2] >> (2 * (j & 3))) & 3u;
}

// Thread per packed word (8 codes): w_hat = fp16(fp32(s) fp32(CB[b][q])).
__global__ void __launch_bounds__(kThreads) q4x_dequant_kernel(Q4xMat m, __half *out) {
    __shared__ float cb[kBooks * kLevels];
    if (threadIdx.x < kBooks * kLevels) cb[threadIdx.x] = __half2float(m.codebooks[threadIdx.x]);
    __syncthreads();
    const int64_t wpr = m.k / 8, words = m.n * wpr;
    for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < words; i += (int64_t)gridDim.x * kThreads) {
        const int64_t row = i / wpr, t = i % wpr;
        const int j = (int)(t >> 3);  // 8 words per group of 64
        const float s = __half2float(m.scales[row * m.G + j]);
        const float *tb = cb + kLevels * book_index(m.books + row * m.bbytes, j);
        const uint32_t w = reinterpret_cast<const uint32_t *>(m.codes)[i];
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
            const uint32_t q0 = (w >> (4 * (e / 2))) & 15u, q1 = (w >> (4 * (e / 2 + 4))) & 15u;
            const uint32_t h0 = __half_as_ushort(__float2half_rn(__fmul_rn(s, tb[q0])));
            const uint32_t h1 = __half_as_ushort(__float2half_rn(__fmul_rn(s, tb[q1])));
            o[e / 2] = h0 | (h1 << 16);
        }
        reinterpret_cast<uint4 *>(out)[i] = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

// ---------------------------------------------------------------- decode matmul
constexpr int kGemvWarps = 8;  // warps per block

// w_hat of one 32-weight unit (16 code bytes): half2 pairs (k = 2i, 2i + 1),
// the codebook entries times s in fp16, which is exactly fp16(fp32(s) fp32(CB)).
__device__ __forceinline__ void unit_weights(const uint4 &cw, const __half *tb, __half2 s2, __half2 (&w)[16]) {
    const uint32_t ws[4] = {cw.x, cw.y, cw.z, cw.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t sel = (ws[t] >> (4 * i)) & 0x000F000Fu;  // codes of k = 8t+2i, 8t+2i+1
            w[4 * t + i] = __hmul2(__halves2half2(tb[sel & 15u], tb[sel >> 16]), s2);
        }
    }
}

// acc[b] += the unit's 32 products with x[b][32u .. 32u+31]: the products and
// their sums over 16 pairs in fp16 (two chains of eight HFMA2), then fp32.
template <int NB>
__device__ __forceinline__ void unit_dot(const __half2 (&w)[16], const __half *x, int64_t k, int u, int batch,
                                         float (&acc)[NB]) {
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        if (b >= batch) break;
        const uint4 *xr = reinterpret_cast<const uint4 *>(x + (int64_t)b * k + 32 * (int64_t)u);
        __half2 c0 = u2h2(0u), c1 = u2h2(0u);
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const uint4 xv = __ldg(xr + v);
            c0 = __hfma2(w[4 * v + 0], u2h2(xv.x), c0);
            c1 = __hfma2(w[4 * v + 1], u2h2(xv.y), c1);
            c0 = __hfma2(w[4 * v + 2], u2h2(xv.z), c0);
            c1 = __hfma2(w[4 * v + 3], u2h2(xv.w), c1);
        }
        const float2 f0 = __half22float2(c0), f1 = __half22float2(c1);
        acc[b] += (f0.x + f0.y) + (f1.x + f1.y);
    }
}

// y_i[b][row] = sum_k w_hat_i[row][k] x_i[b][k] for the rows of up to eight
// matrices, taken as one list (matrix 0's rows, then matrix 1's, ...).  A
// persistent grid of warps strides over the list, one row per warp at a time;
// lane l takes the 32-weight units l, l + 32, ... of the row, two at a time so
// that two code loads are in flight.  The matrices' codebooks sit in shared
// memory (128 bytes each: one word per bank, so any lookup is conflict-free).
template <int NB>
__global__ void __launch_bounds__(32 * kGemvWarps) q4x_gemv_kernel(const __grid_constant__ Q4xGemvMulti a) {
    __shared__ __half cb[kMaxQ4xMats * kBooks * kLevels];
    for (int i = threadIdx.x; i < a.count * kBooks * kLevels; i += 32 * kGemvWarps)
        cb[i] = a.mat[i / (kBooks * kLevels)].codebooks[i % (kBooks * kLevels)];
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int64_t total = a.row_off[a.count];
    const int64_t nwarps = (int64_t)gridDim.x * kGemvWarps;
    for (int64_t gr = (int64_t)blockIdx.x * kGemvWarps + (threadIdx.x >> 5); gr < total; gr += nwarps) {
        int mi = 0;
        while (mi + 1 < a.count && gr >= a.row_off[mi + 1]) ++mi;
        const Q4xMat &m = a.mat[mi];
        const int64_t row = gr - a.row_off[mi];
        const int units = (int)(m.k / 32);
        const uint8_t *brow = m.books + row * m.bbytes;
        const __half *srow = m.scales + row * m.G;
        const uint4 *crow = reinterpret_cast<const uint4 *>(m.codes + row * (m.k / 2));
        const __half *cbm = cb + mi * kBooks * kLevels;
        const __half *x = a.x[mi];
        float acc[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) acc[b] = 0.0f;
        for (int u0 = lane; u0 < units; u0 += 64) {
            const int u1 = u0 + 32;
            const bool two = u1 < units;
            // both units' codes and metadata first, then the arithmetic
            const uint4 c0 = __ldg(crow + u0);
            const uint4 c1 = two ? __ldg(crow + u1) : make_uint4(0u, 0u, 0u, 0u);
            const __half s0 = srow[u0 >> 1], s1 = srow[(two ? u1 : u0) >> 1];
            const uint32_t b0 = book_index(brow, u0 >> 1), b1 = book_index(brow, (two ? u1 : u0) >> 1);
            __half2 w[16];
            unit_weights(c0, cbm + kLevels * b0, __halves2half2(s0, s0), w);
            unit_dot<NB>(w, x, m.k, u0, a.batch, acc);
            if (two) {
                unit_weights(c1, cbm + kLevels * b1, __halves2half2(s1, s1), w);
                unit_dot<NB>(w, x, m.k, u1, a.batch, acc);
            }
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            float v = acc[b];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            acc[b] = v;
        }
        if (lane == 0) {
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                if (b >= a.batch) break;
                if (a.y_f32)
                    reinterpret_cast<float *>(a.y[mi])[(int64_t)b * m.n + row] = acc[b];
                else
                    reinterpret_cast<__half *>(a.y[mi])[(int64_t)b * m.n + row] = __float2half_rn(acc[b]);
            }
        }
    }
}

int grid_for(int64_t items, int per_block, int num_sms) {
    const int64_t need = (items + per_block - 1) / per_block;
    return (int)std::max<int64_t>(1, std::min<int64_t>(need, (int64_t)num_sms * 8));
}

}  // namespace

size_t q4x_workspace_bytes(int64_t n, int64_t k) { return Q4xLayout(n * (k / kQ4xGroup)).total; }

cudaError_t launch_q4x_quantize(const Q4xQuantArgs &a, int num_sms, cudaStream_t st) {
    const int64_t groups = a.n * a.G;
    const Q4xLayout L(groups);
    uint8_t *ws = static_cast<uint8_t *>(a.ws);
    Q4xState *state = reinterpret_cast<Q4xState *>(ws + L.state);
    uint32_t *sel = reinterpret_cast<uint32_t *>(ws + L.select_hist);
    uint32_t *vh = reinterpret_cast<uint32_t *>(ws + L.value_hist);
    uint8_t *va = ws + L.value_assign;
    uint8_t *gh = ws + L.group_hist;
    long long *gm2 = reinterpret_cast<long long *>(ws + L.group_m2);
    uint8_t *a0 = ws + L.assign, *a1 = a0 + groups;
    cudaError_t e = cudaMemsetAsync(ws, 0, L.zeroed, st);
    if (e != cudaSuccess) return e;
    const int gw = grid_for(groups, kThreads / 32, num_sms);  // warp per group
    const int gt = grid_for(groups, kThreads, num_sms);       // thread per group
    q4x_stats_kernel<<<gw, kThreads, 0, st>>>(a.W, a.k, a.G, groups, a.scales, gh, gm2, state, a.status);
    for (int p = 0; p < kSelectPasses; ++p) {
        uint32_t *hp = sel + (size_t)p * kBooks * 256;
        q4x_select_hist_kernel<<<gt, kThreads, 0, st>>>(a.scales, gm2, groups, state, hp, p);
        q4x_select_pick_kernel<<<1, 32 * kBooks, 0, st>>>(state, hp, p);
    }
    q4x_km_init_kernel<<<1, 32 * kBooks, 0, st>>>(gh, groups, state);
    for (int t = 0; t < a.iters; ++t) {
        q4x_km_assign_kernel<<<gt, kThreads, 0, st>>>(a.scales, gh, groups, state, (t & 1) ? a1 : a0,
                                                      (t & 1) ? a0 : a1, t);
        q4x_km_update_kernel<<<1, 32 * kBooks, 0, st>>>(state, t);
    }
    q4x_value_hist_kernel<<<gw, kThreads, 0, st>>>(a.W, a.k, a.G, groups, a.scales, a0, a1, state, vh);
    q4x_distinct_kernel<<<grid_for((int64_t)kBooks * kNV, kThreads, num_sms), kThreads, 0, st>>>(vh, state);
    q4x_lloyd_setup_kernel<<<kBooks, kSetupThreads, 0, st>>>(vh, state);
    for (int t = 0; t < a.iters; ++t) {
        q4x_lloyd_assign_kernel<<<dim3(kLloydBlocks, kBooks), kThreads, 0, st>>>(vh, va, state, t);
        q4x_lloyd_update_kernel<<<1, kBooks * kLevels, 0, st>>>(state, t);
    }
    q4x_codebook_kernel<<<1, 32, 0, st>>>(state, a.codebooks);
    q4x_codes_kernel<<<grid_for(a.n * a.bbytes, kThreads / 32, num_sms), kThreads, 0, st>>>(
        a.W, a.n, a.k, a.G, a.bbytes, a.scales, a0, a1, state, a.codebooks, a.codes, a.books);
    return cudaGetLastError();
}

cudaError_t launch_q4x_dequant(const Q4xMat &m, __half *W, int num_sms, cudaStream_t st) {
    q4x_dequant_kernel<<<grid_for(m.n * (m.k / 8), kThreads, num_sms), kThreads, 0, st>>>(m, W);
    return cudaGetLastError();
}

// Persistent grid: as many blocks as are resident at once (from the kernel's
// occupancy, looked up once per instance), fewer when there are fewer rows.
template <int NB>
cudaError_t launch_gemv_nb(const Q4xGemvMulti &a, int num_sms, cudaStream_t st) {
    static std::atomic<int> per_sm{0};
    int bps = per_sm.load(std::memory_order_relaxed);
    if (bps == 0) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, q4x_gemv_kernel<NB>, 32 * kGemvWarps, 0) !=
                cudaSuccess ||
            bps < 1)
            bps = 1;
        per_sm.store(bps, std::memory_order_relaxed);
    }
    const int64_t blocks = (a.row_off[a.count] + kGemvWarps - 1) / kGemvWarps;
    const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(blocks, (int64_t)bps * num_sms));
    q4x_gemv_kernel<NB><<<grid, 32 * kGemvWarps, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_q4x_gemv(const Q4xGemvMulti &a, int num_sms, cudaStream_t st) {
    if (a.batch <= 1) return launch_gemv_nb<1>(a, num_sms, st);
    if (a.batch <= 2) return launch_gemv_nb<2>(a, num_sms, st);
    if (a.batch <= 4) return launch_gemv_nb<4>(a, num_sms, st);
    if (a.batch <= 8) return launch_gemv_nb<8>(a, num_sms, st);
    return launch_gemv_nb<16>(a, num_sms, st);
}

}  // namespace qx
