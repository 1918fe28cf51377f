// Decode matmul y[b][n] = sum_k w_hat[n][k] x[b][k] on CUDA cores, fed by TMA.
//
// Decoding reads every weight once per token, so it is bound by HBM bandwidth
// and by the cost of unpacking the codes (paper Section 2.4).  On GB300 the
// unpack of a 3-bit code through an 8-entry table costs about one byte-permute
// per weight, which at HBM speed keeps the integer pipe nearly busy: the
// kernel is built to spend as few issue slots as possible on anything else.
//
//   * Work unit: a 32-row block of one matrix.  Lane r of every warp owns row
//     r of the block, so a row's dot product never needs a warp shuffle and
//     the activations x are the same for all lanes (a broadcast load).
//   * The rows are streamed in slices of 1024 weights: one stage of the
//     shared-memory ring holds the codes (and LUTs) of 32 rows x 1024 k,
//     fetched with 2-D/3-D TMA tensor copies in the 128-byte swizzled layout,
//     which makes the per-lane 16-byte reads of 32 different rows free of bank
//     conflicts.
//   * Sixteen warps in four groups of four: group g decodes the stages q with
//     q % 4 == g, and each of its warps one 256-weight part of each of them
//     (two 3-bit superblocks), so four stages are in decode at once.
//   * No producer warp (a seventeenth warp puts five warps on one SM
//     sub-partition, which caps every thread at 96 registers): the first
//     stages are issued from the kernel parameters by one lane each before the
//     programmatic-dependent-launch wait (weights do not depend on the
//     previous kernel); the rest of the ring is requested as those land, and
//     afterwards the last warp of a group to release a stage refills it.
//   * Partial sums of a row block stay in registers across its slices; at the
//     end of the block each warp stores its partials and the last contributor
//     adds them in a fixed order (deterministic) and writes y.
//   * Uniform scales and zero-points are read by each lane from global memory
//     one stage ahead, after the block's first copy has pulled its metadata
//     into L2 with a bulk prefetch.
// One CTA of 512 threads per SM.  Under programmatic dependent launch the
// next decode kernel's CTA takes an SM as soon as this kernel's CTA there has
// exited and issues its weight copies before it waits.  Every wait is
// bounded in time and reports QX_ERR_TIMEOUT through the device status.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kGroups = 4;       // warp groups; group g takes the stages q with q % kGroups == g
constexpr int kGroupWarps = 4;   // warps per group, one 256-weight part of a stage each
constexpr int kWarps = kGroups * kGroupWarps;
constexpr int kThreads = 32 * kWarps;
constexpr int kRows = 32;           // rows per block (one per lane)
constexpr int kSliceK = 1024;       // weights per row per stage
constexpr int kPartK = kSliceK / kGroupWarps;  // weights per warp per stage
constexpr int kBox = kRows * 128;   // one 32-row x 128-byte TMA box
constexpr int kMaxRing = 8;
// Stages issued at start (GemvMulti::initial): one per warp group for a
// standalone launch -- requesting the whole ring at once makes every stage
// land late, as the memory system serves them interleaved; the rest of the
// ring is issued as the first stages land.  A launch that follows another
// kernel under programmatic dependent launch requests the whole ring, whose
// latency then hides behind the previous kernel.
constexpr int kMaxRbSlots = 16;
constexpr int kHeader = 1024;       // barriers, counters, per-matrix CTA plan
constexpr int kSmemBudget = 220 * 1024;

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(b), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(b), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: false after `limit_ns`, or once another warp has raised the
// abort flag (when `abort_flag` is not null).
__device__ __noinline__ bool mbar_wait(uint32_t b, uint32_t parity, uint64_t limit_ns,
                                       volatile uint32_t *abort_flag) {
    if (mbar_try_wait(b, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        if (mbar_try_wait(b, parity)) return true;
        if (abort_flag != nullptr && *abort_flag) return false;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

// Bounded wait for a shared-memory word to reach `want`.
__device__ __noinline__ bool wait_equal(uint32_t *p, uint32_t want, uint64_t limit_ns,
                                        volatile uint32_t *abort_flag) {
    volatile uint32_t *v = p;
    if (*v == want) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        if (*v == want) {
            __threadfence_block();
            return true;
        }
        if (*abort_flag) return false;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

__device__ __forceinline__ void tma_2d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::
            "r"(dst),
        "l"(map), "r"(bar), "r"(x), "r"(y)
        : "memory");
}

__device__ __forceinline__ void tma_3d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y, int z) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], "
        "[%2];" ::"r"(dst),
        "l"(map), "r"(bar), "r"(x), "r"(y), "r"(z)
        : "memory");
}

__device__ __forceinline__ void prefetch_l2_bulk(const void *p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Shared-memory loads with 32-bit shared-window addresses.  The ring's
// contents change between barrier phases, so these are volatile: they are
// neither merged nor moved across the (volatile) barrier waits.
__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
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

// 32 activations x[k .. k+31] from shared memory (the same address in every
// lane: a broadcast).
__device__ __forceinline__ void load_x32(uint32_t p, __half2 (&x)[16]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 t = lds128(p + 16u * i);
        x[4 * i + 0] = u2h2(t.x);
        x[4 * i + 1] = u2h2(t.y);
        x[4 * i + 2] = u2h2(t.z);
        x[4 * i + 3] = u2h2(t.w);
    }
}

// Offset of 16-byte chunk `c` of 128-byte box row `r` inside a 1024-byte-aligned
// TMA box written with CU_TENSOR_MAP_SWIZZLE_128B (chunk index XOR row % 8).
__device__ __forceinline__ uint32_t swz(int r, int c) {
    return (uint32_t)(r * 128 + (((c ^ r) & 7) << 4));
}

// Per-matrix fields of this CTA, built once in shared memory.
struct MatS {
    const uint8_t *zeros;
    const __half *scales;
    const __half *x;
    void *y;
    int n, K, G, zbytes, log2g, nks, nlb;
    int xoff;   // shared-memory offset (halves) of this matrix's x
    int q0;     // first CTA-local stage of this matrix
    int rbq0;   // first CTA-local row block of this matrix
    int rb0;    // first matrix-local row block of this CTA
    int nrb;    // row blocks of this CTA in this matrix
};

struct Header {
    uint64_t full[kMaxRing];
    uint32_t rel[kMaxRing];        // warps done with the stage's current fill
    uint32_t cnt[kMaxRbSlots];     // warps that stored their partials of a block
    uint32_t gen[kMaxRbSlots];     // blocks finished in each partial-sum slot
    uint32_t abort_flag;
    uint32_t issued;               // stages issued so far
    int nstages;
    MatS mats[kMaxGemvMats];
    int q_end[kMaxGemvMats];       // q0 of the next matrix (nstages for the last)
};
static_assert(sizeof(Header) <= kHeader, "header does not fit");

// Stage q of this CTA: matrix, matrix-local row block, slice.
__device__ __forceinline__ void stage_coords(const Header &h, int count, int q, int &m, int &rb, int &ks) {
    m = 0;
    while (m + 1 < count && q >= h.q_end[m]) ++m;
    const int local = q - h.mats[m].q0;
    const int nks = h.mats[m].nks;
    const int rbl = local / nks;
    rb = h.mats[m].rb0 + rbl;
    ks = local - rbl * nks;
}

// Issue the TMA copies of stage q into its ring slot (one thread).
// Geometry a stage copy needs, from the shared-memory table or straight from
// the kernel parameters (the first copy is issued before the table exists).
struct Geom {
    int K, log2g, nlb, G, n, zbytes;
    const __half *scales;
    const uint8_t *zeros;
};

__device__ __forceinline__ Geom geom_of(const MatS &M) {
    return Geom{M.K, M.log2g, M.nlb, M.G, M.n, M.zbytes, M.scales, M.zeros};
}

__device__ __forceinline__ Geom geom_of(const GemvMat &M) {
    return Geom{(int)M.k, M.log2g, M.nlb, M.G, (int)M.n, M.zbytes, M.scales, M.zeros};
}

// Issue the TMA copies of one stage (matrix m, matrix-local row block rb,
// slice ks) into ring slot `slot` (one thread).
template <int BITS, int KIND>
__device__ void issue_geom(const GemvMulti &a, const Geom &M, int m, uint32_t bar, uint32_t base, int rb, int ks) {
    const int row0 = rb * kRows;
    uint32_t tx = 0;
    int ncb = 0;
    if (BITS == 3) {
        tx += 3 * kBox;
    } else {
        const int rowb = M.K / 2;
        for (int j = 0; j < 4; ++j)
            if (ks * 512 + 128 * j < rowb) ++ncb;
        tx += ncb * kBox;
    }
    int nlb = 0;
    if (KIND == 1) {
        const int gps = kSliceK >> M.log2g;  // groups per slice
        for (int b = 0; b < M.nlb; ++b)
            if (ks * gps + 8 * b < M.G) ++nlb;
        tx += nlb * kBox;
    }
    mbar_arrive_expect_tx(bar, tx);
    const CUtensorMap *tc = &a.tm_codes[m];
    if (BITS == 3) {
        tma_3d(base, tc, bar, ks * 128, 0, row0);
    } else {
        for (int j = 0; j < ncb; ++j) tma_2d(base + j * kBox, tc, bar, ks * 512 + 128 * j, row0);
    }
    if (KIND == 1) {
        const CUtensorMap *tl = &a.tm_luts[m];
        const int gps = kSliceK >> M.log2g;
        const uint32_t lbase = base + 3 * kBox;
        for (int b = 0; b < nlb; ++b) tma_2d(lbase + b * kBox, tl, bar, (ks * gps + 8 * b) * 16, row0);
    } else if (ks == 0) {
        // pull this block's scales and zero-points into L2; the lanes read
        // them from there a stage ahead of use
        const int rows = min(kRows, M.n - row0);
        const uint32_t sb = (uint32_t)(rows * M.G * 2) & ~15u;
        const uint32_t zb = (uint32_t)(rows * M.zbytes) & ~15u;
        if (sb) prefetch_l2_bulk(M.scales + (int64_t)row0 * M.G, sb);
        if (zb) prefetch_l2_bulk(M.zeros + (int64_t)row0 * M.zbytes, zb);
    }
}

template <int BITS, int KIND>
__device__ __forceinline__ void issue_at(const GemvMulti &a, Header &h, uint32_t ring_s, int m, int rb, int ks,
                                         int slot) {
    issue_geom<BITS, KIND>(a, geom_of(h.mats[m]), m, smem_u32(&h.full[slot]),
                           ring_s + (uint32_t)(slot * a.stage_bytes), rb, ks);
}

// Issue stage q (set-up path: coordinates from the stage number).
template <int BITS, int KIND>
__device__ void issue_stage(const GemvMulti &a, Header &h, uint32_t ring_s, int q) {
    int m, rb, ks;
    stage_coords(h, a.count, q, m, rb, ks);
    issue_at<BITS, KIND>(a, h, ring_s, m, rb, ks, q % a.ring);
}

// Scales and zero-points of one lane's 256-weight part: up to eight fp16
// scales and eight 4-bit zero-points (group order, lowest first).
struct Meta {
    uint32_t s0, s1, s2, s3;  // scales 0-1, 2-3, 4-5, 6-7
    uint32_t z;
};

__device__ __forceinline__ Meta load_meta(const MatS &M, int row, int k0) {
    Meta t{0u, 0u, 0u, 0u, 0u};
    if (row >= M.n || k0 >= M.K) return t;
    const int g0 = k0 >> M.log2g;
    // groups in the part, within the row (a part may run past k: then only
    // its first half is valid)
    const int ng = min(M.log2g >= 8 ? 1 : kPartK >> M.log2g, M.G - g0);
    const unsigned short *sp = reinterpret_cast<const unsigned short *>(M.scales) + (int64_t)row * M.G + g0;
    const uint8_t *zp = M.zeros + (int64_t)row * M.zbytes;
    uint32_t s[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        if (j < ng) {
            s[j >> 1] |= (uint32_t)sp[j] << ((j & 1) * 16);
            t.z |= (((uint32_t)zp[(g0 + j) >> 1] >> (((g0 + j) & 1) * 4)) & 15u) << (4 * j);
        }
    }
    t.s0 = s[0];
    t.s1 = s[1];
    t.s2 = s[2];
    t.s3 = s[3];
    return t;
}

__device__ __forceinline__ float meta_scale(const Meta &t, int gl) {
    uint32_t w = t.s0;
    if (gl >= 2) w = t.s1;
    if (gl >= 4) w = t.s2;
    if (gl >= 6) w = t.s3;
    return __half2float(__ushort_as_half((unsigned short)(w >> ((gl & 1) * 16))));
}

__device__ __forceinline__ uint32_t meta_zero(const Meta &t, int gl) { return (t.z >> (4 * gl)) & 15u; }

// Row blocks of matrix m in this CTA's range [lo, hi) of the launch's list.
__device__ __forceinline__ int cta_nrb(const GemvMulti &a, int m, int lo, int hi) {
    const int f = max(lo, a.mat[m].rb_off), e = min(hi, a.mat[m].rb_off + a.mat[m].nrb);
    return e > f ? e - f : 0;
}

// Matrix m is the first matrix of this CTA with its activations: it owns
// their shared-memory copy (matrices of a launch may share one x).
__device__ __forceinline__ bool x_owner_p(const GemvMulti &a, int m, int lo, int hi) {
    if (cta_nrb(a, m, lo, hi) == 0) return false;
    for (int j = 0; j < m; ++j)
        if (cta_nrb(a, j, lo, hi) > 0 && a.mat[j].x == a.mat[m].x && a.mat[j].k == a.mat[m].k) return false;
    return true;
}

// Offset (halves) of matrix m's activations in the shared-memory copy.
template <int NB>
__device__ __forceinline__ int x_offset(const GemvMulti &a, int m, int lo, int hi) {
    int off = 0;
    for (int j = 0; j < m; ++j) {
        if (!x_owner_p(a, j, lo, hi)) continue;
        if (a.mat[j].x == a.mat[m].x && a.mat[j].k == a.mat[m].k) return off;
        off += NB * (int)a.mat[j].k;
    }
    return off;
}

// Cursor over one warp's stages: matrix, CTA-local row block of that matrix,
// slice, and the CTA-local stage number.
struct Cursor {
    int m, rbl, ks, q;
};

__device__ __forceinline__ void advance_by(const Header &h, int count, Cursor &c, int d) {
    c.q += d;
    c.ks += d;
    while (c.m < count && c.ks >= h.mats[c.m].nks) {
        c.ks -= h.mats[c.m].nks;
        if (++c.rbl == h.mats[c.m].nrb) {
            c.rbl = 0;
            ++c.m;
            while (c.m < count && h.mats[c.m].nrb == 0) ++c.m;
        }
    }
}

// Wait for a full-barrier phase: a try in line, the bounded loop out of line.
__device__ __forceinline__ bool wait_full(uint32_t bar, uint32_t par, uint64_t limit_ns,
                                          volatile uint32_t *abort_flag) {
    bool ok = mbar_try_wait(bar, par);
    if (!__all_sync(0xffffffffu, ok)) ok = __all_sync(0xffffffffu, mbar_wait(bar, par, limit_ns, abort_flag));
    return ok;
}

// One 3-bit superblock (128 k = four 32-weight units) of one row: codes words
// A/B/C, tables built TPS times (once per group), products with NB rows of x.
template <int KIND, int NB, int TPS>
__device__ __forceinline__ void superblock3(const uint4 &A, const uint4 &B, const uint4 &C, uint32_t lut_s,
                                            int lg0, int r, const Meta &meta, int gl0, uint32_t xk, int K,
                                            bool half_only, float (&acc)[NB]) {
    const uint32_t Aw[4] = {A.x, A.y, A.z, A.w};
    const uint32_t Bw[4] = {B.x, B.y, B.z, B.w};
    const uint32_t Cw[4] = {C.x, C.y, C.z, C.w};
    (void)half_only;
    Table8 tab{};
    float s = 1.0f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        // up to four rows of x are held at once (batch 8 takes them one by one)
        constexpr int XB = NB <= 4 ? NB : 1;
        __half2 xv[XB][16];
#pragma unroll
        for (int b = 0; b < XB; ++b) load_x32(xk + 2u * (uint32_t)(b * K + 32 * i), xv[b]);
        if (i % (4 / TPS) == 0) {
            const int t = i / (4 / TPS);
            if (KIND == 1) {
                const int lg = lg0 + t;
                const uint4 l = lds128(lut_s + (uint32_t)((lg >> 3) * kBox) + swz(r, lg & 7));
                tab = make_table8(l.x, l.y, l.z, l.w);
            } else {
                tab = table8_offsets(meta_zero(meta, gl0 + t));
                s = meta_scale(meta, gl0 + t);
            }
        }
        __half2 w[16];
        lookup_triple(tab, Aw[i], Bw[i], Cw[i], w);
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const __half2(&xb)[16] = xv[XB == NB ? b : 0];
            if (XB != NB && b > 0) load_x32(xk + 2u * (uint32_t)(b * K + 32 * i), xv[0]);
            if (KIND == 1)
                acc[b] += dot16(w, xb);
            else
                acc[b] += s * dot16(w, xb);
        }
    }
}

// Eight 4-bit units (256 k) of one row, UPG units per group.
template <int NB, int UPG>
__device__ __forceinline__ void part4(uint32_t cb, int r, const Meta &meta, uint32_t xk, int K, bool half_only,
                                      float (&acc)[NB]) {
    float s = 1.0f;
    __half2 zl{}, zh{};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        if (i == 4 && half_only) break;  // k is a multiple of 128, not of 256
        constexpr int XB = NB <= 4 ? NB : 1;
        __half2 xv[XB][16];
#pragma unroll
        for (int b = 0; b < XB; ++b) load_x32(xk + 2u * (uint32_t)(b * K + 32 * i), xv[b]);
        if (i % UPG == 0) {
            const int gl = i / UPG;
            const uint32_t z = meta_zero(meta, gl);
            zl = zlo_of(z);
            zh = zhi_of(z);
            s = meta_scale(meta, gl);
        }
        const uint4 cw = lds128(cb + swz(r, i));
        const uint32_t wd[4] = {cw.x, cw.y, cw.z, cw.w};
        __half2 w[16];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            __half2 o[4];
            unpack4_qz(wd[t], zl, zh, o);
#pragma unroll
            for (int u = 0; u < 4; ++u) w[4 * t + u] = o[u];
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const __half2(&xb)[16] = xv[XB == NB ? b : 0];
            if (XB != NB && b > 0) load_x32(xk + 2u * (uint32_t)(b * K + 32 * i), xv[0]);
            acc[b] += s * dot16(w, xb);
        }
    }
}

template <int BITS, int KIND, int NB>
__global__ void __launch_bounds__(kThreads, 1) gemv_kernel(const __grid_constant__ GemvMulti a) {
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment for the swizzled TMA boxes
    const uint32_t raw_s = smem_u32(smem_raw);
    const uint32_t base_s = (raw_s + 1023u) & ~1023u;
    uint8_t *base = smem_raw + (base_s - raw_s);
    Header &h = *reinterpret_cast<Header *>(base);
    float *red = reinterpret_cast<float *>(base + kHeader);
    __half *xs = reinterpret_cast<__half *>(base + kHeader + a.red_bytes);
    const uint32_t xs_s = base_s + (uint32_t)(kHeader + a.red_bytes);
    const uint32_t ring_s = base_s + (uint32_t)(kHeader + a.red_bytes + a.x_smem_bytes);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int count = a.count, ring = a.ring;

    // let the next kernel in the stream start streaming its own weights; it
    // still waits for this grid's completion before it reads activations
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    // ---- set-up from the kernel parameters, spread over threads, with a
    // single barrier before the main loop: the first copies start at once and
    // the activations are staged while the tables are built
    const int lo = a.cta_rb[blockIdx.x], hi = a.cta_rb[blockIdx.x + 1];
    if (warp == 0) {
        if (lane < count) {  // matrix `lane`: this CTA's row blocks, stage numbering, x offset
            const int t = lane;
            const GemvMat &G = a.mat[t];
            MatS &S = h.mats[t];
            const int f = max(lo, G.rb_off);
            S.zeros = G.zeros;
            S.scales = G.scales;
            S.x = G.x;
            S.y = G.y;
            S.n = (int)G.n;
            S.K = (int)G.k;
            S.G = G.G;
            S.zbytes = G.zbytes;
            S.log2g = G.log2g;
            S.nks = G.nks;
            S.nlb = G.nlb;
            S.rb0 = f - G.rb_off;
            S.nrb = cta_nrb(a, t, lo, hi);
            int q = 0, rbq = 0;
            for (int m = 0; m < t; ++m) {
                const int nr = cta_nrb(a, m, lo, hi);
                q += nr * a.mat[m].nks;
                rbq += nr;
            }
            S.q0 = q;
            S.rbq0 = rbq;
            h.q_end[t] = q + S.nrb * G.nks;
            S.xoff = x_offset<NB>(a, t, lo, hi);
        }
        if (lane == 0) {
            int q = 0;
            for (int m = 0; m < count; ++m) q += cta_nrb(a, m, lo, hi) * a.mat[m].nks;
            h.nstages = q;
        }
    } else if (warp == 1) {
        if (lane < count) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(&a.tm_codes[lane]) : "memory");
            if (KIND == 1) asm volatile("prefetch.tensormap [%0];" ::"l"(&a.tm_luts[lane]) : "memory");
        }
    } else if (warp == 2) {
        if (lane == 0) {
            for (int i = 0; i < ring; ++i) mbar_init(smem_u32(&h.full[i]), 1);
            h.abort_flag = 0;
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        __syncwarp();
        // the CTA's first stages straight from the parameters, one per lane, so
        // that their data is on the way while the rest of the set-up runs
        int q = 0;
        for (int m = 0; m < count; ++m) {
            const GemvMat &G = a.mat[m];
            const int nq = cta_nrb(a, m, lo, hi) * G.nks;
            if (lane < a.initial && lane >= q && lane < q + nq) {
                const int j = lane - q, rbl = j / G.nks, ks = j - rbl * G.nks;
                const int rb0 = max(lo, G.rb_off) - G.rb_off;
                issue_geom<BITS, KIND>(a, geom_of(G), m, smem_u32(&h.full[lane]),
                                       ring_s + (uint32_t)(lane * a.stage_bytes), rb0 + rbl, ks);
            }
            q += nq;
        }
        if (lane == 0) h.issued = (uint32_t)min(a.initial, q);
    } else if (threadIdx.x >= 96 && threadIdx.x < 96 + kMaxRing) {
        h.rel[threadIdx.x - 96] = 0;
    } else if (threadIdx.x >= 128 && threadIdx.x < 128 + kMaxRbSlots) {
        h.cnt[threadIdx.x - 128] = 0;
        h.gen[threadIdx.x - 128] = 0;
    }
    // activations -> shared memory (every lane of a warp then reads the same
    // address: a broadcast), after the previous kernel in the stream is done
    asm volatile("griddepcontrol.wait;" ::: "memory");
    for (int m = 0; m < count; ++m) {
        if (!x_owner_p(a, m, lo, hi)) continue;
        const int vecs = NB * (int)a.mat[m].k / 8;
        const uint4 *src = reinterpret_cast<const uint4 *>(a.mat[m].x);
        uint4 *dst = reinterpret_cast<uint4 *>(xs + x_offset<NB>(a, m, lo, hi));
        for (int i = threadIdx.x; i < vecs; i += kThreads) dst[i] = src[i];
    }
    __syncthreads();

    const int nst = h.nstages;
    const int r = lane;
    const int grp = warp / kGroupWarps;   // stages q with q % kGroups == grp
    const int part = warp % kGroupWarps;  // 256-weight part of each of those stages
    bool ok = true;

    // this warp's first stage, and the one after it
    Cursor c{0, 0, 0, 0};
    while (c.m < count && h.mats[c.m].nrb == 0) ++c.m;
    advance_by(h, count, c, grp);
    Cursor cn = c;
    advance_by(h, count, cn, kGroups);
    // the stage that refills this warp's current slot, q + ring: ring is a
    // multiple of kGroups, so it is one of this warp's own later stages
    Cursor cr = c;
    advance_by(h, count, cr, ring);
    // uniform metadata of this warp's stages, loaded one stage ahead
    Meta cur{}, nxt{};
    if (KIND == 0 && c.m < count)
        cur = load_meta(h.mats[c.m], (h.mats[c.m].rb0 + c.rbl) * kRows + r, c.ks * kSliceK + part * kPartK);

    // per-lane offsets of this warp's 3-bit code chunks in a stage (planes 0-2
    // of row r are box rows 3r..3r+2; superblocks 2 part and 2 part + 1)
    uint32_t co[2][3];
#pragma unroll
    for (int hb = 0; hb < 2; ++hb)
#pragma unroll
        for (int p = 0; p < 3; ++p) co[hb][p] = swz(3 * r + p, part * 2 + hb);

    float acc[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) acc[b] = 0.0f;
    int slot = grp, fm = -1, frbl = 0;
    uint32_t par = 0;

    // partials of row block (m, rbl) -> shared memory; the last contributor
    // sums them in a fixed order and writes y
    auto flush = [&](int m, int rbl) -> bool {
        const MatS &M = h.mats[m];
        const int rbi = M.rbq0 + rbl;
        const int rs = rbi % a.rb_slots;
        const uint32_t use = (uint32_t)(rbi / a.rb_slots);
        // the warp groups run independently: the slot's previous block must
        // have been summed before this warp overwrites its partials
        bool okf = true;
        if (lane == 0 && *reinterpret_cast<volatile uint32_t *>(&h.gen[rs]) != use)
            okf = wait_equal(&h.gen[rs], use, a.wait_limit_ns, &h.abort_flag);
        if (!__shfl_sync(0xffffffffu, okf, 0)) return false;
        float *rp = red + (size_t)rs * (kWarps * NB * 32);
#pragma unroll
        for (int b = 0; b < NB; ++b) rp[(warp * NB + b) * 32 + r] = acc[b];
        __syncwarp();
        const int ng = min(M.nks, kGroups);  // groups that worked on this block
        uint32_t fin = 0;
        if (lane == 0) {
            __threadfence_block();
            fin = atomicAdd(&h.cnt[rs], 1u) + 1u == (uint32_t)(ng * kGroupWarps);
            __threadfence_block();
        }
        fin = __shfl_sync(0xffffffffu, fin, 0);
        if (fin) {
            const int q0 = M.q0 + rbl * M.nks;  // the block's first stage
            const int row = (M.rb0 + rbl) * kRows + r;
            float v[NB];
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                v[b] = 0.0f;
                for (int j = 0; j < ng; ++j) {
                    const int g = (q0 + j) % kGroups;
#pragma unroll
                    for (int p = 0; p < kGroupWarps; ++p) v[b] += rp[((g * kGroupWarps + p) * NB + b) * 32 + r];
                }
            }
            // free the slot first: the fence must not wait for the y stores
            __syncwarp();
            if (lane == 0) {
                h.cnt[rs] = 0;
                __threadfence_block();
                *reinterpret_cast<volatile uint32_t *>(&h.gen[rs]) = use + 1u;
            }
            if (row < M.n) {
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                    if (a.y_f32)
                        reinterpret_cast<float *>(M.y)[(int64_t)b * M.n + row] = v[b];
                    else
                        reinterpret_cast<__half *>(M.y)[(int64_t)b * M.n + row] = __float2half_rn(v[b]);
                }
            }
        }
        return true;
    };

    while (c.m < count) {
        const MatS &M = h.mats[c.m];
        if (fm >= 0 && (fm != c.m || frbl != c.rbl)) {  // left the previous row block
            ok = flush(fm, frbl);
            if (!ok) break;
#pragma unroll
            for (int b = 0; b < NB; ++b) acc[b] = 0.0f;
        }
        fm = c.m;
        frbl = c.rbl;
        if (KIND == 0 && cn.m < count) {
            const MatS &N = h.mats[cn.m];
            nxt = load_meta(N, (N.rb0 + cn.rbl) * kRows + r, cn.ks * kSliceK + part * kPartK);
        }
        ok = wait_full(smem_u32(&h.full[slot]), par, a.wait_limit_ns, &h.abort_flag);
        if (!ok) break;
        const int q = c.q;
        if (part == 0 && lane == 0 && q + a.initial < min(ring, nst)) {
            // ramp-up: a stage has landed, request one more of the ring
            issue_stage<BITS, KIND>(a, h, ring_s, q + a.initial);
            atomicMax(&h.issued, (uint32_t)(q + a.initial + 1));
        }
        const int K = M.K;
        const int k0 = c.ks * kSliceK + part * kPartK;
        if (k0 < K) {
            const uint32_t sb = ring_s + (uint32_t)(slot * a.stage_bytes);
            const uint32_t xk = xs_s + 2u * (uint32_t)(M.xoff + k0);
            const bool half_only = k0 + 128 >= K;  // k is a multiple of 128, not of 256
            const int log2g = M.log2g;
            if (BITS == 3) {
                const uint32_t lut_s = sb + 3 * kBox;
#pragma unroll
                for (int hb = 0; hb < 2; ++hb) {
                    if (hb == 1 && half_only) break;
                    const uint4 A = lds128(sb + co[hb][0]);
                    const uint4 B = lds128(sb + co[hb][1]);
                    const uint4 C = lds128(sb + co[hb][2]);
                    const int kk = part * kPartK + 128 * hb;  // within the slice
                    const int gl0 = (128 * hb) >> log2g;       // first group of the superblock in the part
                    const int lg0 = kk >> log2g;               // ... in the slice (LUT boxes)
                    if (log2g >= 7)
                        superblock3<KIND, NB, 1>(A, B, C, lut_s, lg0, r, cur, gl0, xk + 256u * hb, K, half_only, acc);
                    else if (log2g == 6)
                        superblock3<KIND, NB, 2>(A, B, C, lut_s, lg0, r, cur, gl0, xk + 256u * hb, K, half_only, acc);
                    else
                        superblock3<KIND, NB, 4>(A, B, C, lut_s, lg0, r, cur, gl0, xk + 256u * hb, K, half_only, acc);
                }
            } else {
                // 4-bit: box `part` holds this part's 256 k, 16 bytes per 32 k
                const uint32_t cb = sb + (uint32_t)(part * kBox);
                if (log2g >= 8)
                    part4<NB, 8>(cb, r, cur, xk, K, half_only, acc);
                else if (log2g == 7)
                    part4<NB, 4>(cb, r, cur, xk, K, half_only, acc);
                else if (log2g == 6)
                    part4<NB, 2>(cb, r, cur, xk, K, half_only, acc);
                else
                    part4<NB, 1>(cb, r, cur, xk, K, half_only, acc);
            }
        }
        // release the stage; the last warp of the group refills it
        __syncwarp();
        if (lane == 0) {
            __threadfence_block();
            const uint32_t old = atomicAdd(&h.rel[slot], 1u);
            if (old == kGroupWarps - 1) {
                h.rel[slot] = 0;
                __threadfence_block();
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                if (cr.m < count && !*reinterpret_cast<volatile uint32_t *>(&h.abort_flag)) {
                    issue_at<BITS, KIND>(a, h, ring_s, cr.m, h.mats[cr.m].rb0 + cr.rbl, cr.ks, slot);
                    atomicMax(&h.issued, (uint32_t)(q + ring + 1));
                }
            }
        }
        if (KIND == 0) cur = nxt;
        c = cn;
        advance_by(h, count, cn, kGroups);
        advance_by(h, count, cr, kGroups);
        slot += kGroups;
        if (slot >= ring) {
            slot -= ring;
            par ^= 1u;
        }
    }
    if (ok && fm >= 0) ok = flush(fm, frbl);
    if (!ok && lane == 0) {
        h.abort_flag = 1u;
        atomicOr(a.status, kStatusTimeout);
    }
    if (lane == 0 && (!ok || *reinterpret_cast<volatile uint32_t *>(&h.abort_flag))) {
        // a warp that gives up lets the copies still in flight land before
        // it exits, so the CTA's shared memory outlives them
        const int iss = (int)*reinterpret_cast<volatile uint32_t *>(&h.issued);
        for (int qq = max(0, iss - ring); qq < iss; ++qq)
            mbar_wait(smem_u32(&h.full[qq % ring]), (uint32_t)(qq / ring) & 1u, a.wait_limit_ns, nullptr);
    }
}

template <int BITS, int KIND, int NB>
cudaError_t launch_one(const GemvMulti &a, cudaStream_t st, bool pdl) {
    auto kern = gemv_kernel<BITS, KIND, NB>;
    static std::atomic<uint64_t> attrs_ready{0};
    cudaError_t e = ensure_kernel_attrs(reinterpret_cast<const void *>(kern), attrs_ready, true);
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

bool encode(CUtensorMap *map, const void *base, int rank, const cuuint64_t *dims, const cuuint64_t *strides,
            const cuuint32_t *box) {
    EncodeTiledFn enc = encode_fn();
    if (enc == nullptr) return false;
    const cuuint32_t estr[3] = {1, 1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, (cuuint32_t)rank, const_cast<void *>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

// Host-side plan: tensor maps, byte-balanced CTA row-block ranges and the
// shared-memory budget.  Returns false if the matrices cannot share one launch.
bool plan_gemv(GemvMulti &a, int num_sms) {
    const int bmax = a.batch;  // kernels are built for batch 1..4 exactly
    int nks_min = 1 << 30, nlb_max = 1;
    int64_t total = 0, rbs = 0;
    for (int m = 0; m < a.count; ++m) {
        GemvMat &M = a.mat[m];
        M.nks = (int)((M.k + kSliceK - 1) / kSliceK);
        M.nlb = a.kind == 1 ? std::max(1, 128 >> M.log2g) : 0;
        M.nrb = (int)((M.n + kRows - 1) / kRows);
        M.rb_off = (int)rbs;
        rbs += M.nrb;
        nks_min = std::min(nks_min, M.nks);
        nlb_max = std::max(nlb_max, M.nlb);
        if (M.n > (int64_t)1 << 30 || rbs > (int64_t)1 << 30) return false;
        const uint8_t *codes = M.codes;
        if (a.bits == 3) {
            // bytes within a plane, plane, row: box = [32 rows][3 planes][128 bytes]
            const cuuint64_t dims[3] = {(cuuint64_t)(M.k / 8), 3, (cuuint64_t)M.n};
            const cuuint64_t strides[2] = {(cuuint64_t)(M.k / 8), (cuuint64_t)(M.k * 3 / 8)};
            const cuuint32_t box[3] = {128, 3, kRows};
            if (!encode(&a.tm_codes[m], codes, 3, dims, strides, box)) return false;
        } else {
            const cuuint64_t dims[2] = {(cuuint64_t)(M.k / 2), (cuuint64_t)M.n};
            const cuuint64_t strides[1] = {(cuuint64_t)(M.k / 2)};
            const cuuint32_t box[2] = {128, kRows};
            if (!encode(&a.tm_codes[m], codes, 2, dims, strides, box)) return false;
        }
        if (a.kind == 1) {
            const cuuint64_t dims[2] = {(cuuint64_t)M.G * 16, (cuuint64_t)M.n};
            const cuuint64_t strides[1] = {(cuuint64_t)M.G * 16};
            const cuuint32_t box[2] = {128, kRows};
            if (!encode(&a.tm_luts[m], M.luts, 2, dims, strides, box)) return false;
        }
    }
    // bytes per row block (balancing only)
    int64_t rb_bytes[kMaxGemvMats];
    for (int m = 0; m < a.count; ++m) {
        const GemvMat &M = a.mat[m];
        const int64_t row = M.k * a.bits / 8 + (a.kind == 1 ? (int64_t)M.G * 16 : (int64_t)M.G * 2 + M.zbytes);
        rb_bytes[m] = row * kRows;
        total += rb_bytes[m] * M.nrb;
    }
    a.total_bytes = total;
    a.grid = (int)std::min<int64_t>(std::min(num_sms, kMaxGemvCtas), rbs);
    // CTA c owns the row blocks whose first byte lies in [c T / grid, (c+1) T / grid)
    for (int c = 0; c <= a.grid; ++c) {
        const int64_t b = (int64_t)((__int128)c * total / a.grid);
        int64_t acc = 0, r = rbs;
        for (int m = 0; m < a.count; ++m) {
            const GemvMat &M = a.mat[m];
            const int64_t mb = rb_bytes[m] * M.nrb;
            if (b < acc + mb) {
                r = M.rb_off + std::min<int64_t>((b - acc + rb_bytes[m] - 1) / rb_bytes[m], M.nrb);
                break;
            }
            acc += mb;
        }
        a.cta_rb[c] = (int32_t)r;
    }
    // activations of the matrices a CTA touches (one copy per distinct x)
    int64_t xmax = 0;
    for (int c = 0; c < a.grid; ++c) {
        int64_t xb = 0;
        for (int m = 0; m < a.count; ++m) {
            const GemvMat &M = a.mat[m];
            if (std::max<int64_t>(a.cta_rb[c], M.rb_off) >= std::min<int64_t>(a.cta_rb[c + 1], M.rb_off + M.nrb))
                continue;
            bool dup = false;
            for (int j = 0; j < m && !dup; ++j) {
                const GemvMat &P = a.mat[j];
                const bool touched =
                    std::max<int64_t>(a.cta_rb[c], P.rb_off) < std::min<int64_t>(a.cta_rb[c + 1], P.rb_off + P.nrb);
                dup = touched && P.x == M.x && P.k == M.k;
            }
            if (!dup) xb += (int64_t)a.batch * M.k * 2;
        }
        xmax = std::max(xmax, xb);
    }
    a.x_smem_bytes = (int)((xmax + 1023) / 1024 * 1024);  // the ring after it stays 1024-aligned
    a.stage_bytes = (a.bits == 3 ? 3 * kBox : 4 * kBox) + (a.kind == 1 ? nlb_max * kBox : 0);
    // The ring is a multiple of the number of warp groups, so that every
    // slot is only ever used by one group: a warp then never waits on a
    // barrier phase more than one ahead of the slot's current one.
    for (int ring = kMaxRing; ring >= kGroups; ring -= kGroups) {
        // partial-sum slots: any count is safe (a warp waits for the slot's
        // previous block); enough of them keep the warp groups from waiting
        const int slots = bmax > 4 ? 1 : std::min(kMaxRbSlots, (ring + nks_min - 1) / nks_min + 2);
        const int red = (slots * kWarps * bmax * 32 * 4 + 1023) / 1024 * 1024;
        const int smem = 1024 + kHeader + red + a.x_smem_bytes + ring * a.stage_bytes;
        if (smem <= kSmemBudget || ring == kGroups) {
            a.ring = ring;
            a.rb_slots = slots;
            a.red_bytes = red;
            a.smem_bytes = smem;
            break;
        }
    }
    return a.ring >= kGroups && a.smem_bytes <= 227 * 1024;
}

template <int BITS, int KIND>
cudaError_t launch_nb(const GemvMulti &a, cudaStream_t st, bool pdl) {
    switch (a.batch) {
        case 1: return launch_one<BITS, KIND, 1>(a, st, pdl);
        case 2: return launch_one<BITS, KIND, 2>(a, st, pdl);
        case 3: return launch_one<BITS, KIND, 3>(a, st, pdl);
        case 4: return launch_one<BITS, KIND, 4>(a, st, pdl);
        default: return launch_one<BITS, KIND, 8>(a, st, pdl);
    }
}

namespace {

// Failure-detection self-test: one thread waits, with the bounded mbarrier
// wait of the decode and prefill rings, for a phase that nothing completes
// (a barrier expecting one arrival that never comes).  The wait gives up after
// limit_ns; the kernel records the timeout in the device status word and
// returns, leaving the context usable.
__global__ void __launch_bounds__(32) wait_selftest_kernel(uint64_t limit_ns, uint32_t *status) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    if (threadIdx.x == 0 && !mbar_wait(smem_u32(&bar), 0, limit_ns, nullptr)) atomicOr(status, kStatusTimeout);
}

}  // namespace

cudaError_t launch_wait_selftest(uint64_t limit_ns, uint32_t *status, cudaStream_t st) {
    wait_selftest_kernel<<<1, 32, 0, st>>>(limit_ns, status);
    return cudaGetLastError();
}

cudaError_t launch_gemv_multi(GemvMulti &a, cudaStream_t st, bool pdl) {
    a.initial = pdl ? a.ring : kGroups;
    if (a.bits == 4) return launch_nb<4, 0>(a, st, pdl);
    if (a.kind == 1) return launch_nb<3, 1>(a, st, pdl);
    return launch_nb<3, 0>(a, st, pdl);
}

}  // namespace qx
