// Decode matmul y[b][n] = sum_k w_hat[n][k] x[b][k] for 1..16 rows of x, the
// weights dequantized in registers.
//
// Decoding reads every weight once per token, so it is bound by HBM bandwidth
// and by the cost of unpacking the codes (paper Section 2.4).  On GB300 the
// unpack of a 3-bit code through an 8-entry table costs about one byte-permute
// per weight on the integer pipe; everything else a weight needs is kept off
// that pipe and off the issue slots:
//
//   * Lane (g, t) = (lane / 4, lane % 4) of a warp takes the 32-weight unit t
//     of a 128-weight superblock for rows g and g + 8 of a 16-row tile.  Ten
//     code words per lane arrive by two ldmatrix instructions from the
//     128-byte swizzled TMA stage (free of bank conflicts), and the lane
//     decodes them in their natural order.
//   * Products: one or two rows of x on the CUDA cores (fp16 products summed
//     over 8 weight pairs per chain, then fp32); three or more on the tensor
//     cores, mma.sync m16n8k16 with the dequantized weights as A (16 rows x
//     16 k) and x as B (16 k x 8 rows of x), fp32 accumulation.  The order of
//     the contraction inside an MMA is free as long as A and B agree, so a
//     lane loads x for the same 32 k it decodes.  One MMA serves up to 8 rows
//     of x (two up to 16): a small batch costs the weight traffic of one.
//   * A stage of the shared-memory ring holds the codes (and LUTs) of 32 rows
//     x 1024 k.  Sixteen warps in two groups: group g takes the stages q with
//     q % 2 == g, and warp w of a group decodes superblock w of each of its
//     stages for both 16-row tiles (its x fragments serve both).
//   * A producer warp issues the copies, each once the eight warps of the
//     slot's group have released its previous fill (an mbarrier every lane
//     arrives at); waits suspend in hardware rather than spin.
//   * Partial sums of a row block stay in registers across its stages; at the
//     end of the block each warp stores its partials in a shared-memory slot
//     and arrives on the slot's barrier without waiting for anything.  A
//     reducer warp adds them in a fixed order (deterministic), writes y and
//     frees the slot, off the decoding warps' path.
//   * x is read from global memory (L1/L2): no per-launch staging.
//   * One launch may run several groups of matrices one after another
//     (qx_gemv_fused): the producer streams the weights of every group without
//     a break, and the consumers of group p + 1 read x only once every CTA's
//     reducer has counted group p done in a device-side counter.
// Every wait is bounded in time and reports QX_ERR_TIMEOUT through the device
// status.
#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int kWarps = 8;        // warps per group: warp w decodes superblock w of a stage
constexpr int kGroups = 2;       // group g takes the stages q with q % kGroups == g
constexpr int kProducer = kWarps * kGroups;  // the warp after the consumers issues the copies
constexpr int kReducer = kProducer + 1;      // the last warp sums each block's partials and writes y
constexpr int kThreads = 32 * (kWarps * kGroups + 2);
constexpr int kRows = 32;        // rows per block: two 16-row MMA tiles
constexpr int kSliceK = 1024;    // weights per row per stage: eight 128-weight superblocks
constexpr int kBox = kRows * 128;  // one 32-row x 128-byte TMA box
constexpr int kMaxRing = 12;
constexpr int kMaxRbSlots = 8;
constexpr int kHeader = 2048;    // barriers, counters, per-matrix and per-phase CTA plan
constexpr int kSmemBudget = 220 * 1024;
constexpr int kCoreBatch = 2;    // batches up to this take the CUDA-core products
constexpr int kQ4xTableBytes = 4 * 256 * 4;  // Q4X: a matrix's four books as 256-entry pair tables

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(b), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(b) : "memory");
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

// try_wait that lets the hardware suspend the warp until the phase completes
// (for at most about `hint_ns`): a waiting warp takes no issue slots from the
// warps that share its scheduler.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t b, uint32_t parity, uint32_t hint_ns) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(b), "r"(parity), "r"(hint_ns)
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
        if (mbar_try_wait_sleep(b, parity, 1000u)) return true;
        if (abort_flag != nullptr && *abort_flag) return false;
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

// ldmatrix (8x8 b16 matrices): lanes 8i..8i+7 give the row addresses of matrix
// i; lane (g, t) receives bytes 4t..4t+3 of row g of each matrix.
__device__ __forceinline__ void ldsm_x4(uint32_t a, uint32_t &d0, uint32_t &d1, uint32_t &d2, uint32_t &d3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(d0), "=r"(d1), "=r"(d2), "=r"(d3)
                 : "r"(a));
}

__device__ __forceinline__ void ldsm_x2(uint32_t a, uint32_t &d0, uint32_t &d1) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];" : "=r"(d0), "=r"(d1) : "r"(a));
}

// D += A B, m16n8k16, fp16 operands, fp32 accumulators.  Lane (g, t) holds
// a0 = A[g][2t..2t+1], a1 = A[g+8][2t..2t+1], a2 = A[g][2t+8..2t+9],
// a3 = A[g+8][2t+8..2t+9]; b0 = B[2t..2t+1][g], b1 = B[2t+8..2t+9][g];
// d = D[g][2t], D[g][2t+1], D[g+8][2t], D[g+8][2t+1].
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// 16 bytes of x: through the read-only path, or (fused launches, whose x may
// be written by an earlier phase of the same launch) as a plain load, which
// the phase handoff's acquire orders after those writes.
__device__ __forceinline__ uint4 ldg_x(const __half *p, bool written) {
    uint4 v;
    if (written)
        asm volatile("ld.global.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                     : "l"(p));
    else
        asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                     : "l"(p));
    return v;
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
    int q0;     // first CTA-local stage of this matrix
    int rb0;    // first matrix-local row block of this CTA
    int nrb;    // row blocks this CTA has stages of
    int ks_f;   // first slice of the first of them
    int ks_e;   // end slice of the last of them
    int st_off; // first stage of the matrix in its phase's list
};

// Slices [blo, bhi) this CTA takes of its row block rbl of M, and the
// CTA-local index qb of the first of them.
__device__ __forceinline__ void block_slices(const MatS &M, int rbl, int &blo, int &bhi, int &qb) {
    blo = rbl == 0 ? M.ks_f : 0;
    bhi = rbl == M.nrb - 1 ? M.ks_e : M.nks;
    qb = M.q0 + (rbl == 0 ? 0 : (M.nks - M.ks_f) + (rbl - 1) * M.nks);
}

struct Header {
    uint64_t full[kMaxRing];       // a stage's copies have landed
    uint64_t empty[kMaxRing];      // the eight warps of its group are done with it
    uint64_t rfull[kMaxRbSlots];   // every consumer lane has stored its partials of the slot's block
    uint64_t rempty[kMaxRbSlots];  // the reducer has summed the slot's block
    uint32_t abort_flag;
    int ph_q0[kMaxGemvPhases + 1];  // first CTA-local stage of each phase (multiples of kGroups)
    int ph_nst[kMaxGemvPhases];     // stages of each phase in this CTA (before the padding)
    MatS mats[kMaxGemvTotal];
};
static_assert(sizeof(Header) <= kHeader, "header does not fit");

// Geometry a stage copy needs, from the shared-memory table.
struct Geom {
    int K, log2g, nlb, G, n, zbytes;
    const __half *scales;
    const uint8_t *zeros;
};

__device__ __forceinline__ Geom geom_of(const MatS &M) {
    return Geom{M.K, M.log2g, M.nlb, M.G, M.n, M.zbytes, M.scales, M.zeros};
}


// Issue the TMA copies of one stage (matrix m, matrix-local row block rb,
// slice ks) into the ring slot at `base` with full barrier `bar` (one thread).
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
        const uint32_t lbase = base + (BITS == 3 ? 3 : 4) * kBox;
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

// Uniform scales and zero-points (Q4X: scales and codebook indices) of a
// lane's four rows (tile rows g, g + 8 of both 16-row tiles) for its 32-weight
// unit of a stage: scales as half2 pairs (rows g, g + 8) per tile,
// zero-points (book indices) in nibbles 0..3.
struct Meta {
    uint32_t s[2];
    uint32_t z;
};

template <int KIND>
__device__ __forceinline__ Meta load_meta(const MatS &M, int row0, int k0) {
    Meta t{{0u, 0u}, 0u};
    if (k0 >= M.K) return t;
    const int grp = k0 >> M.log2g;
    const unsigned short *sp = reinterpret_cast<const unsigned short *>(M.scales);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int row = row0 + 8 * i;  // g, g + 8, 16 + g, 24 + g
        if (row < M.n) {
            t.s[i >> 1] |= (uint32_t)__ldg(sp + (int64_t)row * M.G + grp) << ((i & 1) * 16);
            if (KIND == 2) {  // 2-bit book index of group grp: bits 2 (grp % 4) of byte grp / 4
                const uint32_t bb = __ldg(M.zeros + (int64_t)row * M.zbytes + (grp >> 2));
                t.z |= ((bb >> ((grp & 3) * 2)) & 3u) << (4 * i);
            } else {
                const uint32_t zb = __ldg(M.zeros + (int64_t)row * M.zbytes + (grp >> 1));
                t.z |= ((zb >> ((grp & 1) * 4)) & 15u) << (4 * i);
            }
        }
    }
    return t;
}

// Stages [f, f + return) of matrix m in this CTA's range [lo, hi) of its
// phase's list.
__device__ __forceinline__ int cta_mat_stages(const GemvMulti &a, int m, int lo, int hi, int &f) {
    const GemvMat &G = a.mat[m];
    f = max(lo, G.st_off);
    const int e = min(hi, G.st_off + G.nrb * G.nks);
    return e > f ? e - f : 0;
}

__device__ __forceinline__ int phase_of(const GemvMulti &a, int m) {
    int p = 0;
    while (p + 1 < a.nphase && m >= a.phase_first[p + 1]) ++p;
    return p;
}

// This CTA's stages of phase p.
__device__ __forceinline__ int phase_stages(const GemvMulti &a, int p) {
    return a.cta_st[p][blockIdx.x + 1] - a.cta_st[p][blockIdx.x];
}

// Pull the activations of phase p into L2 (lane i: matrix i of the phase).
// L2 is the point of coherence, so this is safe even when an earlier phase of
// the launch still writes them.
__device__ __forceinline__ void prefetch_x(const GemvMulti &a, int p, int lane) {
    if (p >= a.nphase) return;
    const int m = a.phase_first[p] + lane;
    if (m >= a.phase_first[p + 1]) return;
    const GemvMat &M = a.mat[m];
    const uint32_t bytes = (uint32_t)(a.batch * M.k * 2) & ~15u;
    if (bytes) prefetch_l2_bulk(M.x, bytes);
}

__device__ __forceinline__ int round_groups(int q) { return (q + kGroups - 1) / kGroups * kGroups; }

// Grid-scope counter of a fused launch: a release increment (everything the
// CTA wrote before it, ordered by the consumers' barrier, is visible to whoever
// acquires the new count) and an acquire read.
__device__ __forceinline__ uint32_t atom_add_release_gpu(uint32_t *p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.add.release.gpu.global.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

__device__ __forceinline__ void red_add_release_gpu(uint32_t *p, uint32_t v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void st_release_gpu(uint32_t *p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// y[b][row] of a block's 32 rows (lane = row within the block).
template <int VMAX>
__device__ __forceinline__ void store_y(const GemvMulti &a, const MatS &M, int row, const float (&v)[VMAX], int nb) {
    if (row >= M.n) return;
#pragma unroll
    for (int b = 0; b < VMAX; ++b) {
        if (b >= nb) break;
        if (a.y_f32)
            reinterpret_cast<float *>(M.y)[(int64_t)b * M.n + row] = v[b];
        else
            reinterpret_cast<__half *>(M.y)[(int64_t)b * M.n + row] = __float2half_rn(v[b]);
    }
}

// A row block whose slices are split between two consecutive CTAs (the plan
// never gives a block more than two).  The tail holder, for which the block is
// the first of its range and so among the first it finishes, stores its fp32
// sums and raises the block's flag (release); the head holder, for which the
// block is the last, fetches them (acquire, bounded wait) before its own part
// is summed, adds them after its own (slice order) and writes y.  Flags and
// sums are indexed by the tail holder's CTA; the head holder clears the flag.
constexpr int kSplitSlot = 16 * kRows;  // floats per CTA: [rows of x][32 rows]

template <int VMAX>
__device__ __forceinline__ void split_publish(const GemvMulti &a, const float (&v)[VMAX], int lane, int nb) {
    float *mine = a.split_part + (size_t)blockIdx.x * kSplitSlot + lane;
#pragma unroll
    for (int b = 0; b < VMAX; ++b)
        if (b < nb) __stcg(mine + b * kRows, v[b]);
    __syncwarp();
    if (lane == 0) st_release_gpu(a.split_flag + blockIdx.x, 1u);
}

template <int VMAX>
__device__ __forceinline__ bool split_fetch(const GemvMulti &a, float (&w)[VMAX], int lane, int nb,
                                            volatile uint32_t *abort_flag) {
    const int partner = blockIdx.x + 1;
    uint32_t ok = 1;
    if (lane == 0 && ld_acquire_gpu(a.split_flag + partner) == 0u) {
        const uint64_t t0 = globaltimer_ns();
        while (ld_acquire_gpu(a.split_flag + partner) == 0u) {
            __nanosleep(100);
            if (*abort_flag || globaltimer_ns() - t0 > a.wait_limit_ns) {
                ok = 0;
                break;
            }
        }
    }
    if (!__shfl_sync(0xffffffffu, ok, 0)) return false;
    __syncwarp();  // lane 0's acquire orders every lane's reads below
    const float *src = a.split_part + (size_t)partner * kSplitSlot + lane;
#pragma unroll
    for (int b = 0; b < VMAX; ++b) w[b] = b < nb ? __ldcg(src + b * kRows) : 0.0f;
    __syncwarp();
    if (lane == 0) a.split_flag[partner] = 0u;  // for the next launch (or phase)
    return true;
}

// Named barrier of the consumer warps (the producer and reducer warps do not
// take part).
__device__ __forceinline__ void consumers_sync() {
    asm volatile("bar.sync 1, %0;" ::"n"(32 * kWarps * kGroups) : "memory");
}

// Products of one 16-row tile's decoded weights with x.  NT = 1, 2: the
// tensor cores (mma.sync m16n8k16, 8 rows of x per n-tile).  NT = -1, -2: CUDA
// cores for one or two rows of x, where an MMA would waste most of its 8
// columns: fp16 products summed in fp16 over 8 weight pairs per chain, then in
// fp32 (the same products the MMA forms; `scaled` false means w holds q - z and
// the group's scale is applied to the fp32 sum).
template <int NT>
struct Dot {
    static constexpr bool kCores = NT < 0;
    static constexpr int NX = kCores ? -NT : NT;  // rows of x (CUDA cores) or n-tiles held
    __half2 h[NX][4];                             // CUDA cores: fp16 chains, rows g and g + 8
    __device__ __forceinline__ void start() {
        if (kCores) {
#pragma unroll
            for (int b = 0; b < NX; ++b)
#pragma unroll
                for (int i = 0; i < 4; ++i) h[b][i] = u2h2(0u);
        }
    }
    // weights (row g: p01 p23, row g + 8: r01 r23) of codes m = 4j .. 4j + 3
    __device__ __forceinline__ void step(int j, __half2 p01, __half2 p23, __half2 r01, __half2 r23,
                                         const uint32_t (&xw)[NX][16], int nb, float (&acc)[NX][4]) {
        if (kCores) {
#pragma unroll
            for (int b = 0; b < NX; ++b) {
                h[b][0] = __hfma2(p01, u2h2(xw[b][2 * j]), h[b][0]);
                h[b][1] = __hfma2(p23, u2h2(xw[b][2 * j + 1]), h[b][1]);
                h[b][2] = __hfma2(r01, u2h2(xw[b][2 * j]), h[b][2]);
                h[b][3] = __hfma2(r23, u2h2(xw[b][2 * j + 1]), h[b][3]);
            }
        } else {
#pragma unroll
            for (int nt = 0; nt < NX; ++nt)
                mma16816(acc[nt], h22u(p01), h22u(r01), h22u(p23), h22u(r23), xw[nt][2 * j], xw[nt][2 * j + 1]);
        }
    }
    // CUDA cores: the fp16 chains into the fp32 sums (times the scales s0, s1 of
    // rows g, g + 8 when the weights were q - z)
    __device__ __forceinline__ void finish(int nb, float s0, float s1, float (&acc)[NX][4]) {
        if (kCores) {
#pragma unroll
            for (int b = 0; b < NX; ++b) {
                const float2 f0 = __half22float2(h[b][0]), f1 = __half22float2(h[b][1]);
                const float2 f2 = __half22float2(h[b][2]), f3 = __half22float2(h[b][3]);
                acc[b][0] += s0 * ((f0.x + f0.y) + (f1.x + f1.y));
                acc[b][1] += s1 * ((f2.x + f2.y) + (f3.x + f3.y));
            }
        }
    }
};

// One 16-row tile, 3-bit codes: the lane's code words of rows g (A0 B0 C0) and
// g + 8 (A1 B1 C1) for its 32-weight unit, their 8-entry tables (a group's LUT,
// or the uniform offsets j - z with scales s0, s1), products with x.
template <int KIND, int NT>
__device__ __forceinline__ void tile3(const Table8 &t0, const Table8 &t1, uint32_t A0, uint32_t B0, uint32_t C0,
                                      uint32_t A1, uint32_t B1, uint32_t C1, __half2 s0, __half2 s1,
                                      const uint32_t (&xw)[Dot<NT>::NX][16], int nb,
                                      float (&acc)[Dot<NT>::NX][4]) {
    const uint32_t msk = 0x77777777u;
    uint32_t e0[4], e1[4];  // selectors of codes m = 8q + nibble
    e0[0] = A0 & msk;
    e0[1] = B0 & msk;
    e0[2] = C0 & msk;
    e0[3] = (shr_fma(A0, 3) & 0x11111111u) | (shr_fma(B0, 2) & 0x22222222u) | (shr_fma(C0, 1) & 0x44444444u);
    e1[0] = A1 & msk;
    e1[1] = B1 & msk;
    e1[2] = C1 & msk;
    e1[3] = (shr_fma(A1, 3) & 0x11111111u) | (shr_fma(B1, 2) & 0x22222222u) | (shr_fma(C1, 1) & 0x44444444u);
    Dot<NT> d;
    d.start();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {  // codes m = 8q + 4hh .. +3: step j = 2q + hh
            const uint32_t s0w = hh ? shr_fma(e0[q], 16) : e0[q];
            const uint32_t s1w = hh ? shr_fma(e1[q], 16) : e1[q];
            __half2 p01, p23, r01, r23;
            lookup4(t0, s0w, p01, p23);
            lookup4(t1, s1w, r01, r23);
            if (KIND == 0 && !Dot<NT>::kCores) {  // tensor cores: the dequantized weights themselves
                p01 = __hmul2(p01, s0);
                p23 = __hmul2(p23, s0);
                r01 = __hmul2(r01, s1);
                r23 = __hmul2(r23, s1);
            }
            d.step(2 * q + hh, p01, p23, r01, r23, xw, nb, acc);
        }
    }
    if (KIND == 0)
        d.finish(nb, __low2float(s0), __low2float(s1), acc);
    else
        d.finish(nb, 1.0f, 1.0f, acc);
}

// One 16-row tile, 4-bit uniform codes: the lane's 16 code bytes of rows g
// (c0) and g + 8 (c1), zero-point constants and scales, products with x.
template <int NT>
__device__ __forceinline__ void tile4(const uint4 &c0, const uint4 &c1, uint32_t z0, uint32_t z1, __half2 s0,
                                      __half2 s1, const uint32_t (&xw)[Dot<NT>::NX][16], int nb,
                                      float (&acc)[Dot<NT>::NX][4]) {
    const uint32_t w0[4] = {c0.x, c0.y, c0.z, c0.w};
    const uint32_t w1[4] = {c1.x, c1.y, c1.z, c1.w};
    const __half2 zl0 = zlo_of(z0), zh0 = zhi_of(z0), zl1 = zlo_of(z1), zh1 = zhi_of(z1);
    Dot<NT> d;
    d.start();
#pragma unroll
    for (int wd = 0; wd < 4; ++wd) {  // codes m = 8 wd .. 8 wd + 7: steps 2 wd, 2 wd + 1
        __half2 o0[4], o1[4];
        unpack4_qz(w0[wd], zl0, zh0, o0);
        unpack4_qz(w1[wd], zl1, zh1, o1);
        if (!Dot<NT>::kCores) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                o0[i] = __hmul2(o0[i], s0);
                o1[i] = __hmul2(o1[i], s1);
            }
        }
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
            d.step(2 * wd + hh, o0[2 * hh], o0[2 * hh + 1], o1[2 * hh], o1[2 * hh + 1], xw, nb, acc);
    }
    d.finish(nb, __low2float(s0), __low2float(s1), acc);
}

// Q4X (paper Section 3.2).  Byte j of code word w (k = 8t .. 8t + 7) holds the
// codes of a pair of k two apart: (8t, 8t + 2), (8t + 4, 8t + 6), (8t + 1,
// 8t + 3), (8t + 5, 8t + 7) for j = 0..3.  Each byte indexes the book's pair
// table (entry v holds CB[v % 16] and CB[v / 16]; tables are 1 KB-aligned, so
// the address is the table's OR'd with 4 v), and one fp16 multiply by the
// group's scale gives w_hat = fp16(s CB[b][q]) with the dequantization's single
// rounding.  x is re-paired the same way (x_pairs_q4x): the order of a dot
// product's terms, and of an MMA's contraction, is free as long as both
// operands follow it.
__device__ __forceinline__ uint32_t lds32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}

template <bool SCALED>
__device__ __forceinline__ void pairs_q4x(uint32_t w, uint32_t tab, __half2 s, __half2 (&o)[4]) {
    o[0] = u2h2(lds32(tab | ((w << 2) & 0x3FCu)));
    o[1] = u2h2(lds32(tab | (shr_fma(w, 6) & 0x3FCu)));
    o[2] = u2h2(lds32(tab | (shr_fma(w, 14) & 0x3FCu)));
    o[3] = u2h2(lds32(tab | (shr_fma(w, 22) & 0x3FCu)));
    if (SCALED) {
#pragma unroll
        for (int i = 0; i < 4; ++i) o[i] = __hmul2(o[i], s);
    }
}

// x words (x[k], x[k + 1]) of 8 k re-paired as the code bytes pair the
// weights: (x0, x2), (x4, x6), (x1, x3), (x5, x7).
template <int NX>
__device__ __forceinline__ void x_pairs_q4x(uint32_t (&xv)[NX][16]) {
#pragma unroll
    for (int nt = 0; nt < NX; ++nt)
#pragma unroll
        for (int wd = 0; wd < 4; ++wd) {
            const uint32_t x01 = xv[nt][4 * wd], x23 = xv[nt][4 * wd + 1];
            const uint32_t x45 = xv[nt][4 * wd + 2], x67 = xv[nt][4 * wd + 3];
            xv[nt][4 * wd] = prmt(x01, x23, 0x5410u);
            xv[nt][4 * wd + 1] = prmt(x45, x67, 0x5410u);
            xv[nt][4 * wd + 2] = prmt(x01, x23, 0x7632u);
            xv[nt][4 * wd + 3] = prmt(x45, x67, 0x7632u);
        }
}

// One 16-row tile, Q4X codes: the lane's 16 code bytes of rows g (c0) and
// g + 8 (c1), the shared addresses of their groups' pair tables and their
// scales.  Tensor cores: products with x of the dequantized weights
// themselves.  CUDA cores: products of the codebook levels (in [-1, 1]) with
// x, and the group's scale applied to their fp32 sum (a 32-weight unit lies in
// one 64-weight group), as the uniform kind does.
template <int NT>
__device__ __forceinline__ void tile4q(const uint4 &c0, const uint4 &c1, uint32_t tab0, uint32_t tab1, __half2 s0,
                                       __half2 s1, const uint32_t (&xw)[Dot<NT>::NX][16], int nb,
                                       float (&acc)[Dot<NT>::NX][4]) {
    const uint32_t w0[4] = {c0.x, c0.y, c0.z, c0.w};
    const uint32_t w1[4] = {c1.x, c1.y, c1.z, c1.w};
    Dot<NT> d;
    d.start();
#pragma unroll
    for (int wd = 0; wd < 4; ++wd) {  // codes m = 8 wd .. 8 wd + 7: steps 2 wd, 2 wd + 1
        __half2 o0[4], o1[4];
        pairs_q4x<!Dot<NT>::kCores>(w0[wd], tab0, s0, o0);
        pairs_q4x<!Dot<NT>::kCores>(w1[wd], tab1, s1, o1);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
            d.step(2 * wd + hh, o0[2 * hh], o0[2 * hh + 1], o1[2 * hh], o1[2 * hh + 1], xw, nb, acc);
    }
    d.finish(nb, __low2float(s0), __low2float(s1), acc);
}

// Row stride (floats) of a block's partial sums in shared memory.  CUDA-core
// path (one or two rows of x, scalar reads): odd, so that the finisher's
// lane-strided reads hit 32 different banks.  Tensor-core path (16-byte
// reads): 4 times an odd number, so that 8 lanes' 16-byte reads cover all 32
// banks.
__host__ __device__ __forceinline__ int partial_stride(int nb, bool cores) {
    if (cores) return nb | 1;
    const int r = (nb + 3) & ~3;
    return (r / 4) % 2 ? r : r + 4;
}

__device__ __forceinline__ __half2 half2_of(uint32_t pair, int hi) {
    const unsigned short v = (unsigned short)(hi ? pair >> 16 : pair);
    return __halves2half2(__ushort_as_half(v), __ushort_as_half(v));
}

template <int BITS, int KIND, int NT>
__global__ void __launch_bounds__(kThreads, 1) gemv_kernel(const __grid_constant__ GemvMulti a) {
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment for the swizzled TMA boxes
    const uint32_t raw_s = smem_u32(smem_raw);
    const uint32_t base_s = (raw_s + 1023u) & ~1023u;
    uint8_t *base = smem_raw + (base_s - raw_s);
    Header &h = *reinterpret_cast<Header *>(base);
    float *red = reinterpret_cast<float *>(base + kHeader);
    const uint32_t tab_s = base_s + (uint32_t)(kHeader + a.red_bytes);  // Q4X pair tables
    const uint32_t ring_s = tab_s + (uint32_t)a.tab_bytes;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int count = a.count, ring = a.ring, nb = a.batch;
    constexpr int NX = Dot<NT>::NX;

    // let the next kernel in the stream start streaming its own weights; it
    // still waits for this grid's completion before it reads activations
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    // ---- set-up from the kernel parameters, with a single barrier before
    // the main loops
    const bool fused = a.nphase > 1;
    if (warp == kProducer) {
        if (lane == 0) {
            for (int i = 0; i < ring; ++i) {
                mbar_init(smem_u32(&h.full[i]), 1);
                mbar_init(smem_u32(&h.empty[i]), 32 * kWarps);
            }
            for (int i = 0; i < a.rb_slots; ++i) {
                mbar_init(smem_u32(&h.rfull[i]), 32 * kWarps * kGroups);
                mbar_init(smem_u32(&h.rempty[i]), 32);
            }
            h.abort_flag = 0;
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        if (lane < count) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(&a.tm_codes[lane]) : "memory");
            if (KIND == 1) asm volatile("prefetch.tensormap [%0];" ::"l"(&a.tm_luts[lane]) : "memory");
        }
        prefetch_x(a, 0, lane);
    } else if (warp == 0) {
        if (lane < count) {  // matrix `lane`: this CTA's row blocks and stage numbering
            const int t = lane;
            const int p = phase_of(a, t);
            const int lo = a.cta_st[p][blockIdx.x], hi = a.cta_st[p][blockIdx.x + 1];
            const GemvMat &G = a.mat[t];
            MatS &S = h.mats[t];
            int f;
            const int ns = cta_mat_stages(a, t, lo, hi, f);
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
            S.st_off = G.st_off;
            if (ns > 0) {
                const int r = f - G.st_off, l = f + ns - 1 - G.st_off;
                S.rb0 = r / G.nks;
                S.ks_f = r % G.nks;
                S.nrb = l / G.nks - S.rb0 + 1;
                S.ks_e = l % G.nks + 1;
            } else {
                S.rb0 = S.nrb = S.ks_f = S.ks_e = 0;
            }
            // stages before this matrix: earlier phases (their stage counts
            // padded to a multiple of kGroups), then this phase's earlier matrices
            int q = 0;
            for (int pp = 0; pp < p; ++pp) q += round_groups(phase_stages(a, pp));
            for (int m = a.phase_first[p]; m < t; ++m) {
                int fm;
                q += cta_mat_stages(a, m, lo, hi, fm);
            }
            S.q0 = q;
        }
    } else if (warp == 1) {
        if (lane == 0) {
            int q = 0;
            for (int p = 0; p < a.nphase; ++p) {
                h.ph_q0[p] = q;
                h.ph_nst[p] = phase_stages(a, p);
                q += round_groups(h.ph_nst[p]);
            }
            h.ph_q0[a.nphase] = q;
        }
    }
    if (KIND == 2) {
        // every matrix's four books as pair tables: entry q0 + 16 q1 of book b
        // holds CB[b][q0] (low half) and CB[b][q1] (high half)
        uint32_t *tab = reinterpret_cast<uint32_t *>(base + kHeader + a.red_bytes);
        for (int e = threadIdx.x; e < count * (kQ4xTableBytes / 4); e += kThreads) {
            const unsigned short *cb =
                reinterpret_cast<const unsigned short *>(a.mat[e >> 10].luts) + ((e >> 8) & 3) * 16;
            tab[e] = (uint32_t)__ldg(cb + (e & 15)) | ((uint32_t)__ldg(cb + ((e >> 4) & 15)) << 16);
        }
    }
    __syncthreads();

    if (warp == kProducer) {
        // ---- producer: every stage in order, each once its slot's previous
        // fill has been released by the eight warps of its group; a phase's
        // stages are padded to a multiple of kGroups with empty stages (a full
        // barrier phase with no bytes), so that every phase starts on group 0
        // as a launch of its own does
        bool okp = true;
        int q = 0;
        for (int p = 0; p < a.nphase && okp; ++p) {
            prefetch_x(a, p + 1, lane);  // the next phase's activations, while this one streams
            if (lane == 0) {
                const int qend = h.ph_q0[p + 1];
                int m = a.phase_first[p], rbl = 0, ks = 0;
                while (m < a.phase_first[p + 1] && h.mats[m].nrb == 0) ++m;
                if (m < a.phase_first[p + 1]) ks = h.mats[m].ks_f;
                for (; q < qend; ++q) {
                    const int slot = q % ring;
                    if (q >= ring) {
                        okp = mbar_wait(smem_u32(&h.empty[slot]), (uint32_t)((q / ring) - 1) & 1u, a.wait_limit_ns,
                                        &h.abort_flag);
                        if (!okp) break;
                    }
                    if (m >= a.phase_first[p + 1]) {  // padding
                        mbar_arrive_expect_tx(smem_u32(&h.full[slot]), 0);
                        continue;
                    }
                    issue_at<BITS, KIND>(a, h, ring_s, m, h.mats[m].rb0 + rbl, ks, slot);
                    const int nrb = h.mats[m].nrb;
                    if (++ks == (rbl == nrb - 1 ? h.mats[m].ks_e : h.mats[m].nks)) {
                        ks = 0;
                        if (++rbl == nrb) {
                            rbl = 0;
                            ++m;
                            while (m < a.phase_first[p + 1] && h.mats[m].nrb == 0) ++m;
                            if (m < a.phase_first[p + 1]) ks = h.mats[m].ks_f;
                        }
                    }
                }
            }
            okp = __shfl_sync(0xffffffffu, okp, 0);
            q = __shfl_sync(0xffffffffu, q, 0);
        }
        if (lane == 0) {
            if (!okp) {
                h.abort_flag = 1u;
                atomicOr(a.status, kStatusTimeout);
            }
            // every issued copy lands before the CTA's shared memory is released
            for (int qq = max(0, q - ring); qq < q; ++qq)
                mbar_wait(smem_u32(&h.full[qq % ring]), (uint32_t)(qq / ring) & 1u, a.wait_limit_ns, nullptr);
        }
        return;
    }

    // x is read, and y written, only after the previous kernel in the stream
    // has finished
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int nbs = partial_stride(nb, Dot<NT>::kCores);  // row stride (floats) of the partial sums

    if (warp == kReducer) {
        // ---- reducer: the CTA's row blocks in order; lane i sums row i of a
        // block over the warps that worked on it, in a fixed order (group by the
        // block's stage order, then superblock warp), and writes y.  In a fused
        // launch it counts the CTA done with a phase once every y of the phase
        // is written.
        bool okr = true;
        int rs = 0;
        uint32_t use = 0;
        for (int p = 0; p < a.nphase && okr; ++p) {
            for (int m = a.phase_first[p]; m < a.phase_first[p + 1] && okr; ++m) {
                const MatS &M = h.mats[m];
                for (int rbl = 0; rbl < M.nrb; ++rbl) {
                    int blo, bhi, qb;
                    block_slices(M, rbl, blo, bhi, qb);
                    constexpr int VMAX = Dot<NT>::kCores ? 2 : 8 * NX;
                    // a block that goes on in the next CTA: fetch that CTA's sums
                    // while this CTA's warps still decode its own part
                    float w[VMAX];
                    if (bhi < M.nks && !split_fetch(a, w, lane, nb, &h.abort_flag)) {
                        okr = false;
                        break;
                    }
                    const uint32_t fb = smem_u32(&h.rfull[rs]);
                    if (!mbar_try_wait(fb, use & 1u) && !mbar_wait(fb, use & 1u, a.wait_limit_ns, &h.abort_flag)) {
                        okr = false;
                        break;
                    }
                    const float *rp = red + (size_t)rs * (kGroups * kWarps * kRows * nbs);
                    const int ng = min(bhi - blo, kGroups);  // groups that worked on the block
                    float v[VMAX];
#pragma unroll
                    for (int b = 0; b < VMAX; ++b) v[b] = 0.0f;
                    for (int j = 0; j < ng; ++j) {
                        const float *src = rp + (size_t)((qb + j) % kGroups * kWarps) * (kRows * nbs) + lane * nbs;
#pragma unroll
                        for (int w = 0; w < kWarps; ++w) {
                            const float *sw = src + (size_t)w * (kRows * nbs);
                            if (Dot<NT>::kCores) {
#pragma unroll
                                for (int b = 0; b < VMAX; ++b)
                                    if (b < nb) v[b] += sw[b];
                            } else {
#pragma unroll
                                for (int c4 = 0; c4 < VMAX / 4; ++c4) {
                                    if (4 * c4 < nb) {
                                        const float4 f = *reinterpret_cast<const float4 *>(sw + 4 * c4);
                                        v[4 * c4] += f.x;
                                        v[4 * c4 + 1] += f.y;
                                        v[4 * c4 + 2] += f.z;
                                        v[4 * c4 + 3] += f.w;
                                    }
                                }
                            }
                        }
                    }
                    // the slot is free once every lane has read it
                    mbar_arrive(smem_u32(&h.rempty[rs]));
                    if (blo > 0) {
                        split_publish(a, v, lane, nb);
                    } else {
                        if (bhi < M.nks) {
#pragma unroll
                            for (int b = 0; b < VMAX; ++b) v[b] += w[b];
                        }
                        store_y(a, M, (M.rb0 + rbl) * kRows + lane, v, nb);
                    }
                    if (++rs == a.rb_slots) {
                        rs = 0;
                        ++use;
                    }
                }
            }
            if (fused && okr) {
                // count the CTA in with a release (the warp barrier orders every
                // lane's y stores before it): whoever acquires the count sees them.
                // Before the last phase a reduction, which the warp does not wait
                // for; in the last one an atomic, whose old value tells the last
                // CTA of the launch
                __syncwarp();
                if (lane == 0) {
                    if (p < a.nphase - 1) {
                        red_add_release_gpu(a.phase_ctr + p, 1u);
                    } else if (atom_add_release_gpu(a.phase_ctr + p, 1u) == gridDim.x - 1) {
                        // every other CTA has passed every wait, so the counters
                        // go back to zero for the next launch
                        for (int i = 0; i < a.nphase; ++i) a.phase_ctr[i] = 0u;
                    }
                }
            }
        }
        if (!okr && lane == 0) {
            h.abort_flag = 1u;
            atomicOr(a.status, kStatusTimeout);
        }
        return;
    }

    // ---- consumers
    const int grp = warp / kWarps;   // stages q with q % kGroups == grp
    const int sb = warp % kWarps;    // superblock of each of those stages
    const int g = lane >> 2, t = lane & 3;
    const int kunit = 128 * sb + 32 * t;  // the lane's 32-weight unit within a slice
    bool ok = true;

    // per-lane shared-memory offsets of the code words of both tiles
    uint32_t co[2][2];
#pragma unroll
    for (int rt = 0; rt < 2; ++rt) {
        if (BITS == 3) {
            // ldmatrix.x4: planes 0, 1 of rows g and g + 8; ldmatrix.x2: plane 2
            const int mat = lane >> 3, rr = lane & 7;
            const int row4 = 16 * rt + 8 * (mat & 1) + rr, rho4 = 3 * row4 + (mat >> 1);
            const int row2 = 16 * rt + 8 * ((lane >> 3) & 1) + rr, rho2 = 3 * row2 + 2;
            co[rt][0] = swz(rho4, sb);
            co[rt][1] = swz(rho2, sb);
        } else {
            const int r0 = 16 * rt + g;
            const int chunk = 4 * (sb & 1) + t;
            co[rt][0] = (uint32_t)((sb >> 1) * kBox) + swz(r0, chunk);
            co[rt][1] = (uint32_t)((sb >> 1) * kBox) + swz(r0 + 8, chunk);
        }
    }

    int slot = grp;
    uint32_t par = 0;
    int blk_slot = 0;       // partial-sum slot of the CTA's next row block (blocks in CTA order)
    uint32_t blk_use = 0;   // uses of that slot before it
    float *rp_base = red;
    for (int p = 0; p < a.nphase; ++p) {
        if (fused && p > 0) {
            // phase p reads its x only once every CTA has finished phase p - 1
            if (threadIdx.x == 0 && ok && ld_acquire_gpu(a.phase_ctr + (p - 1)) < gridDim.x) {
                const uint64_t t0 = globaltimer_ns();
                while (ld_acquire_gpu(a.phase_ctr + (p - 1)) < gridDim.x) {
                    if (*reinterpret_cast<volatile uint32_t *>(&h.abort_flag) ||
                        globaltimer_ns() - t0 > a.wait_limit_ns) {
                        h.abort_flag = 1u;
                        atomicOr(a.status, kStatusTimeout);
                        break;
                    }
                }
            }
            consumers_sync();
            if (*reinterpret_cast<volatile uint32_t *>(&h.abort_flag)) ok = false;
        }
        for (int m = a.phase_first[p]; m < a.phase_first[p + 1] && ok; ++m) {
            const MatS &M = h.mats[m];
            const int nrb = M.nrb;
            if (nrb == 0) continue;
            const int K = M.K, nks = M.nks, n = M.n, log2g = M.log2g;
            const int q0 = M.q0, rb0 = M.rb0;
            const __half *xm = M.x;
            // the lane's LUT chunk in a stage (LUT kind): its group within the slice
            uint32_t lo_off[2][2] = {{0u, 0u}, {0u, 0u}};
            if (KIND == 1) {
                const int lg = kunit >> log2g;
#pragma unroll
                for (int rt = 0; rt < 2; ++rt) {
                    lo_off[rt][0] = (uint32_t)(3 * kBox + (lg >> 3) * kBox) + swz(16 * rt + g, lg & 7);
                    lo_off[rt][1] = (uint32_t)(3 * kBox + (lg >> 3) * kBox) + swz(16 * rt + g + 8, lg & 7);
                }
            }
            // x fragments of the lane's 32 k of slice ks: rows g (and g + 8) of x
            // the lane's rows of x at its unit of slice 0 (CUDA cores: every lane
            // takes every row of x; tensor cores: row g of each n-tile)
            const __half *xl[NX];
#pragma unroll
            for (int nt = 0; nt < NX; ++nt) {
                const int b = Dot<NT>::kCores ? nt : g + 8 * nt;
                xl[nt] = xm + (int64_t)min(b, nb - 1) * K + kunit;
            }
            auto load_x = [&](int ks, uint32_t (&xv)[NX][16]) {
                const bool in = ks * kSliceK + 128 * sb < K;
#pragma unroll
                for (int nt = 0; nt < NX; ++nt) {
                    const int b = Dot<NT>::kCores ? nt : g + 8 * nt;
                    if (in && b < nb) {
                        const __half *xp = xl[nt] + ks * kSliceK;
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const uint4 v = ldg_x(xp + 8 * i, fused);
                            xv[nt][4 * i + 0] = v.x;
                            xv[nt][4 * i + 1] = v.y;
                            xv[nt][4 * i + 2] = v.z;
                            xv[nt][4 * i + 3] = v.w;
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) xv[nt][i] = 0u;
                    }
                }
            };
            for (int rbl = 0; rbl < nrb && ok; ++rbl) {
                // the block's partial-sum slot, and how often the slot was used before
                const int rs = blk_slot;
                const uint32_t use = blk_use;
                if (++blk_slot == a.rb_slots) {
                    blk_slot = 0;
                    ++blk_use;
                }
                int blo, bhi, qb;  // the CTA's slices of the block, the first one's stage
                block_slices(M, rbl, blo, bhi, qb);
                const int ks0 = blo + (grp - qb % kGroups + kGroups) % kGroups;
                // ks0 >= bhi: this group has no stage of the block (it still hands
                // the block on below)
                const int row0 = (rb0 + rbl) * kRows + g;  // the lane's first row (of g, g + 8, g + 16, g + 24)
                float acc[2][NX][4];
#pragma unroll
                for (int rt = 0; rt < 2; ++rt)
#pragma unroll
                    for (int nt = 0; nt < NX; ++nt)
#pragma unroll
                        for (int i = 0; i < 4; ++i) acc[rt][nt][i] = 0.0f;
                Meta cur{};
                if (KIND != 1) cur = load_meta<KIND>(M, row0, ks0 * kSliceK + kunit);
                for (int ks = ks0; ks < bhi; ks += kGroups) {
                    Meta nxt{};
                    if (KIND != 1 && ks + kGroups < bhi) nxt = load_meta<KIND>(M, row0, (ks + kGroups) * kSliceK + kunit);
                    const bool live = ks * kSliceK + 128 * sb < K;  // K is a multiple of 128
                    uint32_t xw[NX][16];
                    load_x(ks, xw);
                    if (KIND == 2) x_pairs_q4x<NX>(xw);
                    const uint32_t fb = smem_u32(&h.full[slot]);
                    if (!mbar_try_wait(fb, par) && !mbar_wait(fb, par, a.wait_limit_ns, &h.abort_flag)) {
                        ok = false;
                        break;
                    }
                    if (live) {
                        const uint32_t sbase = ring_s + (uint32_t)(slot * a.stage_bytes);
#pragma unroll
                        for (int rt = 0; rt < 2; ++rt) {
                            if (BITS == 3) {
                                uint32_t A0, A1, B0, B1, C0, C1;
                                ldsm_x4(sbase + co[rt][0], A0, A1, B0, B1);
                                ldsm_x2(sbase + co[rt][1], C0, C1);
                                Table8 t0, t1;
                                __half2 s0 = u2h2(0u), s1 = s0;
                                if (KIND == 1) {
                                    const uint4 l0 = lds128(sbase + lo_off[rt][0]);
                                    const uint4 l1 = lds128(sbase + lo_off[rt][1]);
                                    t0 = make_table8(l0.x, l0.y, l0.z, l0.w);
                                    t1 = make_table8(l1.x, l1.y, l1.z, l1.w);
                                } else {
                                    t0 = table8_offsets((cur.z >> (8 * rt)) & 15u);
                                    t1 = table8_offsets((cur.z >> (8 * rt + 4)) & 15u);
                                    s0 = half2_of(cur.s[rt], 0);
                                    s1 = half2_of(cur.s[rt], 1);
                                }
                                tile3<KIND, NT>(t0, t1, A0, B0, C0, A1, B1, C1, s0, s1, xw, nb, acc[rt]);
                            } else {
                                const uint4 c0 = lds128(sbase + co[rt][0]);
                                const uint4 c1 = lds128(sbase + co[rt][1]);
                                if (KIND == 2) {
                                    // the pair tables of this matrix's books for rows g, g + 8
                                    const uint32_t tb = tab_s + (uint32_t)m * kQ4xTableBytes;
                                    tile4q<NT>(c0, c1, tb + ((cur.z >> (8 * rt)) & 3u) * 1024u,
                                               tb + ((cur.z >> (8 * rt + 4)) & 3u) * 1024u, half2_of(cur.s[rt], 0),
                                               half2_of(cur.s[rt], 1), xw, nb, acc[rt]);
                                } else {
                                    tile4<NT>(c0, c1, (cur.z >> (8 * rt)) & 15u, (cur.z >> (8 * rt + 4)) & 15u,
                                              half2_of(cur.s[rt], 0), half2_of(cur.s[rt], 1), xw, nb, acc[rt]);
                                }
                            }
                        }
                    }
                    // release the slot (every lane arrives: no warp-level sync needed)
                    mbar_arrive(smem_u32(&h.empty[slot]));
                    if (KIND != 1) cur = nxt;
                    slot += kGroups;
                    if (slot >= ring) {
                        slot -= ring;
                        par ^= 1u;
                    }
                }
                if (!ok) break;
                // ---- partials of this block -> shared memory, then to the
                // reducer warp; the slot's previous block must have been summed
                // before its partials are overwritten (every consumer lane
                // arrives for every block, with or without a stage of it)
                if (use > 0) {
                    const uint32_t eb = smem_u32(&h.rempty[rs]);
                    const uint32_t ep = (use - 1u) & 1u;
                    if (!mbar_try_wait(eb, ep) && !mbar_wait(eb, ep, a.wait_limit_ns, &h.abort_flag)) {
                        ok = false;
                        break;
                    }
                }
                if (ks0 < bhi) {
                    // slot layout: [group][superblock warp][32 rows][nbs]
                    float *mine = rp_base + (size_t)rs * (kGroups * kWarps * kRows * nbs) +
                                  (size_t)(grp * kWarps + sb) * (kRows * nbs);
                    if (Dot<NT>::kCores) {
                        // CUDA cores: sum the four lanes of a row (units t = 0..3), then lane t
                        // stores row of x t
#pragma unroll
                        for (int rt = 0; rt < 2; ++rt)
#pragma unroll
                            for (int b = 0; b < NX; ++b)
#pragma unroll
                                for (int r = 0; r < 2; ++r) {
                                    float v = acc[rt][b][r];
                                    v += __shfl_xor_sync(0xffffffffu, v, 1);
                                    v += __shfl_xor_sync(0xffffffffu, v, 2);
                                    if (t == b && b < nb) mine[(16 * rt + g + 8 * r) * nbs + b] = v;
                                }
                    } else {
#pragma unroll
                        for (int rt = 0; rt < 2; ++rt)
#pragma unroll
                            for (int nt = 0; nt < NX; ++nt) {
                                const int col = 8 * nt + 2 * t;
                                const int r0 = 16 * rt + g;
                                if (col < nb) {
                                    mine[r0 * nbs + col] = acc[rt][nt][0];
                                    mine[(r0 + 8) * nbs + col] = acc[rt][nt][2];
                                }
                                if (col + 1 < nb) {
                                    mine[r0 * nbs + col + 1] = acc[rt][nt][1];
                                    mine[(r0 + 8) * nbs + col + 1] = acc[rt][nt][3];
                                }
                            }
                    }
                }
                mbar_arrive(smem_u32(&h.rfull[rs]));
            }
        }
        // the padding stages of this phase that belong to this group
        for (int q = h.ph_q0[p] + h.ph_nst[p]; q < h.ph_q0[p + 1] && ok; ++q) {
            if (q % kGroups != grp) continue;
            const uint32_t fb = smem_u32(&h.full[slot]);
            if (!mbar_try_wait(fb, par) && !mbar_wait(fb, par, a.wait_limit_ns, &h.abort_flag)) {
                ok = false;
                break;
            }
            mbar_arrive(smem_u32(&h.empty[slot]));
            slot += kGroups;
            if (slot >= ring) {
                slot -= ring;
                par ^= 1u;
            }
        }
    }
    if (!ok && lane == 0) {
        h.abort_flag = 1u;
        atomicOr(a.status, kStatusTimeout);
    }
}

template <int BITS, int KIND, int NT>
cudaError_t launch_one(const GemvMulti &a, cudaStream_t st, bool pdl) {
    auto kern = gemv_kernel<BITS, KIND, NT>;
    static std::atomic<uint64_t> attrs_ready{0};
    cudaError_t e = ensure_kernel_attrs(reinterpret_cast<const void *>(kern), attrs_ready, true);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)a.grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = (size_t)a.smem_bytes;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    int na = 0;
    if (pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    if (a.nphase > 1 || a.has_split) {
        // the phases, or the two halves of a split row block, wait on one
        // another across CTAs: every CTA must be resident
        attr[na].id = cudaLaunchAttributeCooperative;
        attr[na].val.cooperative = 1;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = (unsigned)na;
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

// Host-side plan: tensor maps, byte-balanced CTA row-block ranges (per phase,
// exactly as a launch of that phase alone would have them) and the
// shared-memory budget.  Returns false if the matrices cannot share one launch.
bool plan_gemv(GemvMulti &a, int num_sms) {
    if (a.nphase < 1 || a.nphase > kMaxGemvPhases || a.count < 1 || a.count > kMaxGemvTotal) return false;
    if (a.phase_first[0] != 0 || a.phase_first[a.nphase] != a.count) return false;
    if (a.kind == 2 && (a.bits != 4 || a.count > kMaxGemvMats)) return false;
    int nks_min = 1 << 30, nlb_max = 1;
    for (int m = 0; m < a.count; ++m) {
        GemvMat &M = a.mat[m];
        M.nks = (int)((M.k + kSliceK - 1) / kSliceK);
        M.nlb = a.kind == 1 ? std::max(1, 128 >> M.log2g) : 0;
        M.nrb = (int)((M.n + kRows - 1) / kRows);
        nks_min = std::min(nks_min, M.nks);
        nlb_max = std::max(nlb_max, M.nlb);
        if (M.n > (int64_t)1 << 30) return false;
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
    a.total_bytes = 0;
    a.grid = 1;
    const bool split_ok = a.split_part != nullptr && a.split_flag != nullptr;
    a.has_split = 0;
    int grids[kMaxGemvPhases];
    for (int p = 0; p < a.nphase; ++p) {
        const int m0 = a.phase_first[p], m1 = a.phase_first[p + 1];
        if (m1 <= m0) return false;
        int64_t rbs = 0, nst = 0, total = 0;
        int64_t rb_bytes[kMaxGemvTotal];  // bytes per row block (balancing only)
        for (int m = m0; m < m1; ++m) {
            GemvMat &M = a.mat[m];
            M.rb_off = (int)rbs;
            M.st_off = (int)nst;
            rbs += M.nrb;
            nst += (int64_t)M.nrb * M.nks;
            const int64_t row = M.k * a.bits / 8 + (a.kind == 1 ? (int64_t)M.G * 16 : (int64_t)M.G * 2 + M.zbytes);
            rb_bytes[m] = row * kRows;
            total += rb_bytes[m] * M.nrb;
        }
        if (nst > (int64_t)1 << 30) return false;
        a.total_bytes += total;
        // CTA c's first stage: the first unit (a whole row block, or a stage)
        // that starts at or after byte c T / grid of the phase, in one pass
        auto partition = [&](bool by_stage, int grid, int32_t *cst) {
            cst[0] = 0;
            int c = 1;
            int64_t base = 0, st = 0;  // bytes before the current block, its first stage
            for (int m = m0; m < m1 && c < grid; ++m) {
                const GemvMat &M = a.mat[m];
                for (int rb = 0; rb < M.nrb && c < grid; ++rb, base += rb_bytes[m]) {
                    for (int ks = 0; ks < M.nks; ++ks, ++st) {
                        if (ks > 0 && !by_stage) continue;
                        // the stage's first byte (exact at block starts)
                        const int64_t off = base + rb_bytes[m] * ks * kSliceK / M.k;
                        while (c < grid && off >= (int64_t)((__int128)c * total / grid)) cst[c++] = (int32_t)st;
                    }
                }
            }
            while (c < grid) cst[c++] = (int32_t)nst;
            cst[grid] = (int32_t)nst;
        };
        int grid = (int)std::min<int64_t>(std::min(num_sms, kMaxGemvCtas), rbs);
        int32_t *cst = a.cta_st[p];
        partition(false, grid, cst);
        if (split_ok) {
            // by stages (a block's slices may go to two consecutive CTAs) when
            // that lowers the most stages a CTA has and no block would go to
            // three or more CTAs
            int32_t alt[kMaxGemvCtas + 1];
            const int g2 = (int)std::min<int64_t>(std::min(num_sms, kMaxGemvCtas), nst);
            partition(true, g2, alt);
            for (int i = 1; i < g2; ++i) alt[i] = std::max(alt[i], alt[i - 1] + 1);  // no empty CTA
            for (int i = g2 - 1; i >= 1; --i) alt[i] = std::min(alt[i], alt[i + 1] - 1);
            int most_w = 0, most_s = 0;
            for (int c = 0; c < grid; ++c) most_w = std::max(most_w, cst[c + 1] - cst[c]);
            for (int c = 0; c < g2; ++c) most_s = std::max(most_s, alt[c + 1] - alt[c]);
            // a CTA whose range starts and ends inside one block (not at its
            // edges) would make that block's third contributor
            bool two = true, any = false;
            for (int m = m0; m < m1 && two; ++m) {
                const GemvMat &M = a.mat[m];
                for (int c = 0; c < g2; ++c) {
                    const int lo = std::max(alt[c], M.st_off), hi = std::min(alt[c + 1], M.st_off + M.nrb * M.nks);
                    if (lo >= hi) continue;
                    const bool cut_lo = (lo - M.st_off) % M.nks != 0, cut_hi = (hi - M.st_off) % M.nks != 0;
                    any = any || cut_lo || cut_hi;
                    if (cut_lo && cut_hi && (lo - M.st_off) / M.nks == (hi - 1 - M.st_off) / M.nks) {
                        two = false;
                        break;
                    }
                }
            }
            if (two && most_s < most_w) {
                grid = g2;
                std::copy(alt, alt + g2 + 1, cst);
                a.has_split = a.has_split || any;
            }
        }
        grids[p] = grid;
        a.grid = std::max(a.grid, grid);
    }
    // CTAs beyond a phase's own grid have no stage of that phase
    for (int p = 0; p < a.nphase; ++p)
        for (int c = grids[p] + 1; c <= a.grid; ++c) a.cta_st[p][c] = a.cta_st[p][grids[p]];
    a.stage_bytes = (a.bits == 3 ? 3 * kBox : 4 * kBox) + (a.kind == 1 ? nlb_max * kBox : 0);
    a.tab_bytes = a.kind == 2 ? a.count * kQ4xTableBytes : 0;
    // The ring is a multiple of the number of warp groups, so that every
    // slot is only ever used by one group: a warp then never waits on a
    // barrier phase more than one ahead of the slot's current one.
    const int nbs = partial_stride(a.batch, a.batch <= kCoreBatch);
    const int slot_bytes = kGroups * kWarps * kRows * nbs * 4;
    for (int ring = kMaxRing; ring >= kGroups; ring -= kGroups) {
        // partial-sum slots: any count is safe (a warp waits for the slot's
        // previous block); enough of them keep the warp groups from waiting
        int slots = std::min(kMaxRbSlots, (ring + nks_min - 1) / nks_min + 2);
        while (slots > 2 && slots * slot_bytes > 48 * 1024) --slots;
        const int red = (slots * slot_bytes + 1023) / 1024 * 1024;
        const int smem = 1024 + kHeader + red + a.tab_bytes + ring * a.stage_bytes;
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

namespace {

template <int BITS, int KIND>
cudaError_t launch_nt(const GemvMulti &a, cudaStream_t st, bool pdl) {
    if (a.batch == 1) return launch_one<BITS, KIND, -1>(a, st, pdl);
    if (a.batch <= kCoreBatch) return launch_one<BITS, KIND, -2>(a, st, pdl);
    return a.batch <= 8 ? launch_one<BITS, KIND, 1>(a, st, pdl) : launch_one<BITS, KIND, 2>(a, st, pdl);
}

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
    if (a.kind == 2) return launch_nt<4, 2>(a, st, pdl);
    if (a.bits == 4) return launch_nt<4, 0>(a, st, pdl);
    if (a.kind == 1) return launch_nt<3, 1>(a, st, pdl);
    return launch_nt<3, 0>(a, st, pdl);
}

}  // namespace qx
