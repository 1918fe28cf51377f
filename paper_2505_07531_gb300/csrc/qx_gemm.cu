// Prefill matmul Y[m][n] = sum_k X[m][k] w_hat[n][k] on the 5th-generation
// tensor cores (tcgen05), with the weights dequantized on chip.
//
// Prefill is the one dense contraction on the path (paper Table 2, "Prefill"),
// so it runs on the tensor cores.  The kernel computes transposed tiles
// D = W_hat_tile * X_tile^T: the MMA's M dimension is 128 rows of W, its N
// dimension BN tokens, and the contraction runs over k in stages of 64.
// BN = 256 for prefill (each dequantized W tile feeds 256 tokens, which keeps
// the dequantization below the tensor-core time); BN = 16 for m <= 16, which
// makes the same kernel a decode matmul for batches of up to 16 tokens: the
// tensor cores then take the products, and the dequantization alone bounds
// the rate; BN = 64 (split-k calls only) for short prefills whose 256-token
// tiles would leave SMs idle.
//
// Persistent: one CTA per SM walks the work units -- (W-row tile, token tile,
// k split).  A tile is split along k (at 128-weight superblock boundaries)
// when the tiles alone would leave SMs idle, as a 4096-row decode matrix does
// (32 W tiles for 152 SMs); each split then stores its fp32 partial tile to a
// workspace, and the last of a tile's splits to finish sums them in split
// order (deterministic) and writes Y.  Warp roles (480 threads):
//   warp 0       TMA producer: BN x 64 fp16 X tiles (128B swizzle) -> smem
//   warp 1       allocates tensor memory; one thread issues tcgen05.mma
//   warps 2-9    dequantize 128 x 64 W_hat tiles from the packed codes straight
//                into the 128B-swizzled K-major shared-memory layout the MMA
//                reads (the same unpack primitives as qx_dequant, so W_hat is
//                exact)
//   warps 10-13  epilogue: fp32 accumulator (tensor memory) -> fp16 Y, or
//                the fp32 partial of a k split -> workspace
//   warp 14      TMA producer: packed codes (and LUTs) of 128-weight
//                superblocks -> a ring the dequant warps read a superblock ahead
// Two accumulators of BN columns let the epilogue of one unit overlap the
// main loop of the next.  An mbarrier ring connects producers and the MMA
// issuer; the MMA releases a stage with tcgen05.commit.  Every wait is
// bounded in time: a wait that gives up raises QX_ERR_TIMEOUT in the device
// status word, tells the other roles to stop, lets in-flight copies and MMAs
// drain, frees tensor memory and returns.
#include <cuda.h>

#include <mutex>

#include "qx_kernels.cuh"

namespace qx {

namespace {

constexpr int BM = 128;  // W rows per tile (MMA M)
constexpr int BK = 64;   // k per stage (one 128-byte swizzle row of fp16)
constexpr int A_BYTES = BM * BK * 2;
constexpr int NUM_DQ_WARPS = 8;
constexpr int NUM_EPI_WARPS = 4;
constexpr int PK_WARP = 2 + NUM_DQ_WARPS + NUM_EPI_WARPS;  // packed-code producer
constexpr int THREADS = (PK_WARP + 1) * 32;
constexpr int kMaxPSlots = 8;
constexpr int kMaxSplits = 16;

// Per token-tile constants.  X tiles (TMA) and dequantized W tiles use rings
// of STAGES and W_SLOTS slots tracked by the same per-stage barriers: the
// dequant warps know W slot q % W_SLOTS is free once the MMAs of stage
// q - W_SLOTS are done.  Equal depths measured best for BN = 256 (a deeper X
// ring at the cost of W slots lets the dequantization fall behind); the
// 2 KB and 8 KB X tiles of BN = 16 and 64 leave room for six.
template <int BN>
struct Cfg {
    static_assert(BN == 16 || BN == 64 || BN == 256, "token tile");
    static constexpr int STAGES = BN >= 128 ? 4 : 6;
    static constexpr int W_SLOTS = STAGES;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr uint32_t TMEM_COLS = 2 * BN < 32 ? 32 : 2 * BN;  // two accumulators
    // instruction descriptor, kind::f16: fp16 A and B, fp32 D, both K-major
    static constexpr uint32_t IDESC = (1u << 4)                        // D format f32
                                      | (0u << 7) | (0u << 10)          // A, B format f16
                                      | ((uint32_t)(BN >> 3) << 17)     // N
                                      | ((uint32_t)(BM >> 4) << 24);    // M
    static constexpr int CHUNK = BN < 32 ? BN : 32;  // accumulator columns per tcgen05.ld
};
static_assert(Cfg<256>::W_SLOTS <= Cfg<256>::STAGES && Cfg<64>::W_SLOTS <= Cfg<64>::STAGES &&
                  Cfg<16>::W_SLOTS <= Cfg<16>::STAGES,
              "a W slot's release is read from the stage barrier W_SLOTS back");

template <int BN>
struct SmemLayout {
    uint8_t a[Cfg<BN>::W_SLOTS][A_BYTES];
    uint8_t b[Cfg<BN>::STAGES][Cfg<BN>::B_BYTES];
    // one barrier per direction and stage: the MMA thread waits once and
    // commits once per stage (its per-stage overhead bounds the MMA rate)
    uint64_t full[Cfg<BN>::STAGES];   // 8 dequant-warp arrivals + the X copy's bytes
    uint64_t empty[Cfg<BN>::STAGES];  // tcgen05.commit of the stage's MMAs
    uint64_t accum_full[2];
    uint64_t accum_empty[2];
    uint64_t pfull[kMaxPSlots];   // a packed superblock has landed (TMA bytes)
    uint64_t pempty[kMaxPSlots];  // the 8 dequant warps have read it
    uint64_t done;
    uint32_t tmem_base;
    uint32_t abort_flag;
};

// The packed-code ring follows the layout (its size depends on the recipe).
template <int BN>
__host__ __device__ constexpr size_t layout_bytes() {
    return (sizeof(SmemLayout<BN>) + 1023) / 1024 * 1024;
}

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
// sleeps in hardware (woken when the phase completes) instead of spinning,
// which would take issue slots from the dequantizing warps that share its
// scheduler.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(b)), "r"(parity), "r"(1000000u)
        : "memory");
    return ok != 0;
}

// Wait for the phase of parity `parity` to complete.  Gives up after
// `limit_ns`, or as soon as another role has raised the abort flag (when
// `abort_flag` is not null).  Returns false if it gave up.
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

// Fast path in line (a phase that is already complete costs one try_wait),
// the bounded loop out of line.
__device__ __forceinline__ bool wait_phase(uint64_t *b, uint32_t parity, uint64_t limit_ns,
                                           volatile uint32_t *abort_flag) {
    return mbar_try_wait(b, parity) || mbar_wait(b, parity, limit_ns, abort_flag);
}

__device__ __forceinline__ void raise_abort(uint32_t *abort_flag, uint32_t *status) {
    *reinterpret_cast<volatile uint32_t *>(abort_flag) = 1u;
    atomicOr(status, kStatusTimeout);
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::
            "r"(smem_u32(dst)),
        "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(y)
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, uint64_t *bar, int x, int y, int z) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], "
        "[%2];" ::"r"(dst),
        "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z)
        : "memory");
}

__device__ __forceinline__ void tma_load_2d_s(uint32_t dst, const CUtensorMap *map, uint64_t *bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::
            "r"(dst),
        "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(y)
        : "memory");
}

__device__ __forceinline__ uint32_t lds32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}

__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row (1024-byte) swizzle atoms stacked along M/N.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
    d |= (uint64_t)1 << 16;                   // leading-dimension offset (unused here)
    d |= (uint64_t)(1024 >> 4) << 32;          // stride-dimension offset: 8 rows
    d |= (uint64_t)1 << 46;                   // descriptor version for tcgen05
    d |= (uint64_t)2 << 61;                   // 128-byte swizzle
    return d;
}

__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                        uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

template <int N>
__device__ __forceinline__ void tmem_ld(uint32_t taddr, uint32_t (&r)[N]) {
    static_assert(N == 16 || N == 32, "columns per load");
    if constexpr (N == 32)
        tmem_ld32(taddr, r);
    else
        tmem_ld16(taddr, r);
}

// k range of one work unit: tile t = u / splits, split s = u % splits takes
// superblocks [sb0, sb1) of the nsb in k (128 weights each), i.e. the
// 64-wide k blocks [2 sb0, 2 sb1).
struct Unit {
    int t, sb0, sb1;
};

__device__ __forceinline__ Unit unit_of(int u, int splits, int nsb) {
    const int t = u / splits, s = u - t * splits;
    return Unit{t, (int)((int64_t)s * nsb / splits), (int)((int64_t)(s + 1) * nsb / splits)};
}

// Codes and metadata one dequant thread needs for one 32-weight unit.
struct UnitRaw {
    uint32_t w[4];   // 4-bit: 16 bytes of codes; 3-bit: A, B, C of the triple
    uint4 lut;       // LUT entries (LUT kind)
    uint32_t zero;   // zero-point (uniform)
    __half scale;    // scale (uniform)
};

// Uniform metadata of one unit, from global memory (read ahead of use).
// Q4X (KIND 2): the group's fp16 scale and its 2-bit codebook index (books in
// `zeros`, four per byte, zbytes per row), held in u.scale and u.zero.
template <int KIND>
__device__ __forceinline__ void load_meta(const GemmArgs &a, int64_t row, int64_t k0, UnitRaw &u) {
    if (KIND == 0) {
        const int grp = (int)(k0 >> a.log2g);
        u.zero = zero_nibble(a.zeros + row * a.zbytes, grp);
        u.scale = a.scales[row * a.G + grp];
    } else if (KIND == 2) {
        const int grp = (int)(k0 >> a.log2g);
        u.zero = (a.zeros[row * a.zbytes + (grp >> 2)] >> (2 * (grp & 3))) & 3u;
        u.scale = a.scales[row * a.G + grp];
    }
}

// Codes (and the LUT) of one unit from the packed-code ring: slot `ps` holds
// one superblock of 128 rows -- 3-bit: [row][plane][16 bytes] then the LUTs
// [row][lut_box bytes]; 4-bit: [row][64 bytes].  u = unit in the superblock.
template <int BITS, int KIND>
__device__ __forceinline__ void read_codes(uint32_t ps, int r, int u, int gl, int lut_box, bool need_lut,
                                           UnitRaw &w) {
    if (BITS == 4) {
        const uint4 c = lds128(ps + (uint32_t)(r * 64 + 16 * u));
        w.w[0] = c.x;
        w.w[1] = c.y;
        w.w[2] = c.z;
        w.w[3] = c.w;
    } else {
        const uint32_t rc = ps + (uint32_t)(r * 48 + 4 * u);
        w.w[0] = lds32(rc);
        w.w[1] = lds32(rc + 16);
        w.w[2] = lds32(rc + 32);
        w.w[3] = 0;
        if (KIND == 1 && need_lut) w.lut = lds128(ps + (uint32_t)(BM * 48 + r * lut_box + 16 * gl));
    }
}

template <int BITS, int KIND>
__device__ __forceinline__ void dequant_unit(const UnitRaw &u, __half2 (&v)[16]) {
    if (BITS == 4) {
        const __half2 s2 = __halves2half2(u.scale, u.scale);
        const __half2 zl = zlo_of(u.zero), zh = zhi_of(u.zero);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            __half2 o[4];
            unpack4_qz(u.w[t], zl, zh, o);
#pragma unroll
            for (int p = 0; p < 4; ++p) v[4 * t + p] = __hmul2(o[p], s2);
        }
    } else if (KIND == 1) {
        const Table8 t = make_table8(u.lut.x, u.lut.y, u.lut.z, u.lut.w);
        lookup_triple(t, u.w[0], u.w[1], u.w[2], v);
    } else {
        const Table8 t = table8_offsets(u.zero);
        lookup_triple(t, u.w[0], u.w[1], u.w[2], v);
        const __half2 s2 = __halves2half2(u.scale, u.scale);
#pragma unroll
        for (int p = 0; p < 16; ++p) v[p] = __hmul2(v[p], s2);
    }
}

// Q4X unit: w_hat = codebook[book][q] * s in fp16 (the exact product rounded
// once, as the dequant defines), the four codebooks in shared memory at `cb`
// (128 bytes, one word per bank: any lookup pattern is conflict-free).
__device__ __forceinline__ void dequant_unit_q4x(const UnitRaw &u, const __half *cb, __half2 (&v)[16]) {
    const __half2 s2 = __halves2half2(u.scale, u.scale);
    const __half *tb = cb + 16 * u.zero;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t sel = (u.w[t] >> (4 * i)) & 0x000F000Fu;  // codes of k = 8t+2i, 8t+2i+1
            v[4 * t + i] = __hmul2(__halves2half2(tb[sel & 15u], tb[sel >> 16]), s2);
        }
    }
}

template <int BITS, int KIND, int BN>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ CUtensorMap tmap_c,
                const __grid_constant__ CUtensorMap tmap_l, const __grid_constant__ GemmArgs a) {
    using C = Cfg<BN>;
    constexpr int STAGES = C::STAGES;
    constexpr int W_SLOTS = C::W_SLOTS;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    SmemLayout<BN> &s = *reinterpret_cast<SmemLayout<BN> *>(base);
    const uint32_t pk_s = smem_u32(base + layout_bytes<BN>());  // packed-code ring
    // Q4X: the matrix's four codebooks (64 fp16) after the ring
    __half *q4x_cb = reinterpret_cast<__half *>(base + layout_bytes<BN>() + (size_t)a.pslots * a.pslot_bytes);
    volatile uint32_t *abort_flag = &s.abort_flag;
    uint32_t *abort_w = &s.abort_flag;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int nsb = (int)(a.k / 128);             // superblocks (two 64-k stages) in k
    const int mt = (int)((a.m + BN - 1) / BN);    // token tiles
    const int nt = (int)((a.n + BM - 1) / BM);    // W-row tiles
    const int S = a.splits;
    const int nunits = mt * nt * S;
    // unit u: tile t = u / S, W rows n0 = (t / mt) * BM, tokens m0 = (t % mt) * BN;
    // consecutive CTAs share a W tile (L2 reuse of the packed codes)

    // under programmatic dependent launch the next kernel in the stream may be
    // scheduled now: it waits for this one before it reads what this one writes
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(&s.full[i], NUM_DQ_WARPS + 1);
            mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s.accum_full[i], 1);
            mbar_init(&s.accum_empty[i], NUM_EPI_WARPS);
        }
        for (int i = 0; i < a.pslots; ++i) {
            mbar_init(&s.pfull[i], 1);
            mbar_init(&s.pempty[i], NUM_DQ_WARPS);
        }
        mbar_init(&s.done, 1);
        s.abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(&tmap_x) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(&tmap_c) : "memory");
        if (KIND == 1) asm volatile("prefetch.tensormap [%0];" ::"l"(&tmap_l) : "memory");
    }
    if (KIND == 2 && threadIdx.x >= 64 && threadIdx.x < 128) q4x_cb[threadIdx.x - 64] = a.luts[threadIdx.x - 64];
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(&s.tmem_base)),
                     "r"(C::TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_d = s.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer (X)
        if (lane == 0) {
            // X may be the previous kernel's output (a no-op without PDL)
            asm volatile("griddepcontrol.wait;" ::: "memory");
            int it = 0;  // stage counter across units
            bool ok = true;
            for (int u = blockIdx.x; u < nunits && ok; u += gridDim.x) {
                const Unit w = unit_of(u, S, nsb);
                const int m0 = (w.t % mt) * BN;
                for (int kb = 2 * w.sb0; kb < 2 * w.sb1; ++kb, ++it) {
                    const int st = it % STAGES;
                    const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
                    if (!wait_phase(&s.empty[st], ph ^ 1u, a.wait_limit_ns, abort_flag)) {
                        raise_abort(abort_w, a.status);
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&s.full[st], C::B_BYTES);
                    tma_load_2d(s.b[st], &tmap_x, &s.full[st], kb * BK, m0);
                }
            }
            // drain: never leave the CTA with a bulk copy still writing smem
            // (after an abort the dequant arrivals may be missing: the bounded
            // wait then outlasts the copies by far)
            for (int q = it - STAGES < 0 ? 0 : it - STAGES; q < it; ++q)
                mbar_wait(&s.full[q % STAGES], (uint32_t)(q / STAGES) & 1u, a.wait_limit_ns, nullptr);
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int it = 0, ti = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < nunits && ok; u += gridDim.x, ++ti) {
                const Unit w = unit_of(u, S, nsb);
                const int buf = ti & 1;
                const uint32_t dcol = tmem_d + (uint32_t)(buf * BN);
                if (ti >= 2 && !mbar_wait(&s.accum_empty[buf], (uint32_t)((ti >> 1) - 1) & 1u, a.wait_limit_ns,
                                          abort_flag)) {
                    raise_abort(abort_w, a.status);
                    break;
                }
                tc_fence_after();
                for (int kb = 2 * w.sb0; kb < 2 * w.sb1; ++kb, ++it) {
                    const int st = it % STAGES;
                    const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
                    if (!wait_phase(&s.full[st], ph, a.wait_limit_ns, abort_flag)) {
                        raise_abort(abort_w, a.status);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = sw128_desc(smem_u32(s.a[it % W_SLOTS]));
                    const uint64_t bd = sw128_desc(smem_u32(s.b[st]));
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)  // +32 bytes along k per step
                        mma_f16(dcol, ad + 2 * kk, bd + 2 * kk, C::IDESC, (kb > 2 * w.sb0 || kk > 0) ? 1u : 0u);
                    mma_commit(&s.empty[st]);
                }
                if (ok) mma_commit(&s.accum_full[buf]);
            }
            // do not free tensor memory under running MMAs: wait for them
            mma_commit(&s.done);
            mbar_wait(&s.done, 0, a.wait_limit_ns, nullptr);
        }
        __syncwarp();
    } else if (warp < 2 + NUM_DQ_WARPS) {
        // ------------------------------------------------ dequant producers
        const int d = threadIdx.x - 64;  // 0..255
        const int r = d >> 1;            // tile row 0..127
        const int half_id = d & 1;       // which 32-wide half of a stage
        const int P = a.pslots;
        int q = 0;                       // stage counter across units
        int sbi = 0;                     // superblock counter across units
        bool ok = true;
        // codes of one superblock for this thread: its unit of each of the two stages
        auto read_sb = [&](int sb_global, int sbl, int64_t row, UnitRaw (&w)[2]) -> bool {
            const int ps = sb_global % P;
            if (!wait_phase(&s.pfull[ps], (uint32_t)(sb_global / P) & 1u, a.wait_limit_ns, abort_flag)) return false;
            const uint32_t base_ps = pk_s + (uint32_t)(ps * a.pslot_bytes);
#pragma unroll
            for (int h2 = 0; h2 < 2; ++h2) {
                const int u = 2 * h2 + half_id;
                // with g >= 128 both units use the first unit's table
                read_codes<BITS, KIND>(base_ps, r, u, (32 * u) >> a.log2g, a.lut_box, h2 == 0 || a.log2g < 7, w[h2]);
                if (KIND != 1 && row < a.n) load_meta<KIND>(a, row, (int64_t)sbl * 128 + 32 * u, w[h2]);
            }
            // every lane has its codes in registers: release the slot
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.pempty[ps]);
            return true;
        };
        for (int u = blockIdx.x; u < nunits && ok; u += gridDim.x) {
            const Unit wu = unit_of(u, S, nsb);
            const int64_t row = (int64_t)(wu.t / mt) * BM + r;
            const bool valid = row < a.n;
            UnitRaw cur[2], nxt[2];
            ok = read_sb(sbi, wu.sb0, row, cur);
            for (int sbl = wu.sb0; sbl < wu.sb1 && ok; ++sbl, ++sbi) {
                // the next superblock's codes are read while this one is dequantized
                if (sbl + 1 < wu.sb1 && !read_sb(sbi + 1, sbl + 1, row, nxt)) {
                    raise_abort(abort_w, a.status);
                    ok = false;
                }
                // Both stages of the superblock: wait for both W slots, then
                // dequantize the two units as one block of independent work (the
                // two table lookups interleave: a dequant warp's latency, not the
                // ALU, bounds the producer rate), store both, then one proxy
                // fence (its cost is per fence, not per byte) and one arrival on
                // each stage's full barrier.  W slot (q + h2) % W_SLOTS is free
                // once the MMAs of stage q + h2 - W_SLOTS are done.
#pragma unroll
                for (int h2 = 0; h2 < 2; ++h2) {
                    const int qf = q + h2 - W_SLOTS;
                    if (ok && qf >= 0 &&
                        !wait_phase(&s.empty[qf % STAGES], (uint32_t)(qf / STAGES) & 1u, a.wait_limit_ns, abort_flag)) {
                        raise_abort(abort_w, a.status);
                        ok = false;
                    }
                }
                if (__any_sync(0xffffffffu, !ok)) {
                    ok = false;
                    break;
                }
                __half2 v[2][16];
                if (BITS == 3 && KIND == 1 && a.log2g >= 7) {
                    // one group spans the superblock: one table for both units
                    const Table8 t = make_table8(cur[0].lut.x, cur[0].lut.y, cur[0].lut.z, cur[0].lut.w);
#pragma unroll
                    for (int h2 = 0; h2 < 2; ++h2) lookup_triple(t, cur[h2].w[0], cur[h2].w[1], cur[h2].w[2], v[h2]);
                    if (!valid) {
#pragma unroll
                        for (int h2 = 0; h2 < 2; ++h2)
#pragma unroll
                            for (int p = 0; p < 16; ++p) v[h2][p] = __float2half2_rn(0.0f);
                    }
                } else {
#pragma unroll
                    for (int h2 = 0; h2 < 2; ++h2) {
                        if (valid) {
                            if constexpr (KIND == 2)
                                dequant_unit_q4x(cur[h2], q4x_cb, v[h2]);
                            else
                                dequant_unit<BITS, KIND>(cur[h2], v[h2]);
                        } else {
#pragma unroll
                            for (int p = 0; p < 16; ++p) v[h2][p] = __float2half2_rn(0.0f);
                        }
                    }
                }
#pragma unroll
                for (int h2 = 0; h2 < 2; ++h2) {
                    uint8_t *tile = s.a[(q + h2) % W_SLOTS] + (r >> 3) * 1024 + (r & 7) * 128;
#pragma unroll
                    for (int qq = 0; qq < 4; ++qq) {
                        const int chunk = 4 * half_id + qq;
                        *reinterpret_cast<uint4 *>(tile + ((chunk ^ (r & 7)) << 4)) =
                            make_uint4(h22u(v[h2][4 * qq]), h22u(v[h2][4 * qq + 1]), h22u(v[h2][4 * qq + 2]),
                                       h22u(v[h2][4 * qq + 3]));
                    }
                }
                if (!ok) break;
                fence_proxy_async_smem();  // generic-proxy writes -> visible to the tensor core
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&s.full[q % STAGES]);
                    mbar_arrive(&s.full[(q + 1) % STAGES]);
                }
                q += 2;
                cur[0] = nxt[0];
                cur[1] = nxt[1];
            }
            if (!ok) break;
        }
    } else if (warp == PK_WARP) {
        // ------------------------------------------------ TMA producer (packed codes)
        if (lane == 0) {
            const int P = a.pslots;
            const uint32_t bytes = (uint32_t)(BITS == 3 ? BM * 48 + (KIND == 1 ? BM * a.lut_box : 0) : BM * 64);
            int sbi = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < nunits && ok; u += gridDim.x) {
                const Unit w = unit_of(u, S, nsb);
                const int row0 = (w.t / mt) * BM;
                for (int sb = w.sb0; sb < w.sb1; ++sb, ++sbi) {
                    const int ps = sbi % P;
                    if (!wait_phase(&s.pempty[ps], ((uint32_t)(sbi / P) & 1u) ^ 1u, a.wait_limit_ns, abort_flag)) {
                        raise_abort(abort_w, a.status);
                        ok = false;
                        break;
                    }
                    const uint32_t dst = pk_s + (uint32_t)(ps * a.pslot_bytes);
                    mbar_arrive_expect_tx(&s.pfull[ps], bytes);
                    if (BITS == 3) {
                        tma_load_3d(dst, &tmap_c, &s.pfull[ps], sb * 16, 0, row0);
                        if (KIND == 1)
                            tma_load_2d_s(dst + BM * 48, &tmap_l, &s.pfull[ps], ((sb * 128) >> a.log2g) * 16, row0);
                    } else {
                        tma_load_2d_s(dst, &tmap_c, &s.pfull[ps], sb * 64, row0);
                    }
                }
            }
            // drain: never leave the CTA with a bulk copy still writing smem
            for (int q = sbi - P < 0 ? 0 : sbi - P; q < sbi; ++q)
                mbar_wait(&s.pfull[q % P], (uint32_t)(q / P) & 1u, a.wait_limit_ns, nullptr);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue
        // Y and the workspace may still be in use by the previous kernel
        asm volatile("griddepcontrol.wait;" ::: "memory");
        constexpr int CH = C::CHUNK;
        const int quarter = warp & 3;  // the TMEM lanes (W rows) this warp may read
        int ti = 0;
        for (int u = blockIdx.x; u < nunits; u += gridDim.x, ++ti) {
            const int t = u / S;
            const int buf = ti & 1;
            const bool have = mbar_wait(&s.accum_full[buf], (uint32_t)(ti >> 1) & 1u, a.wait_limit_ns, abort_flag);
            if (!have) raise_abort(abort_w, a.status);
            tc_fence_after();
            // tcgen05.ld is warp-collective: decide for the whole warp at once
            if (!__all_sync(0xffffffffu, have && !*abort_flag)) break;
            const int64_t n = (int64_t)(t / mt) * BM + 32 * quarter + lane;
            const int64_t m0 = (int64_t)(t % mt) * BN;
            // this unit's partial: [BN][BM] fp32, row n of the tile at column
            // 32 quarter + lane (a warp's stores are 128 contiguous bytes)
            float *part = S > 1 ? a.ws_part + (size_t)u * BN * BM + 32 * quarter + lane : nullptr;
#pragma unroll 1
            for (int c = 0; c < BN; c += CH) {
                uint32_t rv[CH];
                tmem_ld<CH>(tmem_d + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(buf * BN + c), rv);
                if (S > 1) {
#pragma unroll
                    for (int j = 0; j < CH; ++j) part[(size_t)(c + j) * BM] = __uint_as_float(rv[j]);
                } else if (n < a.n) {
#pragma unroll
                    for (int j = 0; j < CH; ++j) {
                        const int64_t m = m0 + c + j;
                        if (m < a.m) a.Y[m * a.n + n] = __float2half_rn(__uint_as_float(rv[j]));
                    }
                }
            }
            // this warp's rows of the accumulator are read: free it for unit ti + 2
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.accum_empty[buf]);
            if (S > 1) {
                // the last split of the tile to store its quarter sums all of
                // them in split order and writes Y, then re-arms the counter
                __threadfence();
                __syncwarp();
                uint32_t last = 0;
                if (lane == 0) last = atomicAdd(&a.ws_cnt[(size_t)t * 4 + quarter], 1u) == (uint32_t)(S - 1) ? 1u : 0u;
                last = __shfl_sync(0xffffffffu, last, 0);
                if (last) {
                    __threadfence();
                    const float *p0 = a.ws_part + (size_t)t * S * BN * BM + 32 * quarter + lane;
                    if (n < a.n) {
                        // a chunk of columns at a time, splits outer: the CH loads
                        // of one split are independent (one round trip to L2 per
                        // split, not per column); the sum order stays split order
#pragma unroll 1
                        for (int c = 0; c < BN; c += CH) {
                            float v[CH];
#pragma unroll
                            for (int j = 0; j < CH; ++j) v[j] = 0.0f;
#pragma unroll 1
                            for (int sp = 0; sp < S; ++sp) {
                                const float *ps = p0 + ((size_t)sp * BN + c) * BM;
#pragma unroll
                                for (int j = 0; j < CH; ++j) v[j] += __ldcg(ps + (size_t)j * BM);
                            }
#pragma unroll
                            for (int j = 0; j < CH; ++j) {
                                const int64_t m = m0 + c + j;
                                if (m < a.m) a.Y[m * a.n + n] = __float2half_rn(v[j]);
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) a.ws_cnt[(size_t)t * 4 + quarter] = 0u;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_d), "r"(C::TMEM_COLS)
                     : "memory");
    }
}

template <int BITS, int KIND, int BN>
cudaError_t launch_t(const CUtensorMap &mx, const CUtensorMap &mc, const CUtensorMap &ml, const GemmArgs &a,
                     int64_t units, int num_sms, cudaStream_t st) {
    auto kern = gemm_kernel<BITS, KIND, BN>;
    static std::atomic<uint64_t> attrs_ready{0};
    cudaError_t e = ensure_kernel_attrs(reinterpret_cast<const void *>(kern), attrs_ready, false);
    if (e != cudaSuccess) return e;
    const unsigned grid = (unsigned)std::min<int64_t>(units, num_sms);
    if (!a.pdl) {
        kern<<<grid, THREADS, a.smem_bytes, st>>>(mx, mc, ml, a);
        return cudaGetLastError();
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = (size_t)a.smem_bytes;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, mx, mc, ml, a);
}

template <int BITS, int KIND>
cudaError_t launch_bn(const CUtensorMap &mx, const CUtensorMap &mc, const CUtensorMap &ml, const GemmArgs &a,
                      int64_t units, int num_sms, cudaStream_t st) {
    if (a.bn == 16) return launch_t<BITS, KIND, 16>(mx, mc, ml, a, units, num_sms, st);
    if (a.bn == 64) return launch_t<BITS, KIND, 64>(mx, mc, ml, a, units, num_sms, st);
    return launch_t<BITS, KIND, 256>(mx, mc, ml, a, units, num_sms, st);
}

}  // namespace

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (fn == nullptr) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

GemmPlan plan_gemm(int64_t n, int64_t k, int64_t m, int num_sms, bool allow_split) {
    const int nsb = (int)(k / 128);
    const int64_t nt = (n + BM - 1) / BM;
    GemmPlan p{};
    p.bn = m <= 16 ? 16 : 256;
    p.splits = 1;
    p.tiles = ((m + p.bn - 1) / p.bn) * nt;
    if (allow_split && num_sms > 0) {
        // Time ~ rounds of units per CTA x (superblocks per unit + about two
        // for pipeline fill and epilogue), plus the last split's reduction:
        // per 32 columns about two superblocks of fixed cost (the counter's
        // round trip, the partial tiles' stores and loads) and half a
        // superblock per split -- fitted to 64-token tiles at 576 tokens,
        // where a 1024 x 1024 matrix took 9.9 us unsplit and 11.8 us in two
        // splits.  Decode sizes take 16-token tiles; longer inputs choose
        // between 64-token tiles, which may split k, and 256-token tiles.
        const int cands[2] = {m <= 16 ? 16 : 64, 256};
        double best = -1.0;
        for (int ci = 0; ci < (m <= 16 ? 1 : 2); ++ci) {
            const int bn = cands[ci];
            const int64_t tiles = ((m + bn - 1) / bn) * nt;
            const int smax = (bn == 256 || tiles > (int64_t)(kSplitCounterBytes / 16)) ? 1 : std::min(nsb, kMaxSplits);
            for (int sp = 1; sp <= smax; ++sp) {
                const int64_t rounds = (tiles * sp + num_sms - 1) / num_sms;
                const double cost = (double)rounds * ((nsb + sp - 1) / sp + 2) +
                                    (sp > 1 ? (2.0 + 0.5 * sp) * ((bn + 31) / 32) : 0.0);
                if (best < 0 || cost < best) {
                    best = cost;
                    p.bn = bn;
                    p.splits = sp;
                    p.tiles = tiles;
                }
            }
        }
    }
    p.units = p.tiles * p.splits;
    p.ws_bytes = p.splits > 1 ? kSplitCounterBytes + (size_t)p.units * p.bn * BM * sizeof(float) : 0;
    return p;
}

cudaError_t launch_gemm(const GemmArgs &args, int num_sms, cudaStream_t st) {
    EncodeTiledFn enc = encode_fn();
    if (enc == nullptr) return cudaErrorNotSupported;
    GemmArgs a = args;
    if (a.bn != 16 && a.bn != 64 && a.bn != 256) return cudaErrorInvalidValue;
    if (a.splits < 1 || a.splits > kMaxSplits || a.splits > a.k / 128) return cudaErrorInvalidValue;
    if (a.splits > 1 && (a.ws_part == nullptr || a.ws_cnt == nullptr)) return cudaErrorInvalidValue;
    const int64_t units = ((a.m + a.bn - 1) / a.bn) * ((a.n + BM - 1) / BM) * a.splits;
    if (units > ((int64_t)1 << 31) - 1) return cudaErrorInvalidValue;
    const cuuint32_t estr[3] = {1, 1, 1};
    CUtensorMap mx{}, mc{}, ml{};
    {
        const cuuint64_t dims[2] = {(cuuint64_t)a.k, (cuuint64_t)a.m};
        const cuuint64_t strides[1] = {(cuuint64_t)a.k * 2};
        const cuuint32_t box[2] = {BK, (cuuint32_t)a.bn};
        if (enc(&mx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half *>(a.X), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    // packed codes: one box = one 128-weight superblock of 128 rows
    if (a.bits == 3) {
        const cuuint64_t dims[3] = {(cuuint64_t)(a.k / 8), 3, (cuuint64_t)a.n};
        const cuuint64_t strides[2] = {(cuuint64_t)(a.k / 8), (cuuint64_t)(a.k * 3 / 8)};
        const cuuint32_t box[3] = {16, 3, BM};
        if (enc(&mc, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint8_t *>(a.codes), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    } else {
        const cuuint64_t dims[2] = {(cuuint64_t)(a.k / 2), (cuuint64_t)a.n};
        const cuuint64_t strides[1] = {(cuuint64_t)(a.k / 2)};
        const cuuint32_t box[2] = {64, BM};
        if (enc(&mc, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(a.codes), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    a.lut_box = 0;
    if (a.kind == 1) {
        // the LUTs of the groups one superblock spans (one group for g >= 128)
        a.lut_box = 16 * std::max(1, 128 >> a.log2g);
        const cuuint64_t dims[2] = {(cuuint64_t)a.G * 16, (cuuint64_t)a.n};
        const cuuint64_t strides[1] = {(cuuint64_t)a.G * 16};
        const cuuint32_t box[2] = {(cuuint32_t)a.lut_box, BM};
        if (enc(&ml, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<__half *>(a.luts), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    } else {
        ml = mc;  // unused
    }
    a.pslot_bytes = (a.bits == 3 ? BM * 48 + BM * a.lut_box : BM * 64 + 0);
    a.pslot_bytes = (a.pslot_bytes + 1023) / 1024 * 1024;
    const int layout = (int)(a.bn == 16 ? layout_bytes<16>() : a.bn == 64 ? layout_bytes<64>() : layout_bytes<256>());
    const int cb_bytes = a.kind == 2 ? 128 : 0;  // Q4X codebooks after the ring
    const int budget = 227 * 1024 - layout - 1024 - cb_bytes;
    a.pslots = std::min(kMaxPSlots, budget / a.pslot_bytes);
    if (a.pslots < 2) return cudaErrorInvalidConfiguration;
    a.smem_bytes = layout + 1024 + a.pslots * a.pslot_bytes + cb_bytes;
    if (a.bits == 4 && a.kind == 2) return launch_bn<4, 2>(mx, mc, ml, a, units, num_sms, st);
    if (a.bits == 4) return launch_bn<4, 0>(mx, mc, ml, a, units, num_sms, st);
    if (a.kind == 1) return launch_bn<3, 1>(mx, mc, ml, a, units, num_sms, st);
    return launch_bn<3, 0>(mx, mc, ml, a, units, num_sms, st);
}

// ------------------------------------------------ no-allocation variant
// Scratch of qx_gemm_splitk_noalloc, for callers that cannot allocate device
// memory: a file-scope device array (zero when the module loads) takes the
// place of the caller's workspace -- the 64 KiB counter region, then 4032 KiB
// of fp32 partial tiles (504 units of 16 tokens x 128 rows).
namespace {
constexpr int kNoAllocDevices = 64;
static __device__ __align__(256) uint8_t g_splitk_scratch[kNoAllocScratchBytes];
void *g_splitk_scratch_addr[kNoAllocDevices];
std::mutex g_splitk_scratch_mu;
}  // namespace

cudaError_t noalloc_scratch(void **ptr) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kNoAllocDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_splitk_scratch_mu);
    if (g_splitk_scratch_addr[dev] == nullptr) {
        // once per device, with that device current
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_splitk_scratch);
        if (e != cudaSuccess) return e;
        g_splitk_scratch_addr[dev] = p;
    }
    *ptr = g_splitk_scratch_addr[dev];
    return cudaSuccess;
}

}  // namespace qx
