// Host-thread execution of CUDA kernel sources, for tests only.
//
// The kernels that use no TMA, mbarrier or tensor-core instructions (the
// quantizers, the dequantizers, the W.A8 pair, the error reduction and the Q4X
// path) are compiled for the host with this header and run on host threads, so
// that AddressSanitizer and UBSan check every index they form against buffers
// of exactly the size the C ABI states.  The library never loads this code.
//
// Model: blocks run one after another; the threads of a block are OS threads,
// so __syncthreads and the warp collectives are barriers (std::barrier) and a
// thread that returns leaves them.  __shared__ variables become function
// statics (shared by the block's threads); dynamic shared memory is a heap
// buffer of exactly the launch's size.  Atomics are std::atomic_ref.  IEEE
// float and double arithmetic is the host's (compiled without contraction);
// fp16 values are _Float16, and each fp16 operation rounds the exact (double)
// result once, as the device instruction does for the operands these kernels
// use.
#pragma once
#include <algorithm>
#include <atomic>
#include <barrier>
#include <chrono>
#include <cmath>
#include <condition_variable>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <memory>
#include <mutex>
#include <thread>
#include <unordered_map>
#include <limits>
#include <cstdio>
#include <vector>

#define __global__
#define __device__
#define __host__
#define __forceinline__ inline
#define __launch_bounds__(...)
#define __shared__ static
#define __align__(x) __attribute__((aligned(x)))
#define __grid_constant__

struct dim3 {
    unsigned x = 1, y = 1, z = 1;
    dim3(unsigned a = 1, unsigned b = 1, unsigned c = 1) : x(a), y(b), z(c) {}
};

namespace emu {
struct Warp {
    std::unique_ptr<std::barrier<>> bar;
    uint64_t buf[32];
    uint32_t mbuf[32][10];  // per-lane operands of a warp-wide matrix instruction
};
struct MBar {  // an mbarrier: arrivals still expected, transaction bytes, phase
    uint32_t count = 0, pending = 0, phase = 0;
    int64_t tx = 0;
};
struct Block {
    std::unique_ptr<std::barrier<>> bar;
    std::vector<Warp> warps;
    uint8_t *dyn = nullptr;  // dynamic shared memory, exactly the launch's size
    size_t dyn_bytes = 0;
    std::mutex mbar_mu;
    std::unordered_map<uint32_t, MBar> mbars;  // by shared-memory address
    std::vector<float> tmem;                   // tensor memory: 128 lanes x 512 columns
    uint32_t tmem_cols = 0;
    std::mutex nbar_mu;
    std::unique_ptr<std::barrier<>> nbar;      // named barrier 1 (the first use sets its count)
};
inline thread_local dim3 t_tid, t_bid;
inline thread_local Block *t_block = nullptr;
inline dim3 g_grid, g_blockdim;
}  // namespace emu

// the built-in indices, as variables (the grid's for the running launch)
inline thread_local dim3 &threadIdx = emu::t_tid;
inline thread_local dim3 &blockIdx = emu::t_bid;
inline dim3 &gridDim = emu::g_grid;
inline dim3 &blockDim = emu::g_blockdim;

using std::isfinite;
inline uint8_t *emu_dyn_smem();
inline void __syncthreads() { emu::t_block->bar->arrive_and_wait(); }
inline unsigned emu_lane() { return threadIdx.x & 31u; }
inline emu::Warp &emu_warp() { return emu::t_block->warps[threadIdx.x >> 5]; }
inline void __syncwarp(unsigned = 0xffffffffu) { emu_warp().bar->arrive_and_wait(); }

template <class T>
inline uint64_t emu_bits(T v) {
    uint64_t b = 0;
    std::memcpy(&b, &v, sizeof(T));
    return b;
}
template <class T>
inline T emu_from(uint64_t b) {
    T v;
    std::memcpy(&v, &b, sizeof(T));
    return v;
}
template <class T>
inline T emu_exchange(T v, int src) {
    emu::Warp &w = emu_warp();
    w.buf[emu_lane()] = emu_bits(v);
    w.bar->arrive_and_wait();
    const T r = emu_from<T>(w.buf[src & 31]);
    w.bar->arrive_and_wait();
    return r;
}
template <class T>
inline T __shfl_xor_sync(unsigned, T v, int o) { return emu_exchange(v, (int)emu_lane() ^ o); }
template <class T>
inline T __shfl_sync(unsigned, T v, int src) { return emu_exchange(v, src); }
template <class T>
inline T __shfl_up_sync(unsigned, T v, unsigned d) {
    const T r = emu_exchange(v, (int)emu_lane() >= (int)d ? (int)(emu_lane() - d) : (int)emu_lane());
    return r;
}
inline unsigned __ballot_sync(unsigned, bool p) {
    emu::Warp &w = emu_warp();
    w.buf[emu_lane()] = p ? 1 : 0;
    w.bar->arrive_and_wait();
    unsigned r = 0;
    for (int i = 0; i < 32; ++i) r |= (unsigned)w.buf[i] << i;
    w.bar->arrive_and_wait();
    return r;
}
inline bool __any_sync(unsigned m, bool p) { return __ballot_sync(m, p) != 0; }
inline bool __all_sync(unsigned m, bool p) { return __ballot_sync(m, p) == 0xffffffffu; }

template <class T, class U>
inline T atomicAdd(T *p, U v) {
    return std::atomic_ref<T>(*p).fetch_add((T)v);
}
template <class T, class U>
inline T atomicOr(T *p, U v) {
    return std::atomic_ref<T>(*p).fetch_or((T)v);
}

template <class T>
inline T min(T a, T b) { return a < b ? a : b; }
template <class T>
inline T max(T a, T b) { return a < b ? b : a; }

inline double __ddiv_rn(double a, double b) { return a / b; }
inline double __dmul_rn(double a, double b) { return a * b; }
inline double __dadd_rn(double a, double b) { return a + b; }
inline double __dsub_rn(double a, double b) { return a - b; }
inline float __fmul_rn(float a, float b) { return a * b; }
inline long long __double2ll_rn(double x) { return llrint(x); }
template <class T>
inline T __ldg(const T *p) { return *p; }

// ------------------------------------------------------------------ fp16
struct __half {
    uint16_t b;
};
struct alignas(4) __half2 {
    __half x, y;
};
struct float2 {
    float x, y;
};
struct alignas(16) float4 {
    float x, y, z, w;
};
struct alignas(16) uint4 {
    unsigned x, y, z, w;
};
inline uint4 make_uint4(unsigned a, unsigned b, unsigned c, unsigned d) { return uint4{a, b, c, d}; }
inline __half __ushort_as_half(unsigned short b) { return __half{b}; }
inline unsigned short __half_as_ushort(__half h) { return h.b; }
inline float __half2float(__half h) {
    _Float16 f;
    std::memcpy(&f, &h.b, 2);
    return (float)f;
}
inline __half __float2half_rn(float x) {
    _Float16 f = (_Float16)x;
    __half h;
    std::memcpy(&h.b, &f, 2);
    return h;
}
inline uint16_t emu_f64_to_f16(double x) {
    _Float16 f = (_Float16)x;
    uint16_t b;
    std::memcpy(&b, &f, 2);
    return b;
}
inline __half2 __halves2half2(__half a, __half b) { return __half2{a, b}; }
inline __half2 __hmul2(__half2 a, __half2 b) {
    // exact fp32 product of two fp16 values, one rounding to fp16
    return __half2{__float2half_rn(__half2float(a.x) * __half2float(b.x)),
                   __float2half_rn(__half2float(a.y) * __half2float(b.y))};
}
inline float2 __half22float2(__half2 h) { return float2{__half2float(h.x), __half2float(h.y)}; }
inline float __low2float(__half2 h) { return __half2float(h.x); }

// ------------------------------------------------------------------ runtime
typedef void *cudaStream_t;
enum cudaError_t { cudaSuccess = 0, cudaErrorInvalidValue = 1, cudaErrorInvalidConfiguration = 9, cudaErrorInvalidDevice = 101, cudaErrorCooperativeLaunchTooLarge = 720, cudaErrorNotSupported = 801 };
inline cudaError_t cudaMemsetAsync(void *p, int v, size_t n, cudaStream_t) {
    std::memset(p, v, n);
    return cudaSuccess;
}
inline cudaError_t cudaGetLastError() { return cudaSuccess; }
template <class F>
inline cudaError_t cudaOccupancyMaxActiveBlocksPerMultiprocessor(int *n, F, int, size_t) {
    *n = 3;
    return cudaSuccess;
}

namespace emu {
struct Cfg {
    dim3 grid, block;
    size_t smem = 0;
    cudaStream_t st = nullptr;
};

// Persistent OS threads, one per thread index of a block.
struct Pool {
    std::vector<std::thread> th;
    std::mutex mu;
    std::condition_variable cv, done_cv;
    uint64_t gen = 0;
    int active = 0, remaining = 0;
    std::function<void()> job;
    dim3 bid;
    Block *block = nullptr;
    bool stop = false;

    explicit Pool(int n) {
        for (int i = 0; i < n; ++i) th.emplace_back([this, i] { run(i); });
    }
    ~Pool() {
        {
            std::lock_guard<std::mutex> l(mu);
            stop = true;
            ++gen;
        }
        cv.notify_all();
        for (auto &t : th) t.join();
    }
    void run(int i) {
        uint64_t seen = 0;
        for (;;) {
            std::function<void()> f;
            {
                std::unique_lock<std::mutex> l(mu);
                cv.wait(l, [&] { return gen != seen; });
                seen = gen;
                if (stop) return;
                if (i >= active) continue;
                f = job;
                t_bid = bid;
                t_block = block;
            }
            t_tid = dim3((unsigned)i, 0, 0);
            f();
            // a returning thread leaves the barriers of its block and warp
            t_block->warps[i >> 5].bar->arrive_and_drop();
            t_block->bar->arrive_and_drop();
            {
                std::lock_guard<std::mutex> l(mu);
                if (--remaining == 0) done_cv.notify_one();
            }
        }
    }
    void start_block(int nthreads, dim3 b, Block *blk, const std::function<void()> &f) {
        {
            std::lock_guard<std::mutex> l(mu);
            job = f;
            bid = b;
            block = blk;
            active = nthreads;
            remaining = nthreads;
            ++gen;
        }
        cv.notify_all();
    }
    void wait_block() {
        std::unique_lock<std::mutex> l(mu);
        done_cv.wait(l, [&] { return remaining == 0; });
    }
    void launch_block(int nthreads, dim3 b, Block *blk, const std::function<void()> &f) {
        start_block(nthreads, b, blk, f);
        wait_block();
    }
};

inline Pool &pool() {
    static Pool p(1024);
    return p;
}

struct DynSmem {
    uint8_t *p;
    explicit DynSmem(size_t n) : p(n ? new (std::align_val_t(16)) uint8_t[n] : nullptr) {}
    ~DynSmem() { if (p) ::operator delete[](p, std::align_val_t(16)); }
};

inline void init_block(Block &blk, const DynSmem &dyn, size_t smem, int nt) {
    blk.dyn = dyn.p;
    blk.dyn_bytes = smem;
    blk.bar = std::make_unique<std::barrier<>>(nt);
    const int nw = (nt + 31) / 32;
    blk.warps.resize(nw);
    for (int w = 0; w < nw; ++w) blk.warps[w].bar = std::make_unique<std::barrier<>>(std::min(32, nt - 32 * w));
}

// Blocks one after another (a normal launch), or all at once, each on a thread
// pool of its own (a cooperative launch: its blocks may wait on one another).
inline void launch(const Cfg &c, const std::function<void()> &f, bool concurrent = false) {
    const int nt = (int)(c.block.x * c.block.y * c.block.z);
    g_grid = c.grid;
    g_blockdim = c.block;
    if (concurrent) {
        const int nb = (int)(c.grid.x * c.grid.y);
        std::vector<std::unique_ptr<Block>> blks;
        std::vector<std::unique_ptr<DynSmem>> dyns;
        std::vector<std::unique_ptr<Pool>> pools;
        for (int i = 0; i < nb; ++i) {
            blks.push_back(std::make_unique<Block>());
            dyns.push_back(std::make_unique<DynSmem>(c.smem));
            init_block(*blks.back(), *dyns.back(), c.smem, nt);
            pools.push_back(std::make_unique<Pool>(nt));
        }
        for (int i = 0; i < nb; ++i)
            pools[i]->start_block(nt, dim3((unsigned)(i % c.grid.x), (unsigned)(i / c.grid.x), 0), blks[i].get(), f);
        for (auto &p : pools) p->wait_block();
        return;
    }
    for (unsigned by = 0; by < c.grid.y; ++by)
        for (unsigned bx = 0; bx < c.grid.x; ++bx) {
            Block blk;
            DynSmem dyn(c.smem);
            init_block(blk, dyn, c.smem, nt);
            pool().launch_block(nt, dim3(bx, by, 0), &blk, f);
        }
}
}  // namespace emu

// ------------------------------------------------------------------ more intrinsics
inline uint32_t emu_prmt(uint32_t a, uint32_t b, uint32_t c) {
    const uint64_t v = ((uint64_t)b << 32) | a;
    uint32_t d = 0;
    for (int j = 0; j < 4; ++j) {
        const uint32_t s = (c >> (4 * j)) & 15u;
        uint32_t byte = (uint32_t)(v >> (8 * (s & 7))) & 255u;
        if (s & 8) byte = (byte & 0x80u) ? 0xFFu : 0u;
        d |= byte << (8 * j);
    }
    return d;
}
inline int __dp4a(int a, int b, int c) {
    for (int i = 0; i < 4; ++i) c += (int)(int8_t)(a >> (8 * i)) * (int)(int8_t)(b >> (8 * i));
    return c;
}
inline unsigned __vsub4(unsigned a, unsigned b) {
    unsigned d = 0;
    for (int i = 0; i < 4; ++i) d |= (((a >> (8 * i)) - (b >> (8 * i))) & 255u) << (8 * i);
    return d;
}
inline float __fdiv_rn(float a, float b) { return a / b; }
inline float __fsub_rn(float a, float b) { return a - b; }
inline float __fadd_rn(float a, float b) { return a + b; }
inline __half emu_h(double x) {
    _Float16 f = (_Float16)x;
    __half h;
    std::memcpy(&h.b, &f, 2);
    return h;
}
inline __half2 __hsub2(__half2 a, __half2 b) {
    return __half2{emu_h((double)__half2float(a.x) - (double)__half2float(b.x)),
                   emu_h((double)__half2float(a.y) - (double)__half2float(b.y))};
}
inline __half2 __hfma2(__half2 a, __half2 b, __half2 c) {
    return __half2{emu_h(std::fma((double)__half2float(a.x), (double)__half2float(b.x), (double)__half2float(c.x))),
                   emu_h(std::fma((double)__half2float(a.y), (double)__half2float(b.y), (double)__half2float(c.y)))};
}
inline uint64_t emu_globaltimer() {
    return (uint64_t)std::chrono::duration_cast<std::chrono::nanoseconds>(
               std::chrono::steady_clock::now().time_since_epoch()).count();
}
struct int4 { int x, y, z, w; };
// driver-API types named by the internal header
typedef int CUresult;
typedef int CUtensorMapDataType, CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
    CUtensorMapFloatOOBfill;
typedef unsigned cuuint32_t;
typedef unsigned long long cuuint64_t;
struct alignas(64) CUtensorMap { char b[128]; };
enum cudaFuncAttribute { cudaFuncAttributeMaxDynamicSharedMemorySize, cudaFuncAttributePreferredSharedMemoryCarveout };
inline cudaError_t cudaGetDevice(int *d) { *d = 0; return cudaSuccess; }
template <class F>
inline cudaError_t cudaFuncSetAttribute(F, cudaFuncAttribute, int) { return cudaSuccess; }

inline uint8_t *emu_dyn_smem() { return emu::t_block->dyn; }

// ------------------------------------------------------------------ TMA, mbarrier, launch
#define __noinline__ __attribute__((noinline))

[[noreturn]] inline void emu_fail(const char *what) {
    std::fprintf(stderr, "emulation check failed: %s\n", what);
    std::abort();
}
inline void __threadfence_block() { std::atomic_thread_fence(std::memory_order_seq_cst); }
inline void __threadfence() { std::atomic_thread_fence(std::memory_order_seq_cst); }
template <class T, class U>
inline T atomicMax(T *p, U v) {
    std::atomic_ref<T> r(*p);
    T o = r.load();
    while (o < (T)v && !r.compare_exchange_weak(o, (T)v)) {
    }
    return o;
}

// The shared state space is the block's dynamic shared memory: a shared
// address is an offset into it, checked on every use.
inline uint32_t __cvta_generic_to_shared(const void *p) {
    const emu::Block *b = emu::t_block;
    const ptrdiff_t o = static_cast<const uint8_t *>(p) - b->dyn;
    if (b->dyn == nullptr || o < 0 || (size_t)o >= b->dyn_bytes) emu_fail("generic address outside shared memory");
    return (uint32_t)o;
}
inline uint8_t *emu_shared(uint32_t a, size_t bytes) {
    const emu::Block *b = emu::t_block;
    if ((size_t)a + bytes > b->dyn_bytes) emu_fail("shared-memory access out of range");
    return b->dyn + a;
}
inline uint4 emu_lds128(uint32_t a) {
    if (a & 15u) emu_fail("misaligned 16-byte shared load");
    uint4 v;
    std::memcpy(&v, emu_shared(a, 16), 16);
    return v;
}

// ldmatrix .m8n8 .b16 (nmat = 1, 2 or 4 matrices): lanes 8i..8i+7 give the
// 16-byte row addresses of matrix i; lane l receives bytes 4(l%4)..4(l%4)+3
// of row l/4 of every matrix.
inline void emu_ldsm(uint32_t a, int nmat, uint32_t *d0, uint32_t *d1, uint32_t *d2, uint32_t *d3) {
    emu::Warp &w = emu_warp();
    const unsigned l = emu_lane();
    w.buf[l] = a;
    w.bar->arrive_and_wait();
    uint32_t *d[4] = {d0, d1, d2, d3};
    for (int i = 0; i < nmat; ++i) {
        const uint32_t row = (uint32_t)w.buf[8 * i + l / 4];
        if (row & 15u) emu_fail("misaligned ldmatrix row address");
        std::memcpy(d[i], emu_shared(row + 4 * (l % 4), 4), 4);
    }
    w.bar->arrive_and_wait();
}

// mma.sync m16n8k16 row.col f32.f16.f16.f32, D = A B + C, with lane (g, t)
// holding a0 = A[g][2t..2t+1], a1 = A[g+8][2t..], a2 = A[g][2t+8..],
// a3 = A[g+8][2t+8..], b0 = B[2t..2t+1][g], b1 = B[2t+8..2t+9][g] and
// D[g][2t], D[g][2t+1], D[g+8][2t], D[g+8][2t+1].  The fp16 products are exact;
// the sum is formed in double and rounded once to fp32 (the hardware's adder
// order is not specified, so results are checked within tolerance).
inline float emu_h2f(uint32_t bits16) {
    __half h;
    const uint16_t b = (uint16_t)bits16;
    std::memcpy(&h, &b, 2);
    return __half2float(h);
}
inline void emu_mma16816(float &d0, float &d1, float &d2, float &d3, uint32_t a0, uint32_t a1, uint32_t a2,
                         uint32_t a3, uint32_t b0, uint32_t b1) {
    emu::Warp &w = emu_warp();
    const unsigned l = emu_lane();
    uint32_t *m = w.mbuf[l];
    const float c[4] = {d0, d1, d2, d3};
    m[0] = a0; m[1] = a1; m[2] = a2; m[3] = a3; m[4] = b0; m[5] = b1;
    std::memcpy(&m[6], c, 16);
    w.bar->arrive_and_wait();
    auto A = [&](int row, int k) {  // A[row][k]
        const uint32_t r = w.mbuf[4 * (row % 8) + (k % 8) / 2][(row >= 8 ? 1 : 0) + (k >= 8 ? 2 : 0)];
        return emu_h2f(k % 2 ? r >> 16 : r);
    };
    auto B = [&](int k, int col) {  // B[k][col]
        const uint32_t r = w.mbuf[4 * col + (k % 8) / 2][4 + (k >= 8 ? 1 : 0)];
        return emu_h2f(k % 2 ? r >> 16 : r);
    };
    const int g = (int)l / 4, t = (int)l % 4;
    float out[4];
    for (int i = 0; i < 4; ++i) {
        const int row = g + 8 * (i / 2), col = 2 * t + (i % 2);
        double s = c[i];
        for (int k = 0; k < 16; ++k) s += (double)A(row, k) * (double)B(k, col);
        out[i] = (float)s;
    }
    w.bar->arrive_and_wait();
    d0 = out[0]; d1 = out[1]; d2 = out[2]; d3 = out[3];
}

// atom.add on a shared-memory word (by its shared address)
inline uint32_t emu_atom_add_shared(uint32_t a, uint32_t v) {
    if (a & 3u) emu_fail("misaligned shared atomic");
    return std::atomic_ref<uint32_t>(*reinterpret_cast<uint32_t *>(emu_shared(a, 4))).fetch_add(v);
}
inline void __nanosleep(unsigned) { std::this_thread::yield(); }

// bar.sync 1, n: a barrier of n threads of the block
inline void emu_named_bar(unsigned n) {
    emu::Block *b = emu::t_block;
    {
        std::lock_guard<std::mutex> l(b->nbar_mu);
        if (!b->nbar) b->nbar = std::make_unique<std::barrier<>>((std::ptrdiff_t)n);
    }
    b->nbar->arrive_and_wait();
}

inline emu::MBar &emu_mbar(uint32_t a) {
    auto it = emu::t_block->mbars.find(a);
    if (it == emu::t_block->mbars.end()) emu_fail("mbarrier used before init");
    return it->second;
}
inline void emu_mbar_settle(emu::MBar &m) {
    if (m.pending == 0 && m.tx == 0) {
        m.phase ^= 1u;
        m.pending = m.count;
    }
}
inline void emu_mbar_init(uint32_t a, uint32_t count) {
    if (a & 7u) emu_fail("misaligned mbarrier");
    emu_shared(a, 8);
    std::lock_guard<std::mutex> l(emu::t_block->mbar_mu);
    emu::MBar &m = emu::t_block->mbars[a];
    m.count = m.pending = count;
    m.phase = 0;
    m.tx = 0;
}
inline void emu_mbar_arrive_expect_tx(uint32_t a, uint32_t bytes) {
    std::lock_guard<std::mutex> l(emu::t_block->mbar_mu);
    emu::MBar &m = emu_mbar(a);
    if (m.pending == 0) emu_fail("arrival on a completed mbarrier phase");
    m.tx += bytes;
    --m.pending;
    emu_mbar_settle(m);
}
inline void emu_mbar_complete_tx(uint32_t a, uint32_t bytes) {
    std::lock_guard<std::mutex> l(emu::t_block->mbar_mu);
    emu::MBar &m = emu_mbar(a);
    m.tx -= bytes;
    emu_mbar_settle(m);
}
// true once the phase of the given parity has completed
inline bool emu_mbar_try_wait(uint32_t a, uint32_t parity) {
    bool done;
    {
        std::lock_guard<std::mutex> l(emu::t_block->mbar_mu);
        done = emu_mbar(a).phase != (parity & 1u);
    }
    if (!done) std::this_thread::yield();
    return done;
}

// Tensor maps: the parameters cuTensorMapEncodeTiled takes, checked as the
// driver checks them, kept in the 128-byte descriptor.
enum { CUDA_SUCCESS = 0, CUDA_ERROR_INVALID_VALUE = 1 };
enum { CU_TENSOR_MAP_DATA_TYPE_UINT8 = 0, CU_TENSOR_MAP_DATA_TYPE_FLOAT16 = 6 };
enum { CU_TENSOR_MAP_INTERLEAVE_NONE = 0 };
enum { CU_TENSOR_MAP_SWIZZLE_NONE = 0, CU_TENSOR_MAP_SWIZZLE_128B = 3 };
enum { CU_TENSOR_MAP_L2_PROMOTION_L2_256B = 3 };
enum { CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE = 0 };
struct EmuTensorMap {
    const uint8_t *base;
    uint32_t rank, esize, swizzle128, pad;
    uint64_t dims[5], strides[5];  // strides[0] = element size; strides[i] in bytes
    uint32_t box[5];
};
static_assert(sizeof(EmuTensorMap) <= sizeof(CUtensorMap), "tensor map fits its descriptor");
inline CUresult emu_encode_tiled(CUtensorMap *out, CUtensorMapDataType dt, cuuint32_t rank, void *base,
                                 const cuuint64_t *dims, const cuuint64_t *strides, const cuuint32_t *box,
                                 const cuuint32_t *estr, CUtensorMapInterleave, CUtensorMapSwizzle sw,
                                 CUtensorMapL2promotion, CUtensorMapFloatOOBfill) {
    EmuTensorMap m{};
    m.esize = dt == CU_TENSOR_MAP_DATA_TYPE_FLOAT16 ? 2 : 1;
    if (rank < 1 || rank > 5 || ((uintptr_t)base & 15u)) return CUDA_ERROR_INVALID_VALUE;
    m.base = static_cast<const uint8_t *>(base);
    m.rank = rank;
    m.swizzle128 = sw == CU_TENSOR_MAP_SWIZZLE_128B;
    m.strides[0] = m.esize;
    for (uint32_t i = 0; i < rank; ++i) {
        if (dims[i] < 1 || box[i] < 1 || box[i] > 256 || estr[i] != 1) return CUDA_ERROR_INVALID_VALUE;
        m.dims[i] = dims[i];
        m.box[i] = box[i];
        if (i > 0) {
            if (strides[i - 1] % 16) return CUDA_ERROR_INVALID_VALUE;
            m.strides[i] = strides[i - 1];
        }
    }
    if ((m.box[0] * m.esize) % 16 || (m.swizzle128 && m.box[0] * m.esize > 128)) return CUDA_ERROR_INVALID_VALUE;
    std::memset(out, 0, sizeof(CUtensorMap));
    std::memcpy(out, &m, sizeof(m));
    return CUDA_SUCCESS;
}

// A tiled TMA load: the whole box lands at once (out-of-range elements as
// zeros), with the 128-byte swizzle taken from the shared address bits, then
// its bytes complete on the mbarrier.
inline void emu_tma_load(uint32_t dst, const void *map, uint32_t bar, const int *c, int rank) {
    const EmuTensorMap &m = *static_cast<const EmuTensorMap *>(map);
    if ((uint32_t)rank != m.rank) emu_fail("TMA rank differs from the tensor map");
    if (((int64_t)c[0] * m.esize) % 16) emu_fail("TMA innermost coordinate not 16-byte aligned");
    if (m.swizzle128 && (dst & 1023u)) emu_fail("swizzled TMA destination not 1024-byte aligned");
    if (dst & 15u) emu_fail("TMA destination not 16-byte aligned");
    uint64_t total = 1;
    for (int d = 0; d < rank; ++d) total *= m.box[d];
    const uint64_t bytes = total * m.esize;
    emu_shared(dst, bytes);
    for (uint64_t idx = 0; idx < total; ++idx) {
        uint64_t rem = idx, src = 0;
        bool in = true;
        for (int d = 0; d < rank; ++d) {
            const int64_t g = (int64_t)c[d] + (int64_t)(rem % m.box[d]);
            rem /= m.box[d];
            if (g < 0 || (uint64_t)g >= m.dims[d]) in = false;
            else src += (uint64_t)g * m.strides[d];
        }
        uint32_t a = dst + (uint32_t)(idx * m.esize);
        if (m.swizzle128) a ^= ((a >> 7) & 7u) << 4;
        uint8_t *p = emu_shared(a, m.esize);
        if (in)
            std::memcpy(p, m.base + src, m.esize);
        else
            std::memset(p, 0, m.esize);
    }
    emu_mbar_complete_tx(bar, (uint32_t)bytes);
}

// cudaLaunchKernelEx with its configuration (kernels run one after another;
// of the launch attributes only the cooperative one counts: its blocks run at
// the same time).
enum cudaLaunchAttributeID { cudaLaunchAttributeProgrammaticStreamSerialization = 1, cudaLaunchAttributeCooperative = 2 };
struct cudaLaunchAttributeValue {
    int programmaticStreamSerializationAllowed;
    int cooperative;
};
struct cudaLaunchAttribute {
    cudaLaunchAttributeID id;
    cudaLaunchAttributeValue val;
};
struct cudaLaunchConfig_t {
    dim3 gridDim, blockDim;
    size_t dynamicSmemBytes;
    cudaStream_t stream;
    cudaLaunchAttribute *attrs;
    unsigned numAttrs;
};
template <class K, class... A>
inline cudaError_t cudaLaunchKernelEx(const cudaLaunchConfig_t *c, K k, A... args) {
    bool coop = false;
    for (unsigned i = 0; i < c->numAttrs; ++i)
        coop = coop || (c->attrs[i].id == cudaLaunchAttributeCooperative && c->attrs[i].val.cooperative);
    emu::launch(emu::Cfg{c->gridDim, c->blockDim, c->dynamicSmemBytes, c->stream}, [&] { k(args...); }, coop);
    return cudaSuccess;
}

// ------------------------------------------------------------------ tensor cores
inline float __uint_as_float(uint32_t u) {
    float f;
    std::memcpy(&f, &u, 4);
    return f;
}
inline __half2 __float2half2_rn(float x) { return __half2{__float2half_rn(x), __float2half_rn(x)}; }
template <class T>
inline T __ldcg(const T *p) { return *p; }
template <class T>
inline void __stcg(T *p, T v) { *p = v; }
inline uint32_t emu_lds32(uint32_t a) {
    if (a & 3u) emu_fail("misaligned 4-byte shared load");
    uint32_t v;
    std::memcpy(&v, emu_shared(a, 4), 4);
    return v;
}
inline void emu_mbar_arrive(uint32_t a) {
    std::lock_guard<std::mutex> l(emu::t_block->mbar_mu);
    emu::MBar &m = emu_mbar(a);
    if (m.pending == 0) emu_fail("arrival on a completed mbarrier phase");
    --m.pending;
    emu_mbar_settle(m);
}

// Allocation is warp-collective: lane 0 acts for the warp.  Columns: a power
// of two in 32..512; unwritten accumulators read as NaN.
inline void emu_tmem_alloc(uint32_t dst, uint32_t cols) {
    if (emu_lane() != 0) return;
    emu::Block &b = *emu::t_block;
    if (cols < 32 || cols > 512 || (cols & (cols - 1))) emu_fail("TMEM allocation size");
    if (b.tmem_cols != 0) emu_fail("second TMEM allocation in a CTA");
    b.tmem.assign(128 * 512, std::numeric_limits<float>::quiet_NaN());
    b.tmem_cols = cols;
    const uint32_t base = 0;  // lane 0, column 0
    std::memcpy(emu_shared(dst, 4), &base, 4);
}
inline void emu_tmem_dealloc(uint32_t taddr, uint32_t cols) {
    if (emu_lane() != 0) return;
    emu::Block &b = *emu::t_block;
    if (taddr != 0 || cols != b.tmem_cols) emu_fail("TMEM deallocation differs from the allocation");
    b.tmem_cols = 0;
}
// 32x32b load: lane l of the warp reads row (lane base + l), n columns.  A warp
// reaches only the 32 lanes of its quarter (warp id % 4).
inline void emu_tmem_ld(uint32_t taddr, uint32_t *r, int n) {
    const emu::Block &b = *emu::t_block;
    const uint32_t lane0 = taddr >> 16, col = taddr & 0xFFFFu;
    if (lane0 != 32u * ((threadIdx.x >> 5) & 3u)) emu_fail("TMEM lanes outside the warp's quarter");
    if (col + (uint32_t)n > b.tmem_cols) emu_fail("TMEM columns outside the allocation");
    const float *row = b.tmem.data() + (size_t)(lane0 + emu_lane()) * 512 + col;
    std::memcpy(r, row, 4 * (size_t)n);
}
// K-major operand, 128-byte swizzle: row r, element k (fp16) of the tile a
// shared-memory descriptor names.
inline double emu_desc_elem(uint64_t desc, int r, int k) {
    if ((desc >> 61) != 2u || ((desc >> 46) & 3u) != 1u || ((desc >> 49) & 7u) != 0u)
        emu_fail("shared-memory descriptor: not a 128-byte-swizzle K-major tcgen05 descriptor");
    const uint32_t start = (uint32_t)(desc & 0x3FFFu) << 4, sbo = (uint32_t)((desc >> 32) & 0x3FFFu) << 4;
    const uint32_t lin = start + (uint32_t)(r / 8) * sbo + (uint32_t)(r % 8) * 128u + 2u * (uint32_t)k;
    const uint32_t phys = lin ^ (((lin >> 7) & 7u) << 4);
    __half h;
    std::memcpy(&h, emu_shared(phys, 2), 2);
    return (double)__half2float(h);
}
// D[M][N] (+)= A[M][16] B[N][16]^T, fp16 operands, fp32 accumulators.
inline void emu_mma_f16(uint32_t d, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t acc) {
    emu::Block &b = *emu::t_block;
    if (((idesc >> 4) & 3u) != 1u || ((idesc >> 7) & 7u) != 0u || ((idesc >> 10) & 7u) != 0u ||
        ((idesc >> 15) & 3u) != 0u)
        emu_fail("instruction descriptor: expected fp16 K-major operands and fp32 accumulators");
    const int N = (int)((idesc >> 17) & 63u) << 3, M = (int)((idesc >> 24) & 31u) << 4;
    if (M != 128 || N < 16 || N > 256 || N % 16) emu_fail("MMA shape for cta_group::1, M = 128");
    const uint32_t lane0 = d >> 16, col0 = d & 0xFFFFu;
    if (lane0 != 0 || col0 + (uint32_t)N > b.tmem_cols) emu_fail("MMA accumulator outside the allocation");
    for (int m = 0; m < M; ++m) {
        double a[16];
        for (int k = 0; k < 16; ++k) a[k] = emu_desc_elem(adesc, m, k);
        float *row = b.tmem.data() + (size_t)m * 512 + col0;
        for (int n = 0; n < N; ++n) {
            double sum = 0.0;
            for (int k = 0; k < 16; ++k) sum += a[k] * emu_desc_elem(bdesc, n, k);
            row[n] = acc ? row[n] + (float)sum : (float)sum;
        }
    }
}

// runtime lookups the host code makes
enum cudaDriverEntryPointQueryResult { cudaDriverEntryPointSuccess = 0, cudaDriverEntryPointSymbolNotFound = 1 };
enum { cudaEnableDefault = 0 };
inline cudaError_t cudaGetDriverEntryPointByVersion(const char *name, void **p, unsigned, unsigned long long,
                                                    cudaDriverEntryPointQueryResult *q) {
    const bool ok = std::strcmp(name, "cuTensorMapEncodeTiled") == 0;
    *p = ok ? reinterpret_cast<void *>(&emu_encode_tiled) : nullptr;
    *q = ok ? cudaDriverEntryPointSuccess : cudaDriverEntryPointSymbolNotFound;
    return cudaSuccess;
}
template <class T>
inline cudaError_t cudaGetSymbolAddress(void **p, T &sym) {
    *p = static_cast<void *>(&sym);
    return cudaSuccess;
}

// ------------------------------------------------------------------ the C ABI's runtime calls
// One emulated device; its SM count comes from QX_EMU_SMS (default 4).
enum cudaDeviceAttr { cudaDevAttrMultiProcessorCount = 16 };
enum cudaMemcpyKind { cudaMemcpyHostToHost = 0, cudaMemcpyHostToDevice = 1, cudaMemcpyDeviceToHost = 2,
                      cudaMemcpyDeviceToDevice = 3, cudaMemcpyDefault = 4 };
inline cudaError_t cudaDeviceGetAttribute(int *v, cudaDeviceAttr attr, int) {
    if (attr != cudaDevAttrMultiProcessorCount) return cudaErrorInvalidValue;
    const char *e = std::getenv("QX_EMU_SMS");
    *v = e != nullptr ? std::atoi(e) : 4;
    return *v > 0 ? cudaSuccess : cudaErrorInvalidValue;
}
inline cudaError_t cudaMemcpy(void *d, const void *s, size_t n, cudaMemcpyKind) {
    std::memcpy(d, s, n);
    return cudaSuccess;
}
inline cudaError_t cudaMemcpyAsync(void *d, const void *s, size_t n, cudaMemcpyKind, cudaStream_t) {
    std::memcpy(d, s, n);
    return cudaSuccess;
}
inline cudaError_t cudaStreamSynchronize(cudaStream_t) { return cudaSuccess; }
inline cudaError_t cudaDeviceSynchronize() { return cudaSuccess; }
// Graphs: the emulation runs every call in order, so a decode step is never
// captured (no stream reports capturing, no host memory counts as pinned).
enum cudaStreamCaptureStatus { cudaStreamCaptureStatusNone = 0, cudaStreamCaptureStatusActive = 1 };
enum cudaStreamCaptureMode { cudaStreamCaptureModeThreadLocal = 1 };
enum cudaMemoryType { cudaMemoryTypeUnregistered = 0, cudaMemoryTypeHost = 1, cudaMemoryTypeDevice = 2 };
enum { cudaStreamNonBlocking = 1 };
struct cudaPointerAttributes {
    cudaMemoryType type;
    void *devicePointer;
};
typedef struct EmuGraph *cudaGraph_t;
typedef struct EmuGraphExec *cudaGraphExec_t;
inline cudaError_t cudaStreamIsCapturing(cudaStream_t, cudaStreamCaptureStatus *s) {
    *s = cudaStreamCaptureStatusNone;
    return cudaSuccess;
}
inline cudaError_t cudaPointerGetAttributes(cudaPointerAttributes *a, const void *) {
    a->type = cudaMemoryTypeUnregistered;
    a->devicePointer = nullptr;
    return cudaSuccess;
}
inline cudaError_t cudaStreamCreateWithFlags(cudaStream_t *s, unsigned) {
    *s = nullptr;
    return cudaErrorNotSupported;
}
inline cudaError_t cudaStreamBeginCapture(cudaStream_t, cudaStreamCaptureMode) { return cudaErrorNotSupported; }
inline cudaError_t cudaStreamEndCapture(cudaStream_t, cudaGraph_t *g) {
    *g = nullptr;
    return cudaErrorNotSupported;
}
inline cudaError_t cudaGraphInstantiate(cudaGraphExec_t *e, cudaGraph_t, unsigned long long) {
    *e = nullptr;
    return cudaErrorNotSupported;
}
inline cudaError_t cudaGraphDestroy(cudaGraph_t) { return cudaSuccess; }
inline cudaError_t cudaGraphExecDestroy(cudaGraphExec_t) { return cudaSuccess; }
inline cudaError_t cudaGraphLaunch(cudaGraphExec_t, cudaStream_t) { return cudaErrorNotSupported; }
inline const char *cudaGetErrorName(cudaError_t e) { return e == cudaSuccess ? "cudaSuccess" : "cudaErrorEmulated"; }
