// Shared device-side definitions of the qx library (sm_103a).
//
// The packed layout these helpers decode is fixed in include/qx.h.  Two code
// families share the unpack path (paper Section 2.2: uniform vs non-uniform):
//   * 4-bit uniform codes become fp16 (q - z) through the fp16 "magic number"
//     trick: OR-ing a nibble into the mantissa of 1024.0 gives 1024 + q exactly,
//     so one LOP3 plus one HSUB2/HFMA2 yields two exact (q - z) values.
//   * 3-bit codes (uniform or LUT) are looked up in an 8-entry fp16 table held
//     in four registers, split into low-byte and high-byte halves so that one
//     PRMT (byte permute) gathers four table bytes at once.
#pragma once

#include <cstdint>
#include <cuda_fp16.h>

namespace qx {

enum : uint32_t {
    kStatusNonfinite = 1u,  // qx_quantize met NaN/Inf
    kStatusTimeout = 2u,    // a bounded wait gave up
};

// ---------------------------------------------------------------- bit helpers
__device__ __forceinline__ uint32_t lop3_and_or(uint32_t a, uint32_t b, uint32_t c) {
    // (a & b) | c
    uint32_t d;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

__device__ __forceinline__ __half2 u2h2(uint32_t u) {
    __half2 h;
    *reinterpret_cast<uint32_t *>(&h) = u;
    return h;
}

__device__ __forceinline__ uint32_t h22u(__half2 h) { return *reinterpret_cast<uint32_t *>(&h); }

// ------------------------------------------------------------- 4-bit unpack
// One 32-bit word holds the codes of k = 8t..8t+7 with the code of j in nibble
// j/2 + 4*(j%2).  Returns the four half2 (q - z) pairs (k0,k1) (k2,k3) (k4,k5)
// (k6,k7), all exact.  zlo = half2(1024 + z), zhi = half2(-(64 + z)).
__device__ __forceinline__ void unpack4_qz(uint32_t w, __half2 zlo, __half2 zhi, __half2 (&o)[4]) {
    const uint32_t kMagic = 0x64006400u;  // half2(1024, 1024)
    const __half2 kSixteenth = u2h2(0x2C002C00u);  // half2(1/16, 1/16)
    uint32_t a = lop3_and_or(w, 0x000F000Fu, kMagic);       // 1024 + q(k0), 1024 + q(k1)
    uint32_t b = lop3_and_or(w, 0x00F000F0u, kMagic);       // 1024 + 16 q(k2), ...
    uint32_t c = lop3_and_or(w >> 8, 0x000F000Fu, kMagic);  // k4, k5
    uint32_t d = lop3_and_or(w >> 8, 0x00F000F0u, kMagic);  // k6, k7
    o[0] = __hsub2(u2h2(a), zlo);
    o[1] = __hfma2(u2h2(b), kSixteenth, zhi);
    o[2] = __hsub2(u2h2(c), zlo);
    o[3] = __hfma2(u2h2(d), kSixteenth, zhi);
}

__device__ __forceinline__ __half2 zlo_of(uint32_t z) { return u2h2((0x6400u | z) * 0x10001u); }

__device__ __forceinline__ __half2 zhi_of(uint32_t z) {
    __half h = __float2half_rn(-64.0f - (float)z);  // exact: small integer
    return __halves2half2(h, h);
}

// ------------------------------------------------------------- 3-bit unpack
// An 8-entry fp16 table split for PRMT: lo = the entries' low bytes (lo0 holds
// entries 0-3, lo1 entries 4-7), hi = their high bytes.
struct Table8 {
    uint32_t lo0, lo1, hi0, hi1;
};

// From four words u0..u3 holding entries (e0,e1) (e2,e3) (e4,e5) (e6,e7).
__device__ __forceinline__ Table8 make_table8(uint32_t u0, uint32_t u1, uint32_t u2, uint32_t u3) {
    Table8 t;
    t.lo0 = prmt(u0, u1, 0x6420u);
    t.hi0 = prmt(u0, u1, 0x7531u);
    t.lo1 = prmt(u2, u3, 0x6420u);
    t.hi1 = prmt(u2, u3, 0x7531u);
    return t;
}

// sel: four 3-bit codes in nibbles 0..3 of its low 16 bits (bit 3 of each
// nibble clear).  Returns half2(T[c0], T[c1]) and half2(T[c2], T[c3]).
__device__ __forceinline__ void lookup4(const Table8 &t, uint32_t sel, __half2 &p01, __half2 &p23) {
    uint32_t l = prmt(t.lo0, t.lo1, sel);
    uint32_t h = prmt(t.hi0, t.hi1, sel);
    p01 = u2h2(prmt(l, h, 0x5140u));
    p23 = u2h2(prmt(l, h, 0x7362u));
}

// x >> n (n = 1..31) computed as the high word of x * 2^(32-n): an integer
// multiply-add, which runs on the FMA pipe.  The 3-bit unpack is bound by the
// (half-rate) integer ALU pipe, which its byte permutes already fill.
__device__ __forceinline__ uint32_t shr_fma(uint32_t x, int n) {
    uint32_t d;
    asm("mul.hi.u32 %0, %1, %2;" : "=r"(d) : "r"(x), "r"(1u << (32 - n)));
    return d;
}

// One triple (A, B, C) codes 32 consecutive k.  Returns 16 half2 = T[code]
// for k = 0..31 of the triple in natural order.
__device__ __forceinline__ void lookup_triple(const Table8 &t, uint32_t A, uint32_t B, uint32_t C,
                                              __half2 (&o)[16]) {
    const uint32_t m = 0x77777777u;
    uint32_t a = A & m, b = B & m, c = C & m;
    uint32_t e = (shr_fma(A, 3) & 0x11111111u) | (shr_fma(B, 2) & 0x22222222u) | (shr_fma(C, 1) & 0x44444444u);
    lookup4(t, a, o[0], o[1]);
    lookup4(t, shr_fma(a, 16), o[2], o[3]);
    lookup4(t, b, o[4], o[5]);
    lookup4(t, shr_fma(b, 16), o[6], o[7]);
    lookup4(t, c, o[8], o[9]);
    lookup4(t, shr_fma(c, 16), o[10], o[11]);
    lookup4(t, e, o[12], o[13]);
    lookup4(t, shr_fma(e, 16), o[14], o[15]);
}

// Table of the uniform 3-bit grid offsets (j - z), j = 0..7, exact in fp16.
__device__ __forceinline__ Table8 table8_offsets(uint32_t z) {
    const __half2 zz = zlo_of(z);  // 1024 + z
    uint32_t u0 = h22u(__hsub2(u2h2(0x64016400u), zz));
    uint32_t u1 = h22u(__hsub2(u2h2(0x64036402u), zz));
    uint32_t u2 = h22u(__hsub2(u2h2(0x64056404u), zz));
    uint32_t u3 = h22u(__hsub2(u2h2(0x64076406u), zz));
    return make_table8(u0, u1, u2, u3);
}

// ------------------------------------------------------------- misc helpers
__device__ __forceinline__ uint32_t zero_nibble(const uint8_t *zrow, int grp) {
    return (zrow[grp >> 1] >> ((grp & 1) * 4)) & 15u;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

}  // namespace qx
