// Device helpers shared by the single-layer and the stack tensor-core conv
// kernels: layer arguments, tile geometry, the packed-code gather and the
// k-bit -> e4m3 expansion into tensor memory.  See conv_tc.cuh for the data
// path and the exactness argument.
#pragma once
#include <cuda.h>

#include <cstdint>

#include "ptx.cuh"

namespace ifq {


// n / d for 0 <= n < 2^31 by multiply-high (Granlund-Montgomery), set up on the host.
struct FastDiv {
  uint32_t d, mul, shift;
};
__device__ __forceinline__ uint32_t fdiv(uint32_t n, FastDiv f) {
  return (uint32_t)(((uint64_t)__umulhi(n, f.mul) + n) >> f.shift);
}

struct ConvArgs {
  const uint8_t* x;      // packed input codes, NHWC
  const uint8_t* wbits;  // filter sign bits in the e4m3 rows' K order, [cout][Kpad / 8] bytes (bit = +1),
                         // read by the kernels that expand B in shared memory (BX), else unused
  const int32_t* thr;    // [cout][lvl]
  const int8_t* sign;    // [cout]
  uint8_t* y_codes;      // packed output codes or nullptr
  int32_t* y_acc;        // int32 accumulators or nullptr
  int n, h, w, cin, cout, kh, kw, stride, pad, ho, wo;
  int cinb;              // bytes of packed codes per input pixel (cin * field bits / 8)
  int lvl;               // thresholds per channel, 2^k - 1
  int M;                 // n*ho*wo
  int K;                 // kh*kw*cin
  int nk;                // number of 128-wide K stages (Kpad / 128)
  int nt;                // number of BN-wide output-channel tiles
  int ntiles;            // M tiles * nt
  int ntab;              // entries of the K-granule table (packed bytes of Kpad / granule bytes)
  FastDiv div_hw, div_wo, div_nt;   // by ho*wo, wo, nt
  // Fused p x p / stride p pool (p = 1 << lpool, lpool = 0: none).  Tile rows are then ordered
  // by pooled pixel and, within it, by window position (p*p consecutive rows, dy-major), so
  // that a window's rows sit in consecutive lanes of one epilogue warp.
  int lpool;
  FastDiv div_phw, div_pwo;         // by (ho/p)*(wo/p), wo/p
  // 1: the kernels before this one in the stream write neither its filters nor its thresholds (a
  // layer of a stack after the first), so only the warps that read the previous layer's codes wait
  // for them; the filter and threshold loads start at once
  int early;
};

constexpr int kBM = 128;         // output pixels per tile (MMA M)
constexpr int kBK = 128;         // K elements (= bytes) per pipeline stage
constexpr int kGatherGroups = 4;
constexpr int kGatherWarps = 4 * kGatherGroups;
constexpr int kEpiWarps = 8;
constexpr int kTcThreads = 32 * (kGatherWarps + 2 + kEpiWarps);   // 832
constexpr int kWarpTma = kGatherWarps, kWarpMma = kGatherWarps + 1, kWarpEpi0 = kGatherWarps + 2;
constexpr int kMaxTab = 1024;    // K-granule table entries
constexpr int kStages = 8;       // K stages in flight (A in tensor memory, B in shared memory)
constexpr int kTmemA = 256;      // first tensor-memory column of the A stages
constexpr int kAhead = 2;        // own K stages of packed codes a gather thread keeps in registers

// SB: bits per stored code (2, or 4 for 3- and 4-bit codes).  Thresholds per column: a float4
// (3 thresholds and the sign) for SB = 2, five float4 (15 thresholds, padded with +inf, in the
// order of the 4-ary search, and the sign) for SB = 4.
// KS > 1 (split K over a cluster of KS CTAs): KS - 1 receive slots of fp32 partial sums, one per
// partner, each 128 rows x BN / KS columns (rows padded by 16 bytes), and two more barriers.
// BX = 1 (filter tiles expanded from sign bits): a ring of kBitStages slots of BN rows x 16 bytes
// (one K stage's 128 sign bits a row), filled by TMA ahead of the gather, and its two barriers a slot.
template <int BN, int SB = 2, int KS = 1, int BX = 0>
struct TcSmem {
  static constexpr int kB = BN * kBK;
  static constexpr int kThrCol = SB == 2 ? 16 : 80;       // bytes of thresholds per column
  static constexpr int kRecvRow = BN / KS + 4;             // floats per row of a receive slot
  static constexpr int kRecvSlot = kBM * kRecvRow * 4;     // bytes of a receive slot
  static constexpr int kBitStages = BX ? 32 : 0;
  static constexpr int kBitSlot = BN * 16;
  static constexpr int offB = 0;
  static constexpr int offThr = offB + kStages * kB;       // 2 buffers of BN columns
  static constexpr int offTab = offThr + 2 * BN * kThrCol; // kMaxTab x int2
  static constexpr int offRecv = offTab + kMaxTab * 8;
  static constexpr int offBits = offRecv + (KS - 1) * kRecvSlot;
  static constexpr int offBar = offBits + kBitStages * kBitSlot;
  // full, empty, acc_full[2], acc_empty[2], done (+ recv_full, send_ok) (+ bits_full, bits_empty)
  static constexpr int nBar = 2 * kStages + 5 + (KS > 1 ? 2 : 0) + 2 * kBitStages;
  static constexpr int offTmem = offBar + nBar * 8;
  static constexpr int bytes = offTmem + 16 + 1024;        // + alignment slack
};

// The input row (output pixel) that a gather thread reads in one tile: a base
// pointer for tap (0,0) (possibly outside the image; dereferenced only when
// valid) and the taps that fall inside the image: bit dy of vyx for the filter
// rows, bit 16 + dx for the filter columns (kh, kw <= 15, so bits 15 and 31
// are never set).
struct RowGeom {
  const uint8_t* base;
  uint32_t vyx;
};

// A K-granule's tap as a mask for tap_ok: bit dy and bit 16 + dx; past K, all ones (never inside,
// because bits 15 and 31 of a row's mask are clear).
__host__ __device__ constexpr int tap_mask(int dy, int dx) { return (int)((1u << dy) | (1u << (16 + dx))); }
constexpr int kTapNone = -1;

// bits lo..hi-1 of a tap mask (empty when hi <= lo); hi - lo <= 32
__device__ __forceinline__ uint32_t bit_range(int lo, int hi) {
  return hi > lo ? (uint32_t)(((1ull << (hi - lo)) - 1ull) << lo) : 0u;
}

__device__ __forceinline__ RowGeom row_geom(const ConvArgs& a, int m) {
  RowGeom g;
  g.base = a.x;
  g.vyx = 0;
  if (m < a.M) {
    int b, oy, ox;
    if (a.lpool == 0) {
      b = (int)fdiv((uint32_t)m, a.div_hw);
      const int rem = m - b * a.ho * a.wo;
      oy = (int)fdiv((uint32_t)rem, a.div_wo);
      ox = rem - oy * a.wo;
    } else {   // row m = window position w of pooled pixel P
      const int P = m >> (2 * a.lpool), wpos = m & ((1 << (2 * a.lpool)) - 1);
      const int pwo = a.wo >> a.lpool;
      b = (int)fdiv((uint32_t)P, a.div_phw);
      const int rem = P - b * (a.ho >> a.lpool) * pwo;
      const int py = (int)fdiv((uint32_t)rem, a.div_pwo), px = rem - py * pwo;
      oy = (py << a.lpool) + (wpos >> a.lpool);
      ox = (px << a.lpool) + (wpos & ((1 << a.lpool) - 1));
    }
    const int iy0 = oy * a.stride - a.pad, ix0 = ox * a.stride - a.pad;
    g.base = a.x + ((long long)b * a.h * a.w + (long long)iy0 * a.w + ix0) * a.cinb;
    g.vyx = bit_range(max(0, -iy0), min(a.kh, a.h - iy0)) | (bit_range(max(0, -ix0), min(a.kw, a.w - ix0)) << 16);
  }
  return g;
}

// Whether a granule's tap (e.y = tap_mask(dy, dx), or kTapNone past K) lies inside the image for
// this row: both its row bit and its column bit are set.
__device__ __forceinline__ bool tap_ok(const RowGeom& g, int2 e) { return (g.vyx & (uint32_t)e.y) == (uint32_t)e.y; }

// Loads of packed codes.  COHERENT = false: the codes were written by an earlier kernel and
// stay read-only for this one, so they may take the non-coherent read-only path (ld.global.nc).
// COHERENT = true: another CTA of the same kernel wrote them and this thread ordered itself
// after those writes with an acquire load of a completion counter, so only ordinary weak loads
// are allowed (the memory model makes them see the released writes; .nc loads carry no such
// guarantee).  Plain dereferences keep the compiler from moving them above the acquire.
template <bool COHERENT>
__device__ __forceinline__ uint4 ld_codes16(const uint8_t* p) {
  if constexpr (COHERENT) return *(const uint4*)p;
  else return __ldg((const uint4*)p);
}
template <bool COHERENT>
__device__ __forceinline__ uint2 ld_codes8(const uint8_t* p) {
  if constexpr (COHERENT) return *(const uint2*)p;
  else return __ldg((const uint2*)p);
}
template <bool COHERENT>
__device__ __forceinline__ uint32_t ld_codes4(const uint8_t* p) {
  if constexpr (COHERENT) return *(const uint32_t*)p;
  else return __ldg((const uint32_t*)p);
}
template <bool COHERENT>
__device__ __forceinline__ uint32_t ld_codes1(const uint8_t* p) {
  if constexpr (COHERENT) return (uint32_t)*p;
  else return (uint32_t)__ldg(p);
}

// 16 packed bytes of row g: unit u of the row's K sequence (bytes 16u .. 16u+15 of the packed
// K codes, 64 two-bit or 32 four-bit codes), zero outside the image.  The table has one entry
// per GB bytes (GB = 16, 8, 4 or 1), so unit u starts at entry u * 16 / GB.
template <int GB, bool COHERENT = false>
__device__ __forceinline__ uint4 load_unit(const int2* tab, const RowGeom& g, int u) {
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if constexpr (GB == 16) {
    const int2 e = tab[u];
    if (tap_ok(g, e)) v = ld_codes16<COHERENT>(g.base + e.x);
  } else if constexpr (GB == 8) {
    const int2 e0 = tab[u * 2], e1 = tab[u * 2 + 1];
    const uint2 lo = tap_ok(g, e0) ? ld_codes8<COHERENT>(g.base + e0.x) : make_uint2(0u, 0u);
    const uint2 hi = tap_ok(g, e1) ? ld_codes8<COHERENT>(g.base + e1.x) : make_uint2(0u, 0u);
    v = make_uint4(lo.x, lo.y, hi.x, hi.y);
  } else if constexpr (GB == 4) {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int2 e = tab[u * 4 + q];
      w[q] = tap_ok(g, e) ? ld_codes4<COHERENT>(g.base + e.x) : 0u;
    }
    v = make_uint4(w[0], w[1], w[2], w[3]);
  } else {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint32_t x = 0;
#pragma unroll
      for (int bq = 0; bq < 4; ++bq) {
        const int2 e = tab[u * 16 + q * 4 + bq];
        if (tap_ok(g, e)) x |= ld_codes1<COHERENT>(g.base + e.x) << (8 * bq);
      }
      w[q] = x;
    }
    v = make_uint4(w[0], w[1], w[2], w[3]);
  }
  return v;
}

// 16 columns of zeros into tensor memory (this warp's 32 lanes), with the wait for the store.
__device__ __forceinline__ void tmem_zero16_sync(uint32_t taddr) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1};\n\t"
      "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
      "r"(0u)
      : "memory");
}

// 32 lanes x 16 consecutive columns of 32-bit tensor memory -> 16 registers per thread.  The load
// writes its destination registers asynchronously; the wait is in the same asm statement, so the
// compiler never sees the registers before they hold the data.
__device__ __forceinline__ void tmem_ld16_sync(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
      : "r"(taddr)
      : "memory");
}

// 16 registers -> 16 consecutive tensor-memory columns of this warp's 32 lanes, and the wait for
// the store in the same asm statement, so the compiler cannot reuse the source registers while the
// asynchronous store may still read them.
__device__ __forceinline__ void tmem_st16_sync(uint32_t taddr, const uint32_t* o) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n\t"
      "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
      "r"(o[0]), "r"(o[1]), "r"(o[2]), "r"(o[3]), "r"(o[4]), "r"(o[5]), "r"(o[6]), "r"(o[7]), "r"(o[8]), "r"(o[9]),
      "r"(o[10]), "r"(o[11]), "r"(o[12]), "r"(o[13]), "r"(o[14]), "r"(o[15])
      : "memory");
}

// fma(a, b, c) saturated to [0, 1] (one fma.sat on the FMA pipe).  The threshold epilogues use it
// as an exact step function: for integers x, sat(x) = [x > 0], and a * 512 s - T with a = A / 512
// is the integer s A - T (|s A - T| < 2^24 for every layer the tensor-core paths admit).
__device__ __forceinline__ float sat_fma(float a, float b, float c) {
  float r;
  asm("fma.rn.sat.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// 16 packed two-bit codes (one word) -> 4 registers of e4m3 bytes: register q holds, in byte t,
// code 4t + q.  Registers with q odd keep the code where it sits, in bits 2..3 of the byte: the
// e4m3 byte 4c, the value 4c * 2^-9 (e4m3 bytes 0..15 are the values 0..15 times 2^-9).  Their
// filter bytes are +-0.25 instead of +-1 (prep_weights_kernel), so every product is still c * 2^-9
// exactly, and one shift by 4 serves all four registers: five ALU instructions per word instead of
// seven.
__device__ __forceinline__ void expand2w(uint32_t w, uint32_t* o) {
  const uint32_t h = w >> 4;
  o[0] = w & 0x03030303u;
  o[1] = w & 0x0C0C0C0Cu;
  o[2] = h & 0x03030303u;
  o[3] = h & 0x0C0C0C0Cu;
}

// 64 packed two-bit codes -> 16 registers (register 4j+q from word j, as expand2w).
__device__ __forceinline__ void expand2(uint4 v, uint32_t* o) {
  expand2w(v.x, o);
  expand2w(v.y, o + 4);
  expand2w(v.z, o + 8);
  expand2w(v.w, o + 12);
}

// 8 registers -> 8 consecutive tensor-memory columns of this warp's 32 lanes, with the wait for the
// store in the same asm statement (the store reads its source registers asynchronously).
__device__ __forceinline__ void tmem_st8_sync(uint32_t taddr, const uint32_t* o) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};\n\t"
      "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
      "r"(o[0]), "r"(o[1]), "r"(o[2]), "r"(o[3]), "r"(o[4]), "r"(o[5]), "r"(o[6]), "r"(o[7])
      : "memory");
}

// 64 four-bit codes (two 16-byte units, 8 words) -> 16 registers of e4m3 bytes: word j of the 8
// gives register 2j (its codes 0, 2, 4, 6 as bytes 0..3) and register 2j+1 (codes 1, 3, 5, 7).
// A code c in 0..15 is the e4m3 byte c, the value c * 2^-9 (0..7 subnormal, 8..15 with exponent
// field 1).
__device__ __forceinline__ void expand4(uint4 a, uint4 b, uint32_t* o) {
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    o[2 * j] = w[j] & 0x0F0F0F0Fu;
    o[2 * j + 1] = (w[j] >> 4) & 0x0F0F0F0Fu;
  }
}

}  // namespace ifq
