// Warp-level tensor-core path for the narrow 3x3 layers at the start of a network: few input
// channels (8 or 16 two-bit codes, or the 8-bit image with 4 channels) and few output channels
// (8, 16 or 32), usually followed by a 2 x 2 max pool (Sec. 4.2's Tiny-YOLO / Tinier-YOLO
// backbones).  Eq. (1) as an implicit GEMM on mma.sync.m16n8k32 e4m3 -> f32: M = 16 output pixels of
// one row, N = 8 output channels, K = the 3 x 3 window; then the pool on the accumulators and the
// integer thresholds of Eq. (7).
//
// Why a warp-level MMA here.  These layers have 8-32 output channels: a 128 x N tcgen05 tile is
// mostly padding or Toeplitz zeros, and the tensor-memory round trip makes their epilogue (the
// thresholds of every output value) the bottleneck.  m16n8k32 returns the accumulators in registers
// in a 16-pixel x 8-channel shape, the 2 x 2 pool happens in registers before any threshold, and
// the MMA rate is far above what these layers need.
//
// Exactness.  A code c is the e4m3 byte c, i.e. c * 2^-9 (subnormal below 8, exponent field 1 from
// 8 to 15), a +1 / -1 weight is 0x38 / 0xB8, so every product is an exact multiple of 2^-9.  An
// 8-bit input value v is its two 4-bit fields: the low one with weight +-1 and the high one with
// weight +-16 (0x58 / 0xD8), so the two products add to v * w * 2^-9.  The f32 accumulation of
// these products was measured exact on GB300 up to 2^24 units of 2^-9, both for the accumulator
// input plus a product and for the sum inside one instruction; the layers admitted here stay below
// 255 * 36 = 9180 units, so D = A / 512 exactly.
//
// K order.  For filter row dy, the 3 taps x E bytes of a pixel (E = 8: 8 codes, or the 4 low then
// the 4 high fields of 4 8-bit values; E = 16: 16 codes) are cut into 8-byte pieces j = 0 .. 3E/8-1
// (tap j / (E/8), byte 8 (j % (E/8)) of that pixel).  K step s of the row gives lane t piece
// j = 4 s + t: its A registers a0 / a2 are that piece's two words for pixel row g, a1 / a3 for pixel
// row g + 8, and its B registers hold the weights of channel g at the same bytes.  Pieces past 3E/8
// have zero weights.  The A fragment is therefore two 8-byte shared-memory loads, which no two lanes
// of a half-warp make to the same bank pair.
//
// Work.  Persistent CTAs take bands of `rb` output rows of one image in turn.  The copy engine
// brings a band's input rows (one contiguous bulk copy: the rows of an image are consecutive in
// NHWC) into one of two raw buffers while the CTA computes the previous band; the CTA then expands
// them in shared memory into e4m3 bytes, with a zero halo of one pixel on each side and zero rows
// outside the image.  A warp takes (16-pixel strip, output row pair) items of the band: it loads the
// A fragments of the 4 input rows the pair reads, issues 3 filter rows x K steps x channel tiles
// MMAs per output row, and runs the epilogue.  With the fused pool the vertical pair is in the same
// thread, and the horizontal pair is one shuffle away (pixel rows g and g ^ 1 of the fragment).
// Rows that are not a whole number of 16-byte units (no bulk copy) are expanded straight from
// global memory instead.  Every wait is bounded (IFQ_ETIMEOUT; the CTA then waits, bounded, for
// the copies it issued and returns).
#pragma once
#include <cstdint>

#include "conv_common.cuh"   // FastDiv
#include "ptx.cuh"

namespace ifq {

// Threads and resident CTAs per SM of an instance: the 16-byte, 32-channel one keeps 48 registers of
// filter fragments and 32 of accumulators, so it runs 4 warps a CTA, 3 CTAs an SM.
__host__ __device__ constexpr int warp_conv_threads(int E, int NT) { return E * NT >= 64 ? 128 : 256; }
__host__ __device__ constexpr int warp_conv_min_ctas(int E, int NT) { return E * NT >= 64 ? 2 : 2; }

struct WarpConvArgs {
  const uint8_t* x;        // 2-bit codes [n][h][w][cin / 4] bytes, or 8-bit values [n][h][w][cin]
  const uint32_t* wbits;   // sign words [cout][kwords]: bit k of filter n set = +1 at K position k ((dy, dx, c))
  const int32_t* thr;      // [cout][3] or nullptr (accumulators only)
  const int8_t* sign;      // [cout]
  uint8_t* y_codes;        // [n][pho][pwo][cout / 4] packed codes, or nullptr
  int32_t* y_acc;          // [n][h][w][cout] int32 (no pool), or nullptr
  int n, h, w, cin, cout, kwords;
  int pho, pwo;            // output shape after the fused pool (h, w without one)
  int strips;              // 16-pixel strips covering a row
  int rb;                  // output rows per band (even)
  int bands;               // bands per image
  int row_bytes;           // shared-memory bytes of one staged row: (16 strips + 2) pixels x E
  int units;               // (strip, output row pair) items of a band
  int bulk;                // input rows of whole 16-byte units: staged by the copy engine
  int raw_pitch;           // input bytes per row (w x input bytes per pixel)
  int total;               // bands of the whole batch: n x bands
  FastDiv div_bands, div_strips, div_slots;
};

// Shared-memory layout of an instance: filter fragments, thresholds, the expanded band, two raw
// row buffers (copy-engine staging) and their two mbarriers.
struct WarpSmem {
  uint32_t b_off, t_off, band_off, raw_off, raw_bytes, bar_off, bytes;
};
__host__ __device__ inline WarpSmem warp_smem(int nb, int cout, int rb, int row_bytes, int raw_pitch, int bulk) {
  WarpSmem m;
  m.b_off = 0;
  m.t_off = (uint32_t)nb * 256u;
  m.band_off = m.t_off + (uint32_t)cout * 16u;
  m.raw_off = m.band_off + (uint32_t)((rb + 2) * row_bytes + 15) / 16u * 16u;
  m.raw_bytes = bulk ? (uint32_t)((rb + 2) * raw_pitch + 15) / 16u * 16u : 0u;
  m.bar_off = m.raw_off + 2u * m.raw_bytes;
  m.bytes = m.bar_off + 16u;
  return m;
}

__device__ __forceinline__ void mma_e4m3_16832(float (&d)[4], const uint32_t (&a)[4], uint2 b) {
  asm volatile(
      "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b.x), "r"(b.y));
}

// 8 two-bit codes (one 16-bit field) -> 8 e4m3 bytes; byte i of the result is code i.
__device__ __forceinline__ uint32_t spread4(uint32_t b) {   // b: 4 codes in 8 bits
  uint32_t t = (b | (b << 12)) & 0x000F000Fu;
  return (t | (t << 6)) & 0x03030303u;
}

// The 2-bit code of f = A / 512 against the channel's thresholds (ascending, in the same domain),
// flipped (c ^ 3) for a channel with a negative BN scale: th.w holds the flip bits.
__device__ __forceinline__ uint32_t warp_code(float f, float4 th) {
  const uint32_t c = (uint32_t)(f > th.x) + (uint32_t)(f > th.y) + (uint32_t)(f > th.z);
  return c ^ __float_as_uint(th.w);
}

// E: staged bytes per pixel (8 or 16); NT: 8-channel tiles (cout = 8 NT); POOL: 1 or 2; IN8: 8-bit input.
template <int E, int NT, int POOL, int IN8>
__global__ void __launch_bounds__(warp_conv_threads(E, NT), warp_conv_min_ctas(E, NT))
    conv_warp_kernel(const WarpConvArgs a) {
  constexpr int kThreads = warp_conv_threads(E, NT);
  constexpr int PP = E / 8;                 // 8-byte pieces per pixel
  constexpr int NJ = 3 * PP;                // pieces per filter row
  constexpr int KSD = (NJ + 3) / 4;         // K steps per filter row
  constexpr int NB = NT * 3 * KSD;          // B fragments per lane
  constexpr int NW = NT >= 2 ? NT / 2 : 1;  // 32-bit words of codes per output pixel (16 bits when NT = 1)
  static_assert(E == 8 || E == 16, "staged pixel of 8 or 16 bytes");
  static_assert(!IN8 || E == 8, "8-bit input: 4 channels, two fields each");
  extern __shared__ __align__(16) uint8_t smem[];
  const WarpSmem L = warp_smem(NB, a.cout, a.rb, a.row_bytes, a.raw_pitch, a.bulk);
  uint2* sB = reinterpret_cast<uint2*>(smem + L.b_off);      // [NB][32 lanes]
  float4* sT = reinterpret_cast<float4*>(smem + L.t_off);    // [cout]
  uint8_t* band = smem + L.band_off;                         // [rb + 2][row_bytes]
  uint8_t* raw = smem + L.raw_off;                           // [2][rb + 2][raw_pitch]
  const uint32_t bar0 = smem_u32(smem + L.bar_off);          // raw buffer s is full: bar0 + 8 s
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, t = lane & 3;

  if (tid == 0 && a.bulk) {
    mbar_init(bar0, 1);
    mbar_init(bar0 + 8, 1);
    fence_mbar_init();
  }
  grid_dep_launch();
  grid_dep_wait();   // the input (and, for a first layer, the prepared filters) come from earlier kernels

  // B fragments: entry ((jn * 3 + dy) * KSD + s) of lane (gl, tl) holds the weights of channel
  // 8 jn + gl at piece 4 s + tl of filter row dy, as 8 e4m3 bytes.
  for (int i = tid; i < NB * 64; i += kThreads) {
    const int e = i >> 6, l = (i >> 1) & 31, half = i & 1;
    const int s = e % KSD, dy = (e / KSD) % 3, jn = e / (3 * KSD);
    const int n = 8 * jn + (l >> 2), j = 4 * s + (l & 3);
    uint32_t word = 0;
    if (j < NJ) {
      const int dx = j / PP, off = 8 * (j % PP) + 4 * half;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int p = off + q;                              // byte within the staged pixel
        const int c = IN8 ? (p & 3) : p;                    // input channel
        const bool hi = IN8 && p >= 4;
        const int k = (dy * 3 + dx) * a.cin + c;
        const bool plus = (a.wbits[(size_t)n * a.kwords + (k >> 5)] >> (k & 31)) & 1u;
        const uint32_t byte = plus ? (hi ? 0x58u : 0x38u) : (hi ? 0xD8u : 0xB8u);
        word |= byte << (8 * q);
      }
    }
    reinterpret_cast<uint32_t*>(sB)[i] = word;
  }
  // thresholds in the domain of D = A / 512; a negative BN scale: ascending (-T - 1) / 512, flip 3
  for (int n = tid; n < a.cout; n += kThreads) {
    float4 th = make_float4(0.f, 0.f, 0.f, __uint_as_float(0u));
    if (a.thr) {
      const int32_t T0 = a.thr[3 * n], T1 = a.thr[3 * n + 1], T2 = a.thr[3 * n + 2];
      if (a.sign[n] >= 0) {
        th = make_float4((float)T0 * (1.0f / 512.0f), (float)T1 * (1.0f / 512.0f), (float)T2 * (1.0f / 512.0f),
                         __uint_as_float(0u));
      } else {
        th = make_float4((float)(-T2 - 1) * (1.0f / 512.0f), (float)(-T1 - 1) * (1.0f / 512.0f),
                         (float)(-T0 - 1) * (1.0f / 512.0f), __uint_as_float(3u));
      }
    }
    sT[n] = th;
  }
  __syncthreads();

  uint2 bf[NB];
#pragma unroll
  for (int e = 0; e < NB; ++e) bf[e] = sB[e * 32 + lane];
  // this lane's pieces: pixel offset (tap) and byte offset of piece 4 s + t
  int poff[KSD];
#pragma unroll
  for (int s = 0; s < KSD; ++s) {
    const int j = 4 * s + t;
    poff[s] = j < NJ ? (j / PP) * E + 8 * (j % PP) : 0;   // zero-weight pieces read tap 0
  }
  constexpr int nwarps = kThreads / 32;
  const int rowb = a.cout >> 2;                  // output bytes per pixel
  const int cinb = IN8 ? a.cin : a.cin / 4;      // input bytes per pixel
  const int slots = 16 * a.strips + 2;

  // the copy of band blk's input rows (those inside the image, one contiguous range) into raw
  // buffer s, completing on its mbarrier; raw row r is input row y0 - 1 + r
  auto issue = [&](int blk, int s) {
    const int bb = (int)fdiv((uint32_t)blk, a.div_bands), yy0 = (blk - bb * a.bands) * a.rb;
    const int r0 = max(0, yy0 - 1), r1 = min(a.h, yy0 + a.rb + 1);
    const uint32_t bytes = (uint32_t)((r1 - r0) * a.raw_pitch);
    const uint32_t bar = bar0 + 8u * (uint32_t)s;
    mbar_arrive_expect_tx(bar, bytes);
    bulk_copy_g2s(smem_u32(raw + (size_t)s * L.raw_bytes + (size_t)(r0 - (yy0 - 1)) * a.raw_pitch),
                  a.x + ((size_t)bb * a.h + r0) * a.raw_pitch, bytes, bar);
  };
  // staged row r of the band: input row y0 - 1 + r as e4m3 bytes, slot q = pixel q - 1, zero outside
  // the image; `row(r)` is the input row's first byte (shared or global memory)
  auto expand = [&](int y0, auto row) {
    const int total = (a.rb + 2) * slots;
    for (int i = tid; i < total; i += kThreads) {
      const int r = (int)fdiv((uint32_t)i, a.div_slots), q = i - r * slots;
      const int iy = y0 - 1 + r, ix = q - 1;
      const bool in = iy >= 0 && iy < a.h && ix >= 0 && ix < a.w;
      uint8_t* dst = band + (size_t)r * a.row_bytes + (size_t)q * E;
      const uint8_t* src = in ? row(r) + (size_t)ix * cinb : nullptr;
      if constexpr (IN8) {
        const uint32_t v = in ? *reinterpret_cast<const uint32_t*>(src) : 0u;
        *reinterpret_cast<uint2*>(dst) = make_uint2(v & 0x0F0F0F0Fu, (v >> 4) & 0x0F0F0F0Fu);
      } else if constexpr (E == 8) {
        const uint32_t v = in ? (uint32_t)*reinterpret_cast<const uint16_t*>(src) : 0u;
        *reinterpret_cast<uint2*>(dst) = make_uint2(spread4(v & 0xFFu), spread4(v >> 8));
      } else {
        const uint32_t v = in ? *reinterpret_cast<const uint32_t*>(src) : 0u;
        *reinterpret_cast<uint4*>(dst) =
            make_uint4(spread4(v & 0xFFu), spread4((v >> 8) & 0xFFu), spread4((v >> 16) & 0xFFu), spread4(v >> 24));
      }
    }
  };

  int issued = 0, waited = 0;   // bands whose copies thread 0 issued / this thread saw complete
  if (a.bulk && tid == 0 && (int)blockIdx.x < a.total) {
    issue((int)blockIdx.x, 0);
    issued = 1;
  }
  int it = 0;
#pragma unroll 1
  for (int blk = (int)blockIdx.x; blk < a.total; blk += (int)gridDim.x, ++it) {
    const int b = (int)fdiv((uint32_t)blk, a.div_bands);
    const int y0 = (blk - b * a.bands) * a.rb;
    if (a.bulk) {
      // the next band's copy into the other buffer (read by the expansion before the last barrier)
      if (tid == 0 && blk + (int)gridDim.x < a.total) {
        issue(blk + (int)gridDim.x, (it + 1) & 1);
        ++issued;
      }
      const bool ok = mbar_wait(bar0 + 8u * (uint32_t)(it & 1), (uint32_t)(it >> 1) & 1u);
      if (ok) waited = it + 1;
      if (__syncthreads_or(!ok)) break;
      const uint8_t* rbuf = raw + (size_t)(it & 1) * L.raw_bytes;
      expand(y0, [&](int r) { return rbuf + (size_t)r * a.raw_pitch; });
    } else {
      expand(y0, [&](int r) { return a.x + ((size_t)b * a.h + (y0 - 1 + r)) * a.raw_pitch; });
    }
    __syncthreads();

#pragma unroll 1
    for (int u = warp; u < a.units; u += nwarps) {
      const int yp = (int)fdiv((uint32_t)u, a.div_strips), sx = u - yp * a.strips;
      const int y = y0 + 2 * yp;   // output rows y, y + 1
      if (y >= a.h) continue;      // warp-uniform
      const int x0 = 16 * sx;
      float acc[2][NT][4];
#pragma unroll
      for (int m = 0; m < 2; ++m)
#pragma unroll
        for (int jn = 0; jn < NT; ++jn)
#pragma unroll
          for (int q = 0; q < 4; ++q) acc[m][jn][q] = 0.f;
      const uint8_t* base = band + (size_t)(2 * yp) * a.row_bytes + (size_t)(x0 + g) * E;
#pragma unroll
      for (int r = 0; r < 4; ++r) {   // staged row 2 yp + r: filter row r of output row y, r - 1 of y + 1
        uint32_t af[KSD][4];
#pragma unroll
        for (int s = 0; s < KSD; ++s) {
          const uint8_t* p = base + (size_t)r * a.row_bytes + poff[s];
          const uint2 lo = *reinterpret_cast<const uint2*>(p);
          const uint2 hi = *reinterpret_cast<const uint2*>(p + 8 * E);
          af[s][0] = lo.x; af[s][1] = hi.x; af[s][2] = lo.y; af[s][3] = hi.y;
        }
#pragma unroll
        for (int m = 0; m < 2; ++m) {
          const int dy = r - m;
          if (dy < 0 || dy > 2) continue;
#pragma unroll
          for (int s = 0; s < KSD; ++s)
#pragma unroll
            for (int jn = 0; jn < NT; ++jn) mma_e4m3_16832(acc[m][jn], af[s], bf[(jn * 3 + dy) * KSD + s]);
        }
      }

      if constexpr (POOL == 2) {
        // pooled pixel of this lane: even g pools pixels (g, g + 1), odd g pools (g + 7, g + 8)
        const bool odd = (g & 1) != 0;
        const int py = y >> 1, px = (x0 >> 1) + (g >> 1) + (odd ? 4 : 0);
        uint32_t words[NW];
#pragma unroll
        for (int i = 0; i < NW; ++i) words[i] = 0;
#pragma unroll
        for (int jn = 0; jn < NT; ++jn) {
          const float v0 = fmaxf(acc[0][jn][0], acc[1][jn][0]), v1 = fmaxf(acc[0][jn][1], acc[1][jn][1]);
          const float v2 = fmaxf(acc[0][jn][2], acc[1][jn][2]), v3 = fmaxf(acc[0][jn][3], acc[1][jn][3]);
          const float r0 = __shfl_xor_sync(0xffffffffu, odd ? v0 : v2, 4);
          const float r1 = __shfl_xor_sync(0xffffffffu, odd ? v1 : v3, 4);
          const float p0 = fmaxf(odd ? v2 : v0, r0), p1 = fmaxf(odd ? v3 : v1, r1);
          const int n0 = 8 * jn + 2 * t;
          const uint32_t c = warp_code(p0, sT[n0]) | (warp_code(p1, sT[n0 + 1]) << 2);
          words[jn >> 1] |= c << (16 * (jn & 1) + 4 * t);
        }
#pragma unroll
        for (int i = 0; i < NW; ++i) {
          words[i] |= __shfl_xor_sync(0xffffffffu, words[i], 1);
          words[i] |= __shfl_xor_sync(0xffffffffu, words[i], 2);
        }
        if (a.y_codes && py < a.pho && px < a.pwo) {
          uint8_t* dst = a.y_codes + (((size_t)b * a.pho + py) * a.pwo + px) * rowb;
          if constexpr (NT == 1) {
            if (t == 0) *reinterpret_cast<uint16_t*>(dst) = (uint16_t)words[0];
          } else {
#pragma unroll
            for (int i = 0; i < NW; ++i)
              if (t == i) *reinterpret_cast<uint32_t*>(dst + 4 * i) = words[i];
          }
        }
      } else {
#pragma unroll
        for (int m = 0; m < 2; ++m) {
          const int yy = y + m;
          if (yy >= a.h) continue;   // warp-uniform
          uint32_t wg[NW], wh[NW];   // codes of pixels x0 + g and x0 + g + 8
#pragma unroll
          for (int i = 0; i < NW; ++i) wg[i] = wh[i] = 0;
#pragma unroll
          for (int jn = 0; jn < NT; ++jn) {
            const int n0 = 8 * jn + 2 * t;
            if (a.y_acc) {
              int32_t* da = a.y_acc + (((size_t)b * a.h + yy) * a.w + x0 + g) * a.cout + n0;
              if (x0 + g < a.w)
                *reinterpret_cast<int2*>(da) = make_int2(__float2int_rn(acc[m][jn][0] * 512.0f),
                                                         __float2int_rn(acc[m][jn][1] * 512.0f));
              if (x0 + g + 8 < a.w)
                *reinterpret_cast<int2*>(da + 8 * a.cout) = make_int2(__float2int_rn(acc[m][jn][2] * 512.0f),
                                                                      __float2int_rn(acc[m][jn][3] * 512.0f));
            }
            const float4 t0 = sT[n0], t1 = sT[n0 + 1];
            const int sh = 16 * (jn & 1) + 4 * t;
            wg[jn >> 1] |= (warp_code(acc[m][jn][0], t0) | (warp_code(acc[m][jn][1], t1) << 2)) << sh;
            wh[jn >> 1] |= (warp_code(acc[m][jn][2], t0) | (warp_code(acc[m][jn][3], t1) << 2)) << sh;
          }
          if (!a.y_codes) continue;
#pragma unroll
          for (int i = 0; i < NW; ++i) {
            wg[i] |= __shfl_xor_sync(0xffffffffu, wg[i], 1);
            wg[i] |= __shfl_xor_sync(0xffffffffu, wg[i], 2);
            wh[i] |= __shfl_xor_sync(0xffffffffu, wh[i], 1);
            wh[i] |= __shfl_xor_sync(0xffffffffu, wh[i], 2);
          }
          uint8_t* dst = a.y_codes + (((size_t)b * a.h + yy) * a.w + x0 + g) * rowb;
          const bool okg = x0 + g < a.w, okh = x0 + g + 8 < a.w;
          if constexpr (NT == 1) {
            if (t == 0 && okg) *reinterpret_cast<uint16_t*>(dst) = (uint16_t)wg[0];
            if (t == 0 && okh) *reinterpret_cast<uint16_t*>(dst + 8 * rowb) = (uint16_t)wh[0];
          } else {
#pragma unroll
            for (int i = 0; i < NW; ++i) {
              if (t == i && okg) *reinterpret_cast<uint32_t*>(dst + 4 * i) = wg[i];
              if (t == i && okh) *reinterpret_cast<uint32_t*>(dst + 8 * rowb + 4 * i) = wh[i];
            }
          }
        }
      }
    }
    __syncthreads();   // the band and this raw buffer are free again
  }
  // after a timeout: wait (bounded) for the copies thread 0 issued that nobody saw complete
  if (a.bulk && tid == 0)
    for (int k = waited; k < issued; ++k) mbar_wait(bar0 + 8u * (uint32_t)(k & 1), (uint32_t)(k >> 1) & 1u);
}

}  // namespace ifq
