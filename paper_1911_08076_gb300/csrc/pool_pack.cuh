// Max pooling of packed codes (Sec. 2.1 placement, on codes with channel signs)
// and the packing / filter-preparation kernels.
#pragma once
#include <cstdint>

#include "conv_common.cuh"   // FastDiv

namespace ifq {

// ---------------------------------------------------------------- pooling
//
// Channel c of a pixel is the SB-bit field c % (8/SB) of byte c / (8/SB) (SB = 2,
// or 4 for 3- and 4-bit codes).  With a channel sign of -1 the pool takes the
// min of the codes; with F = 2^SB - 1, min(a, b) = F - max(F-a, F-b) and
// F - x = x ^ F on an SB-bit field, so flipping those fields (XOR with a
// per-channel mask), taking a plain field-wise max, and flipping back gives
// both cases with one max.

// Field-wise max of two packed words.  2-bit fields (h1 h0): the larger high bit wins, and equal
// high bits take the OR of the low bits; 4-bit fields: a byte-lane max on the low and on the high
// nibbles (each masked in place, so no shifts).
template <int SB>
__device__ __forceinline__ uint32_t field_max(uint32_t a, uint32_t b) {
  if constexpr (SB == 2) {
    const uint32_t a1 = a & 0xAAAAAAAAu, b1 = b & 0xAAAAAAAAu;
    const uint32_t ga = (a1 & ~b1) >> 1, gb = (b1 & ~a1) >> 1;   // where a (b) has the larger high bit
    return a1 | b1 | (((a & ~gb) | (b & ~ga)) & 0x55555555u);
  } else {
    return __vmaxu4(a & 0x0F0F0F0Fu, b & 0x0F0F0F0Fu) | __vmaxu4(a & 0xF0F0F0F0u, b & 0xF0F0F0F0u);
  }
}

// mask of the N fields of channels c0 .. c0+N-1: all ones in the fields of sign -1 channels
template <int SB, int N>
__device__ __forceinline__ uint32_t flip_mask(const int8_t* sign, int c0, int c) {
  if (!sign) return 0u;
  uint32_t m = 0;
#pragma unroll
  for (int j = 0; j < N; ++j)
    if (c0 + j < c && sign[c0 + j] < 0) m |= ((1u << SB) - 1u) << (SB * j);
  return m;
}

struct PoolArgs {
  const uint8_t* x;
  const int8_t* sign;
  uint8_t* y;
  int n, h, w, c, k, stride, pad, ho, wo;
  int groups;                          // vector groups (of U words or of single bytes) per pixel
  int total;                           // n * ho * wo * groups (< 2^31)
  FastDiv div_groups, div_wo, div_ho;
  int wq;                              // 2x2 row-pair kernel: items per output row
  FastDiv div_wq;
};

template <int U>
struct WordVec;
template <>
struct WordVec<1> {
  static __device__ __forceinline__ void ld(const uint32_t* p, uint32_t* v) { v[0] = __ldg(p); }
  static __device__ __forceinline__ void st(uint32_t* p, const uint32_t* v) { p[0] = v[0]; }
};
template <>
struct WordVec<2> {
  static __device__ __forceinline__ void ld(const uint32_t* p, uint32_t* v) {
    const uint2 q = __ldg((const uint2*)p);
    v[0] = q.x; v[1] = q.y;
  }
  static __device__ __forceinline__ void st(uint32_t* p, const uint32_t* v) { *(uint2*)p = make_uint2(v[0], v[1]); }
};
template <>
struct WordVec<4> {
  static __device__ __forceinline__ void ld(const uint32_t* p, uint32_t* v) {
    const uint4 q = __ldg((const uint4*)p);
    v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
  }
  static __device__ __forceinline__ void st(uint32_t* p, const uint32_t* v) {
    *(uint4*)p = make_uint4(v[0], v[1], v[2], v[3]);
  }
};

// U = 32-bit words handled per thread (4, 2 or 1, one vector load per window cell); needs the
// packed bytes of a pixel to be a multiple of 4U.  Item it = pixel * groups + group.  KW = 2 or 3:
// the k x k window (k == KW) is loaded before it is reduced, so all its loads are in flight
// together; the top-left cell (oy*stride, ox*stride) is always inside the image, and a cell past
// the bottom or right edge takes its value (a no-op for the max).  KW = 0: any k, cell by cell.
// When the grid stride is a multiple of the groups per pixel, a thread's group never changes and
// its sign masks are built once.
template <int U, int SB, int KW>
__global__ void __launch_bounds__(256) maxpool_codes_kernel(const PoolArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  constexpr int kCpw = 32 / SB;             // codes per word
  const int cw = a.c / kCpw;                // 32-bit words per pixel
  const size_t rowb = (size_t)a.w * (cw * 4);
  const int stride = gridDim.x * blockDim.x;
  const bool fixed_group = stride % a.groups == 0;
  int mask_g = -1;
  uint32_t mask[U];
  for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < a.total; it += stride) {
    const int pix = (int)fdiv((uint32_t)it, a.div_groups);
    const int gi = it - pix * a.groups;
    const int t = (int)fdiv((uint32_t)pix, a.div_wo);
    const int ox = pix - t * a.wo;
    const int b = (int)fdiv((uint32_t)t, a.div_ho);
    const int oy = t - b * a.ho;
    if (gi != mask_g) {
#pragma unroll
      for (int u = 0; u < U; ++u) mask[u] = flip_mask<SB, kCpw>(a.sign, (gi * U + u) * kCpw, a.c);
      mask_g = fixed_group ? gi : -1;
    }
    const int iy0 = oy * a.stride, ix0 = ox * a.stride;
    const uint8_t* base = a.x + ((size_t)b * a.h + iy0) * rowb + (size_t)ix0 * (cw * 4) + (size_t)gi * (U * 4);
    uint32_t m[U];                           // the window max of the flipped fields
    if constexpr (KW > 0) {
      uint32_t v[KW * KW][U];
      WordVec<U>::ld((const uint32_t*)base, v[0]);
#pragma unroll
      for (int q = 1; q < KW * KW; ++q) {
        const int dy = q / KW, dx = q % KW;
        if (iy0 + dy < a.h && ix0 + dx < a.w) {
          WordVec<U>::ld((const uint32_t*)(base + dy * rowb + (size_t)dx * (cw * 4)), v[q]);
        } else {
#pragma unroll
          for (int u = 0; u < U; ++u) v[q][u] = v[0][u];
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        m[u] = v[0][u] ^ mask[u];
#pragma unroll
        for (int q = 1; q < KW * KW; ++q) m[u] = field_max<SB>(m[u], v[q][u] ^ mask[u]);
      }
    } else {
      bool first = true;
      for (int dy = 0; dy < a.k; ++dy) {
        if (iy0 + dy >= a.h) continue;
        for (int dx = 0; dx < a.k; ++dx) {
          if (ix0 + dx >= a.w) continue;
          uint32_t v[U];
          WordVec<U>::ld((const uint32_t*)(base + dy * rowb + (size_t)dx * (cw * 4)), v);
#pragma unroll
          for (int u = 0; u < U; ++u) m[u] = first ? v[u] ^ mask[u] : field_max<SB>(m[u], v[u] ^ mask[u]);
          first = false;
        }
      }
    }
    uint32_t* dst = (uint32_t*)(a.y + (size_t)pix * (cw * 4)) + gi * U;
#pragma unroll
    for (int u = 0; u < U; ++u) m[u] ^= mask[u];
    WordVec<U>::st(dst, m);
  }
}

// 2x2 / stride 2 pool without padding on narrow pixels of PB = 4 or 8 packed bytes.  An item is
// the 16 contiguous bytes of input row 2*oy under P = 16 / (2 PB) adjacent output pixels (2 P input
// pixels) and the same 16 bytes of row 2*oy + 1: two 128-bit loads and one 64-bit store, where the
// general kernel issues a 4- or 8-byte load per window cell.  Each thread takes two items per
// round (four loads in flight); the loads are streaming (evict-first: each input byte is read once).
// Needs w * PB % 16 == 0 and wo % P == 0 (checked by the host); every cell is inside the image
// because ho = h / 2 and wo = w / 2 (floor).
template <int SB, int PB>
__global__ void __launch_bounds__(256) maxpool2x2_rowpair_kernel(const PoolArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  constexpr int kCpw = 32 / SB;             // codes per word
  constexpr int kP = 16 / (2 * PB);         // output pixels per item
  static_assert(PB == 4 || PB == 8, "pixel bytes");
  // flip masks of the pixel's words (one word for PB = 4, two for PB = 8)
  const uint32_t m0 = flip_mask<SB, kCpw>(a.sign, 0, a.c);
  const uint32_t m1 = PB == 8 ? flip_mask<SB, kCpw>(a.sign, kCpw, a.c) : m0;
  const size_t rowb = (size_t)a.w * PB;
  // item it: output row t = (b, oy), segment q; returns the first input byte of the segment
  auto src = [&](int it, int& t, int& q) {
    t = (int)fdiv((uint32_t)it, a.div_wq);
    q = it - t * a.wq;
    const int b = (int)fdiv((uint32_t)t, a.div_ho);
    const int oy = t - b * a.ho;
    return a.x + ((size_t)b * a.h + 2 * oy) * rowb + (size_t)q * 16;
  };
  auto max4 = [](uint32_t p, uint32_t q, uint32_t r, uint32_t u, uint32_t m) {
    return field_max<SB>(field_max<SB>(p ^ m, q ^ m), field_max<SB>(r ^ m, u ^ m)) ^ m;
  };
  auto reduce_store = [&](const uint4& r0, const uint4& r1, int t, int q) {
    uint2 o;
    if constexpr (PB == 8) {   // input pixels (x, y) and (z, w) -> one output pixel of two words
      o.x = max4(r0.x, r0.z, r1.x, r1.z, m0);
      o.y = max4(r0.y, r0.w, r1.y, r1.w, m1);
    } else {                   // input pixels x, y -> output pixel 2q; z, w -> 2q + 1
      o.x = max4(r0.x, r0.y, r1.x, r1.y, m0);
      o.y = max4(r0.z, r0.w, r1.z, r1.w, m0);
    }
    *(uint2*)(a.y + ((size_t)t * a.wo + (size_t)q * kP) * PB) = o;
  };
  const int gs = gridDim.x * blockDim.x;
  int it = blockIdx.x * blockDim.x + threadIdx.x;
  for (; it + gs < a.total; it += 2 * gs) {   // items it and it + gs
    int t0, q0, t1, q1;
    const uint8_t* p0 = src(it, t0, q0);
    const uint8_t* p1 = src(it + gs, t1, q1);
    const uint4 a0 = __ldcs((const uint4*)p0), b0 = __ldcs((const uint4*)(p0 + rowb));
    const uint4 a1 = __ldcs((const uint4*)p1), b1 = __ldcs((const uint4*)(p1 + rowb));
    reduce_store(a0, b0, t0, q0);
    reduce_store(a1, b1, t1, q1);
  }
  if (it < a.total) {
    int t, q;
    const uint8_t* p = src(it, t, q);
    reduce_store(__ldcs((const uint4*)p), __ldcs((const uint4*)(p + rowb)), t, q);
  }
}

// byte-granular variant for any c % 4 == 0
template <int SB>
__global__ void __launch_bounds__(256) maxpool_codes_bytes_kernel(const PoolArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  constexpr int kCpb = 8 / SB;
  const int cb = a.c / kCpb;
  for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < a.total; it += gridDim.x * blockDim.x) {
    const int pix = (int)fdiv((uint32_t)it, a.div_groups);
    const int bi = it - pix * cb;
    const int t = (int)fdiv((uint32_t)pix, a.div_wo);
    const int ox = pix - t * a.wo;
    const int b = (int)fdiv((uint32_t)t, a.div_ho);
    const int oy = t - b * a.ho;
    const uint32_t mask = flip_mask<SB, kCpb>(a.sign, bi * kCpb, a.c);
    uint32_t m = 0;
    bool first = true;
    for (int dy = 0; dy < a.k; ++dy) {
      const int iy = oy * a.stride + dy;
      if (iy >= a.h) continue;
      for (int dx = 0; dx < a.k; ++dx) {
        const int ix = ox * a.stride + dx;
        if (ix >= a.w) continue;
        const uint32_t v = a.x[(((size_t)b * a.h + iy) * a.w + ix) * cb + bi];
        m = first ? v ^ mask : field_max<SB>(m, v ^ mask);
        first = false;
      }
    }
    a.y[(size_t)pix * cb + bi] = (uint8_t)((m ^ mask) & 0xFFu);
  }
}

// ---------------------------------------------------------------- fixed-point output

// y = floor((mul[n] * A + add[n]) / 2^m) for item i = r * cout + n (the separated conversion of a
// non-quantized substructure's output, Sec. 2.2), in 128-bit integers, saturated to int32.
__global__ void fixed_output_kernel(const int32_t* acc, int total, FastDiv div_cout, const int64_t* mul,
                                    const int64_t* add, int m, int32_t* y) {
  grid_dep_launch();
  grid_dep_wait();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
    const int r = (int)fdiv((uint32_t)i, div_cout);
    const int n = i - r * (int)div_cout.d;
    const __int128 v = (__int128)mul[n] * acc[i] + add[n];
    const __int128 q = v >> m;   // arithmetic shift: the floor of v / 2^m
    y[i] = q > (__int128)INT32_MAX ? INT32_MAX : (q < (__int128)INT32_MIN ? INT32_MIN : (int32_t)q);
  }
}

// ---------------------------------------------------------------- packing

// 16-byte vector copy on the SMs (either side may be host memory the device addresses directly:
// pinned host memory under unified addressing, read or written over the CPU-GPU link).
__global__ void copy16_kernel(const uint4* src, uint4* dst, size_t n16) {
  grid_dep_launch();
  grid_dep_wait();
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += (size_t)gridDim.x * blockDim.x)
    dst[i] = src[i];
}


// one code per byte <-> SB-bit fields, 8/SB codes per packed byte (codes keep their low SB bits)
template <int SB>
__global__ void pack_codes_kernel(const uint8_t* codes, uint8_t* packed, size_t nbytes) {
  constexpr int kCpb = 8 / SB;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nbytes; i += (size_t)gridDim.x * blockDim.x) {
    uint32_t v = 0;
#pragma unroll
    for (int l = 0; l < kCpb; ++l) v |= ((uint32_t)codes[kCpb * i + l] & ((1u << SB) - 1u)) << (SB * l);
    packed[i] = (uint8_t)v;
  }
}

template <int SB>
__global__ void unpack_codes_kernel(const uint8_t* packed, uint8_t* codes, size_t nbytes) {
  constexpr int kCpb = 8 / SB;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nbytes; i += (size_t)gridDim.x * blockDim.x) {
    const uint32_t v = packed[i];
#pragma unroll
    for (int l = 0; l < kCpb; ++l) codes[kCpb * i + l] = (uint8_t)((v >> (SB * l)) & ((1u << SB) - 1u));
  }
}

__global__ void pack_signs_kernel(const int8_t* w, uint32_t* bits, int rows, int K, int kwords) {
  const long total = (long)rows * kwords;
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long)gridDim.x * blockDim.x) {
    const int r = (int)(i / kwords), q = (int)(i % kwords);
    uint32_t v = 0;
    for (int t = 0; t < 32; ++t) {
      const int k = q * 32 + t;
      if (k < K && w[(size_t)r * K + k] > 0) v |= 1u << t;
    }
    bits[i] = v;
  }
}

// Prepared filter: e4m3 rows [cout][Kpad] in the chunk order of the
// tensor-core A expansion: with cpw codes per packed word (16 for 2-bit, 8 for
// 4-bit fields), byte p of chunk j holds k = cpw*j + (cpw/4)*(p%4) + p/4;
// +1 -> 0x38, -1 -> 0xB8, k >= K -> 0; followed by a copy of the sign words.
// 2-bit fields: the bytes of the odd 4-byte words of a chunk (p/4 odd) hold
// +-0.25 (0x28 / 0xA8) instead, because the expansion leaves those codes as 4c
// (the e4m3 value 4c * 2^-9); each product is c * 2^-9 either way.
// in8: the input is 8-bit values read as two 4-bit fields, so kernel position k
// is filter position k/2 times 1 (low nibble, k even) or 16 (high nibble):
// +-16 are the e4m3 bytes 0x58 / 0xD8.  K is the kernel's K (twice the filter's).
__global__ void prep_weights_kernel(const uint32_t* bits, uint8_t* e4m3, uint32_t* bits_copy, uint32_t* pbits, int cout,
                                    int K, int Kpad, int kwords, int cpw, int in8) {
  const long total = (long)cout * (Kpad / 4);
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long)gridDim.x * blockDim.x) {
    const int n = (int)(i / (Kpad / 4));
    const int p4 = (int)(i % (Kpad / 4)) * 4;  // first byte position of this 32-bit output word
    uint32_t out = 0;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int pos = p4 + t;
      const int j = pos / cpw, p = pos - j * cpw;
      const int k = cpw * j + (cpw >> 2) * (p & 3) + (p >> 2);
      uint32_t byte = 0;
      if (k < K) {
        const int kf = in8 ? (k >> 1) : k;                       // filter position
        const bool hi = in8 && (k & 1);
        const bool pos = (bits[(size_t)n * kwords + (kf >> 5)] >> (kf & 31)) & 1u;
        // 2-bit fields: the odd words of a chunk (p / 4 odd) carry the codes as 4c (expand2), so
        // their weights are +-0.25 (0x28 / 0xA8)
        const bool quarter = cpw == 16 && ((p >> 2) & 1);
        byte = pos ? (hi ? 0x58u : (quarter ? 0x28u : 0x38u)) : (hi ? 0xD8u : (quarter ? 0xA8u : 0xB8u));
      }
      out |= byte << (8 * t);
    }
    *(uint32_t*)(e4m3 + (size_t)n * Kpad + p4) = out;
  }
  const long tw = (long)cout * kwords;
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < tw; i += (long)gridDim.x * blockDim.x)
    bits_copy[i] = bits[i];
  // the same signs in the e4m3 rows' K order, one bit per byte position (set: +1): what the kernels
  // that expand the filter tile in shared memory read; positions past K are 0 (-1 there is harmless:
  // the gathered codes are zero)
  if (pbits && !in8) {
    const long tp = (long)cout * (Kpad / 32);
    for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < tp; i += (long)gridDim.x * blockDim.x) {
      const int n = (int)(i / (Kpad / 32));
      const int p0 = (int)(i % (Kpad / 32)) * 32;
      uint32_t w = 0;
      for (int b = 0; b < 32; ++b) {
        const int pos = p0 + b;
        const int j = pos / cpw, p = pos - j * cpw;
        const int k = cpw * j + (cpw >> 2) * (p & 3) + (p >> 2);
        if (k < K && ((bits[(size_t)n * kwords + (k >> 5)] >> (k & 31)) & 1u)) w |= 1u << b;
      }
      pbits[i] = w;
    }
  }
}

}  // namespace ifq
