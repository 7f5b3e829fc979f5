// Max pooling of packed codes (Sec. 2.1 placement, on codes with channel signs)
// and the packing / filter-preparation kernels.
#pragma once
#include <cstdint>

#include "ptx.cuh"

namespace ifq {

// ---------------------------------------------------------------- pooling
//
// Channel c of a pixel is the SB-bit field c % (8/SB) of byte c / (8/SB) (SB = 2,
// or 4 for 3- and 4-bit codes).  With a channel sign of -1 the pool takes the
// min of the codes; with F = 2^SB - 1, min(a, b) = F - max(F-a, F-b) and
// F - x = x ^ F on an SB-bit field, so flipping those fields (XOR with a
// per-channel mask), taking a plain field-wise max, and flipping back gives
// both cases with one max.

// field-wise max of the 32/SB fields of a word, kept as 8/SB groups of byte lanes
template <int SB>
struct Lanes {
  static constexpr int kG = 8 / SB;
  static constexpr uint32_t kMask = SB == 2 ? 0x03030303u : 0x0F0F0F0Fu;
  uint32_t g[kG];
};
template <int SB>
__device__ __forceinline__ void lanes_split(uint32_t v, Lanes<SB>& L) {
#pragma unroll
  for (int s = 0; s < Lanes<SB>::kG; ++s) L.g[s] = (v >> (SB * s)) & Lanes<SB>::kMask;
}
template <int SB>
__device__ __forceinline__ void lanes_max(Lanes<SB>& acc, uint32_t v) {
#pragma unroll
  for (int s = 0; s < Lanes<SB>::kG; ++s) acc.g[s] = __vmaxu4(acc.g[s], (v >> (SB * s)) & Lanes<SB>::kMask);
}
template <int SB>
__device__ __forceinline__ uint32_t lanes_join(const Lanes<SB>& L) {
  uint32_t v = 0;
#pragma unroll
  for (int s = 0; s < Lanes<SB>::kG; ++s) v |= L.g[s] << (SB * s);
  return v;
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
};

// U = 32-bit words handled per thread (4 or 1); needs the packed bytes of a pixel to be a
// multiple of 4U.
template <int U, int SB>
__global__ void __launch_bounds__(256) maxpool_codes_kernel(const PoolArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  constexpr int kCpw = 32 / SB;             // codes per word
  const int cw = a.c / kCpw;                // 32-bit words per pixel
  const int groups = cw / U;
  const long total = (long)a.n * a.ho * a.wo * groups;
  for (long it = (long)blockIdx.x * blockDim.x + threadIdx.x; it < total; it += (long)gridDim.x * blockDim.x) {
    const int gi = (int)(it % groups);
    const long pix = it / groups;
    const int ox = (int)(pix % a.wo);
    const long t = pix / a.wo;
    const int oy = (int)(t % a.ho);
    const int b = (int)(t / a.ho);
    uint32_t mask[U];
#pragma unroll
    for (int u = 0; u < U; ++u) mask[u] = flip_mask<SB, kCpw>(a.sign, (gi * U + u) * kCpw, a.c);
    Lanes<SB> acc[U];
    bool first = true;
    for (int dy = 0; dy < a.k; ++dy) {
      const int iy = oy * a.stride + dy;
      if (iy >= a.h) continue;
      for (int dx = 0; dx < a.k; ++dx) {
        const int ix = ox * a.stride + dx;
        if (ix >= a.w) continue;
        const uint32_t* src = (const uint32_t*)(a.x + (((size_t)b * a.h + iy) * a.w + ix) * (size_t)(cw * 4)) + gi * U;
        uint32_t v[U];
        if constexpr (U == 4) {
          const uint4 q = __ldg((const uint4*)src);
          v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
        } else {
#pragma unroll
          for (int u = 0; u < U; ++u) v[u] = __ldg(src + u);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (first) lanes_split(v[u] ^ mask[u], acc[u]);
          else lanes_max(acc[u], v[u] ^ mask[u]);
        }
        first = false;
      }
    }
    uint32_t* dst = (uint32_t*)(a.y + (size_t)pix * (cw * 4)) + gi * U;
    uint32_t o[U];
#pragma unroll
    for (int u = 0; u < U; ++u) o[u] = lanes_join(acc[u]) ^ mask[u];
    if constexpr (U == 4) *(uint4*)dst = make_uint4(o[0], o[1], o[2], o[3]);
    else {
#pragma unroll
      for (int u = 0; u < U; ++u) dst[u] = o[u];
    }
  }
}

// byte-granular variant for any c % 4 == 0
template <int SB>
__global__ void __launch_bounds__(256) maxpool_codes_bytes_kernel(const PoolArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  constexpr int kCpb = 8 / SB;
  const int cb = a.c / kCpb;
  const long total = (long)a.n * a.ho * a.wo * cb;
  for (long it = (long)blockIdx.x * blockDim.x + threadIdx.x; it < total; it += (long)gridDim.x * blockDim.x) {
    const int bi = (int)(it % cb);
    const long pix = it / cb;
    const int ox = (int)(pix % a.wo);
    const long t = pix / a.wo;
    const int oy = (int)(t % a.ho);
    const int b = (int)(t / a.ho);
    const uint32_t mask = flip_mask<SB, kCpb>(a.sign, bi * kCpb, a.c);
    Lanes<SB> acc;
    bool first = true;
    for (int dy = 0; dy < a.k; ++dy) {
      const int iy = oy * a.stride + dy;
      if (iy >= a.h) continue;
      for (int dx = 0; dx < a.k; ++dx) {
        const int ix = ox * a.stride + dx;
        if (ix >= a.w) continue;
        const uint32_t v = a.x[(((size_t)b * a.h + iy) * a.w + ix) * cb + bi];
        if (first) lanes_split(v ^ mask, acc);
        else lanes_max(acc, v ^ mask);
        first = false;
      }
    }
    a.y[(size_t)pix * cb + bi] = (uint8_t)((lanes_join(acc) ^ mask) & 0xFFu);
  }
}

// ---------------------------------------------------------------- packing

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
__global__ void prep_weights_kernel(const uint32_t* bits, uint8_t* e4m3, uint32_t* bits_copy, int cout, int K,
                                    int Kpad, int kwords, int cpw) {
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
      if (k < K) byte = ((bits[(size_t)n * kwords + (k >> 5)] >> (k & 31)) & 1u) ? 0x38u : 0xB8u;
      out |= byte << (8 * t);
    }
    *(uint32_t*)(e4m3 + (size_t)n * Kpad + p4) = out;
  }
  const long tw = (long)cout * kwords;
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < tw; i += (long)gridDim.x * blockDim.x)
    bits_copy[i] = bits[i];
}

}  // namespace ifq
