// 2-bit max pooling (Sec. 2.1 placement, on codes with channel signs) and the
// packing / filter-preparation kernels.
#pragma once
#include <cstdint>

#include "ptx.cuh"

namespace ifq {

// ---------------------------------------------------------------- pooling
//
// Channel c of a pixel is the 2-bit lane c%4 of byte c/4.  With a channel
// sign of -1 the pool takes the min of the codes; min(a, b) = 3 - max(3-a, 3-b)
// and 3 - x = x ^ 3 on a 2-bit lane, so flipping those lanes (XOR with a
// per-channel mask), taking a plain lane-wise max, and flipping back gives
// both cases with one max.

// lane-wise max of 16 two-bit lanes, kept as four groups of byte lanes
struct Lanes4 {
  uint32_t g[4];
};
__device__ __forceinline__ void lanes_split(uint32_t v, Lanes4& L) {
#pragma unroll
  for (int s = 0; s < 4; ++s) L.g[s] = (v >> (2 * s)) & 0x03030303u;
}
__device__ __forceinline__ void lanes_max(Lanes4& acc, uint32_t v) {
#pragma unroll
  for (int s = 0; s < 4; ++s) acc.g[s] = __vmaxu4(acc.g[s], (v >> (2 * s)) & 0x03030303u);
}
__device__ __forceinline__ uint32_t lanes_join(const Lanes4& L) {
  return L.g[0] | (L.g[1] << 2) | (L.g[2] << 4) | (L.g[3] << 6);
}

// mask word for the 16 channels of word `wi` of a pixel: lanes of sign -1 channels are 0b11
__device__ __forceinline__ uint32_t flip_mask(const int8_t* sign, int c0, int c) {
  if (!sign) return 0u;
  uint32_t m = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j)
    if (c0 + j < c && sign[c0 + j] < 0) m |= 3u << (2 * j);
  return m;
}

struct PoolArgs {
  const uint8_t* x;
  const int8_t* sign;
  uint8_t* y;
  int n, h, w, c, k, stride, pad, ho, wo;
};

// U = 32-bit words handled per thread (4: 64 channels, 1: 16 channels).
template <int U>
__global__ void __launch_bounds__(256) maxpool2bit_kernel(const PoolArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  const int cw = a.c >> 4;                  // 32-bit words per pixel (c % 16 == 0)
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
    for (int u = 0; u < U; ++u) mask[u] = flip_mask(a.sign, (gi * U + u) * 16, a.c);
    Lanes4 acc[U];
    bool first = true;
    for (int dy = 0; dy < a.k; ++dy) {
      const int iy = oy * a.stride + dy;
      if (iy >= a.h) continue;
      for (int dx = 0; dx < a.k; ++dx) {
        const int ix = ox * a.stride + dx;
        if (ix >= a.w) continue;
        const uint32_t* src = (const uint32_t*)(a.x + (((size_t)b * a.h + iy) * a.w + ix) * (size_t)(a.c >> 2)) + gi * U;
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
    uint32_t* dst = (uint32_t*)(a.y + (size_t)pix * (a.c >> 2)) + gi * U;
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

// byte-granular variant for c % 16 != 0 (c % 4 == 0)
__global__ void __launch_bounds__(256) maxpool2bit_bytes_kernel(const PoolArgs a) {
  grid_dep_launch();
  grid_dep_wait();
  const int cb = a.c >> 2;
  const long total = (long)a.n * a.ho * a.wo * cb;
  for (long it = (long)blockIdx.x * blockDim.x + threadIdx.x; it < total; it += (long)gridDim.x * blockDim.x) {
    const int bi = (int)(it % cb);
    const long pix = it / cb;
    const int ox = (int)(pix % a.wo);
    const long t = pix / a.wo;
    const int oy = (int)(t % a.ho);
    const int b = (int)(t / a.ho);
    uint32_t mask = 0;
    if (a.sign)
      for (int j = 0; j < 4; ++j)
        if (a.sign[bi * 4 + j] < 0) mask |= 3u << (2 * j);
    Lanes4 acc;
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

__global__ void pack_codes_kernel(const uint8_t* codes, uint8_t* packed, size_t nbytes) {
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nbytes; i += (size_t)gridDim.x * blockDim.x) {
    const uchar4 c = *(const uchar4*)(codes + 4 * i);
    packed[i] = (uint8_t)((c.x & 3) | ((c.y & 3) << 2) | ((c.z & 3) << 4) | ((c.w & 3) << 6));
  }
}

__global__ void unpack_codes_kernel(const uint8_t* packed, uint8_t* codes, size_t nbytes) {
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nbytes; i += (size_t)gridDim.x * blockDim.x) {
    const uint32_t v = packed[i];
    *(uchar4*)(codes + 4 * i) = make_uchar4(v & 3, (v >> 2) & 3, (v >> 4) & 3, (v >> 6) & 3);
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
// tensor-core A expansion (byte p of chunk j holds k = 16j + 4*(p%4) + p/4),
// +1 -> 0x38, -1 -> 0xB8, k >= K -> 0; followed by a copy of the sign words.
__global__ void prep_weights_kernel(const uint32_t* bits, uint8_t* e4m3, uint32_t* bits_copy, int cout, int K,
                                    int Kpad, int kwords) {
  const long total = (long)cout * (Kpad / 4);
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long)gridDim.x * blockDim.x) {
    const int n = (int)(i / (Kpad / 4));
    const int p4 = (int)(i % (Kpad / 4)) * 4;  // first byte position of this 32-bit output word
    uint32_t out = 0;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int pos = p4 + t;
      const int j = pos >> 4, p = pos & 15;
      const int k = 16 * j + 4 * (p & 3) + (p >> 2);
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
