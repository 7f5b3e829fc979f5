// Bit-serial CUDA-core path of the quantized convolution.
//
// With bit planes a_0, a_1 of the 2-bit codes (x = a_0 + 2*a_1) and the sign
// plane w+ of the +-1 filter (w = 2*w+ - 1), the integer core of Eq. (1) is
//   A = sum_p 2^p * (2*popc(a_p & w+) - popc(a_p))
//     = sum_words (2*popc(a_0 & w+) + 4*popc(a_1 & w+)) - S,
// where S = sum of the codes in the window (independent of the output channel).
// A CTA gathers the planes of TM output pixels for a K chunk into shared
// memory once and reuses them for TN output channels.
#pragma once
#include <cstdint>

#include "ptx.cuh"

namespace ifq {

struct BsArgs {
  const uint8_t* x;
  const uint32_t* wbits;  // [cout][kwords]
  const int32_t* thr;
  const int8_t* sign;
  uint8_t* y_codes;
  int32_t* y_acc;
  int n, h, w, cin, cout, kh, kw, stride, pad, ho, wo;
  int M, K, kwords;
};

constexpr int kBsTM = 32;       // output pixels per CTA
constexpr int kBsTN = 64;       // output channels per CTA
constexpr int kBsKC = 32;       // 32-bit words of K per chunk (1024 k)
constexpr int kBsThreads = 256;

__global__ void __launch_bounds__(kBsThreads) conv_bitserial_kernel(const BsArgs a) {
  __shared__ uint32_t sP0[kBsTM][kBsKC + 1];
  __shared__ uint32_t sP1[kBsTM][kBsKC + 1];
  __shared__ uint32_t sW[kBsTN][kBsKC + 1];
  __shared__ int sS[kBsTM];

  grid_dep_launch();
  grid_dep_wait();
  const int tid = threadIdx.x;
  const int m0 = blockIdx.x * kBsTM, n0 = blockIdx.y * kBsTN;
  // each thread: one pixel (tid % 32) and 8 consecutive channels ((tid / 32) * 8 ..)
  const int pm = tid & 31, pq = tid >> 5;
  int acc[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) acc[j] = 0;
  if (tid < kBsTM) sS[tid] = 0;
  const int cinb = a.cin >> 2;
  const int hw = a.ho * a.wo;

  for (int kw0 = 0; kw0 < a.kwords; kw0 += kBsKC) {
    __syncthreads();
    // gather bit planes: item = (pixel, word)
    for (int it = tid; it < kBsTM * kBsKC; it += kBsThreads) {
      const int p = it / kBsKC, q = it % kBsKC;
      const int m = m0 + p, word = kw0 + q;
      uint32_t b0 = 0, b1 = 0;
      if (m < a.M && word < a.kwords) {
        const int b = m / hw, rem = m - b * hw;
        const int oy = rem / a.wo, ox = rem - oy * a.wo;
        const uint8_t* img = a.x + (size_t)b * a.h * a.w * cinb;
        int k = word * 32;
        int tap = k / a.cin, c = k - tap * a.cin;
        for (int t = 0; t < 32 && k < a.K; t += 4, k += 4) {
          const int dy = tap / a.kw, dx = tap - dy * a.kw;
          const int iy = oy * a.stride + dy - a.pad, ix = ox * a.stride + dx - a.pad;
          uint32_t byte = 0;
          if ((unsigned)iy < (unsigned)a.h && (unsigned)ix < (unsigned)a.w)
            byte = img[((size_t)iy * a.w + ix) * cinb + (c >> 2)];
#pragma unroll
          for (int l = 0; l < 4; ++l) {
            const uint32_t code = (byte >> (2 * l)) & 3u;
            b0 |= (code & 1u) << (t + l);
            b1 |= (code >> 1) << (t + l);
          }
          c += 4;
          if (c == a.cin) { c = 0; ++tap; }
        }
      }
      sP0[p][q] = b0;
      sP1[p][q] = b1;
    }
    for (int it = tid; it < kBsTN * kBsKC; it += kBsThreads) {
      const int nn = it / kBsKC, q = it % kBsKC;
      const int n = n0 + nn, word = kw0 + q;
      sW[nn][q] = (n < a.cout && word < a.kwords) ? a.wbits[(size_t)n * a.kwords + word] : 0u;
    }
    __syncthreads();
    if (tid < kBsTM) {
      int s = 0;
      for (int q = 0; q < kBsKC; ++q) s += __popc(sP0[tid][q]) + 2 * __popc(sP1[tid][q]);
      sS[tid] += s;
    }
    for (int q = 0; q < kBsKC; ++q) {
      const uint32_t p0 = sP0[pm][q], p1 = sP1[pm][q];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint32_t wv = sW[pq * 8 + j][q];
        acc[j] += 2 * __popc(p0 & wv) + 4 * __popc(p1 & wv);
      }
    }
  }
  __syncthreads();
  const int m = m0 + pm;
  if (m >= a.M) return;
  const int S = sS[pm];
  uint32_t packed = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int n = n0 + pq * 8 + j;
    const int A = acc[j] - S;
    if (n < a.cout) {
      if (a.y_acc) a.y_acc[(size_t)m * a.cout + n] = A;
      if (a.y_codes) {
        const int sv = (int)a.sign[n] * A;
        const uint32_t code = (uint32_t)(sv > a.thr[3 * n]) + (uint32_t)(sv > a.thr[3 * n + 1]) +
                              (uint32_t)(sv > a.thr[3 * n + 2]);
        packed |= code << (2 * j);
      }
    }
  }
  if (a.y_codes) {
    // 8 channels = 2 bytes; cout % 4 == 0 so a byte never straddles the end
    const int nb = n0 + pq * 8;
    uint8_t* dst = a.y_codes + (size_t)m * (a.cout >> 2) + (nb >> 2);
    if (nb < a.cout) dst[0] = (uint8_t)packed;
    if (nb + 4 < a.cout) dst[1] = (uint8_t)(packed >> 8);
  }
}

}  // namespace ifq
