// Bit-serial CUDA-core path of the quantized convolution.
//
// With bit planes a_p of the codes (x = sum_p 2^p a_p; 2 planes for 2-bit
// codes, 4 for codes stored in 4-bit fields) and the sign plane w+ of the +-1
// filter (w = 2*w+ - 1), the integer core of Eq. (1) is
//   A = sum_p 2^p * (2*popc(a_p & w+) - popc(a_p))
//     = sum_words sum_p 2^(p+1) popc(a_p & w+) - S,
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
  const int32_t* thr;     // [cout][lvl]
  const int8_t* sign;
  uint8_t* y_codes;
  int32_t* y_acc;
  int n, h, w, cin, cout, kh, kw, stride, pad, ho, wo;
  int M, K, kwords;
  int lvl;                // 2^k - 1 thresholds per channel
};

constexpr int kBsTM = 32;       // output pixels per CTA
constexpr int kBsTN = 64;       // output channels per CTA
constexpr int kBsKC = 32;       // 32-bit words of K per chunk (1024 k)
constexpr int kBsThreads = 256;

// SB: bits per stored code (2, or 4 for 3- and 4-bit codes) = number of bit planes.
template <int SB>
__global__ void __launch_bounds__(kBsThreads) conv_bitserial_kernel(const BsArgs a) {
  constexpr int kCpb = 8 / SB;   // codes per byte
  __shared__ uint32_t sP[SB][kBsTM][kBsKC + 1];
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
  const int cinb = a.cin / kCpb;
  const int hw = a.ho * a.wo;

  for (int kw0 = 0; kw0 < a.kwords; kw0 += kBsKC) {
    __syncthreads();
    // gather bit planes: item = (pixel, word)
    for (int it = tid; it < kBsTM * kBsKC; it += kBsThreads) {
      const int p = it / kBsKC, q = it % kBsKC;
      const int m = m0 + p, word = kw0 + q;
      uint32_t bp[SB];
#pragma unroll
      for (int q2 = 0; q2 < SB; ++q2) bp[q2] = 0;
      if (m < a.M && word < a.kwords) {
        const int b = m / hw, rem = m - b * hw;
        const int oy = rem / a.wo, ox = rem - oy * a.wo;
        const uint8_t* img = a.x + (size_t)b * a.h * a.w * cinb;
        int k = word * 32;
        int tap = k / a.cin, c = k - tap * a.cin;
        // cin % 4 == 0, so a byte of codes never straddles two taps
        for (int t = 0; t < 32 && k < a.K; t += kCpb, k += kCpb) {
          const int dy = tap / a.kw, dx = tap - dy * a.kw;
          const int iy = oy * a.stride + dy - a.pad, ix = ox * a.stride + dx - a.pad;
          uint32_t byte = 0;
          if ((unsigned)iy < (unsigned)a.h && (unsigned)ix < (unsigned)a.w)
            byte = img[((size_t)iy * a.w + ix) * cinb + c / kCpb];
#pragma unroll
          for (int l = 0; l < kCpb; ++l) {
            const uint32_t code = (byte >> (SB * l)) & ((1u << SB) - 1u);
#pragma unroll
            for (int q2 = 0; q2 < SB; ++q2) bp[q2] |= ((code >> q2) & 1u) << (t + l);
          }
          c += kCpb;
          if (c == a.cin) { c = 0; ++tap; }
        }
      }
#pragma unroll
      for (int q2 = 0; q2 < SB; ++q2) sP[q2][p][q] = bp[q2];
    }
    for (int it = tid; it < kBsTN * kBsKC; it += kBsThreads) {
      const int nn = it / kBsKC, q = it % kBsKC;
      const int n = n0 + nn, word = kw0 + q;
      sW[nn][q] = (n < a.cout && word < a.kwords) ? a.wbits[(size_t)n * a.kwords + word] : 0u;
    }
    __syncthreads();
    if (tid < kBsTM) {
      int s = 0;
      for (int q = 0; q < kBsKC; ++q)
#pragma unroll
        for (int q2 = 0; q2 < SB; ++q2) s += __popc(sP[q2][tid][q]) << q2;
      sS[tid] += s;
    }
    for (int q = 0; q < kBsKC; ++q) {
      uint32_t pl[SB];
#pragma unroll
      for (int q2 = 0; q2 < SB; ++q2) pl[q2] = sP[q2][pm][q];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint32_t wv = sW[pq * 8 + j][q];
#pragma unroll
        for (int q2 = 0; q2 < SB; ++q2) acc[j] += __popc(pl[q2] & wv) << (q2 + 1);
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
        const int32_t* t = a.thr + (size_t)a.lvl * n;
        uint32_t code = 0;
        for (int i = 0; i < a.lvl; ++i) code += (uint32_t)(sv > t[i]);
        packed |= code << (SB * j);
      }
    }
  }
  if (a.y_codes) {
    // 8 channels = SB bytes; cout % 4 == 0 so a byte never straddles the end
    const int nb = n0 + pq * 8;
    uint8_t* dst = a.y_codes + (size_t)m * (a.cout / kCpb) + nb / kCpb;
#pragma unroll
    for (int q = 0; q < SB; ++q)
      if (nb + q * kCpb < a.cout) dst[q] = (uint8_t)(packed >> (8 * q));
  }
}

}  // namespace ifq
