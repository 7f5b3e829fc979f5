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

#include "conv_common.cuh"   // FastDiv

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

namespace ifq {

// Narrow-layer form of the bit-serial path: 2-bit codes, cin = 4, 8 or 16, 3x3, stride 1, at most 32
// output channels, pool 1 or 2.  No bit planes are split off: with M the +1 taps of filter n
// widened to two bits per code (0b11 where w = +1) and X a word of 16 interleaved 2-bit codes,
//   P = sum over +1 taps of x = popc(X & M) + popc(X & M & 0xAAAAAAAA),
//   S = sum of x           = popc(X) + popc(X & 0xAAAAAAAA),          A = 2 P - S.
// The 9 taps of a window are packed 32/(2 cin) to a word (in (dy, dx, c) order, so the masks
// follow the filter's K order).  One thread computes one output or pooled pixel: it loads its
// (P + 2)^2 input pixels once, builds the words of each of the P^2 conv pixels, and for each
// channel reads that channel's masks once for all of them, takes the max of A over the pool
// window (Sec. 2.1) and compares sign*A with the thresholds.
constexpr int kNarrowThreads = 128;

struct NarrowArgs {
  const uint8_t* x;           // packed 2-bit codes NHWC
  const uint32_t* wbits;      // sign words [cout][kwords], K in (dy, dx, c) order
  const int32_t* thr;         // [cout][3]
  const int8_t* sign;
  uint8_t* y_codes;           // [n][pho][pwo][cout/4] or nullptr
  int32_t* y_acc;             // [n][ho][wo][cout] or nullptr (pool 1)
  int n, h, w, cout, pad, ho, wo, pho, pwo, kwords;
  int total;                  // n * pho * pwo
  FastDiv div_pwo, div_pho;
};

// NC: channel bound (8, 16 or 32; cout <= NC), so the channel loop unrolls.
template <int CIN, int P, int NC>
__global__ void __launch_bounds__(kNarrowThreads) conv_bitserial_narrow_kernel(const NarrowArgs a) {
  constexpr int PB = 2 * CIN;                  // bits of one pixel's codes
  constexpr int TPW = 32 / PB;                 // taps per word
  constexpr int NW = (9 + TPW - 1) / TPW;      // words of a 3x3 window
  constexpr int WIN = P + 2;
  constexpr uint32_t HI = 0xAAAAAAAAu;
  __shared__ uint32_t sM[32 * NW];
  __shared__ int32_t sT[32 * 3];
  __shared__ int32_t sS[32];
  grid_dep_launch();
  grid_dep_wait();
  // widened masks: code position pos = (t % TPW) * CIN + c of word t / TPW holds tap t, channel c
  for (int i = threadIdx.x; i < a.cout * NW; i += blockDim.x) {
    const int n = i / NW, wd = i - n * NW;
    uint32_t m = 0;
    for (int j = 0; j < TPW; ++j) {
      const int t = wd * TPW + j;
      if (t >= 9) break;
      for (int c = 0; c < CIN; ++c) {
        const int k = t * CIN + c;
        if ((a.wbits[(size_t)n * a.kwords + (k >> 5)] >> (k & 31)) & 1u) m |= 3u << (2 * (j * CIN + c));
      }
    }
    sM[i] = m;
  }
  if (a.thr)
    for (int i = threadIdx.x; i < a.cout * 3; i += blockDim.x) sT[i] = a.thr[i];
  if (a.sign)
    for (int i = threadIdx.x; i < a.cout; i += blockDim.x) sS[i] = a.sign[i];
  __syncthreads();
  for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < a.total; it += gridDim.x * blockDim.x) {
    const int t = (int)fdiv((uint32_t)it, a.div_pwo);
    const int px = it - t * a.pwo;
    const int b = (int)fdiv((uint32_t)t, a.div_pho);
    const int py = t - b * a.pho;
    const int iy0 = py * P - a.pad, ix0 = px * P - a.pad;
    uint32_t win[WIN * WIN];
#pragma unroll
    for (int wy = 0; wy < WIN; ++wy)
#pragma unroll
      for (int wx = 0; wx < WIN; ++wx) {
        const int iy = iy0 + wy, ix = ix0 + wx;
        uint32_t v = 0;                              // zero padding: code 0
        if ((unsigned)iy < (unsigned)a.h && (unsigned)ix < (unsigned)a.w) {
          const uint8_t* p = a.x + (((size_t)b * a.h + iy) * a.w + ix) * (CIN / 4);
          if constexpr (CIN == 4) v = __ldg(p);
          else if constexpr (CIN == 8) v = __ldg((const unsigned short*)p);
          else v = __ldg((const uint32_t*)p);
        }
        win[wy * WIN + wx] = v;
      }
    uint32_t wds[P * P][NW];
    int S[P * P];
#pragma unroll
    for (int q = 0; q < P * P; ++q) {
#pragma unroll
      for (int wd = 0; wd < NW; ++wd) {
        uint32_t v = 0;
#pragma unroll
        for (int j = 0; j < TPW; ++j) {
          const int tp = wd * TPW + j;
          if (tp < 9) v |= win[(q / P + tp / 3) * WIN + (q % P + tp % 3)] << (PB * j);
        }
        wds[q][wd] = v;
      }
      int s = 0;
#pragma unroll
      for (int wd = 0; wd < NW; ++wd) s += __popc(wds[q][wd]) + __popc(wds[q][wd] & HI);
      S[q] = s;
    }
    uint32_t byte = 0;
#pragma unroll
    for (int n = 0; n < NC; ++n) {
      if (n >= a.cout) break;
      uint32_t m[NW];
#pragma unroll
      for (int wd = 0; wd < NW; ++wd) m[wd] = sM[n * NW + wd];
      int amax = INT32_MIN;
#pragma unroll
      for (int q = 0; q < P * P; ++q) {
        int pp = 0;
#pragma unroll
        for (int wd = 0; wd < NW; ++wd) {
          const uint32_t xm = wds[q][wd] & m[wd];
          pp += __popc(xm) + __popc(xm & HI);
        }
        amax = max(amax, 2 * pp - S[q]);
      }
      if (P == 1 && a.y_acc) a.y_acc[(size_t)it * a.cout + n] = amax;
      if (a.y_codes) {
        const int sv = sS[n] * amax;
        const uint32_t code = (uint32_t)(sv > sT[3 * n]) + (uint32_t)(sv > sT[3 * n + 1]) + (uint32_t)(sv > sT[3 * n + 2]);
        byte |= code << (2 * (n & 3));
        if ((n & 3) == 3) {
          a.y_codes[(size_t)it * (a.cout >> 2) + (n >> 2)] = (uint8_t)byte;
          byte = 0;
        }
      }
    }
  }
}

}  // namespace ifq
