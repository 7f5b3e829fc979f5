// Direct CUDA-core path of the quantized convolution for a layer on 8-bit input values with few
// output channels: the first layer of IFQ-Tinier-YOLO (Sec. 4.2: every conv binarized, the first
// one on the RGB image), Eq. (1) with integer inputs followed by the thresholds of Eq. (7).
//
// With the sign plane w+ of the +-1 filter (w = 2 w+ - 1), A[n] = 2 P[n] - S, where
// P[n] = sum of the inputs under the +1 taps of filter n and S = sum of all inputs in the window
// (independent of n).  P of two channels is kept in the two 16-bit halves of one register: each
// input byte x adds x * m to it, with m = w+[2j] | w+[2j+1] << 16, so one multiply-add serves two
// channels; P <= 255 K < 2^16 for K <= 257 keeps the halves apart.  One thread computes one output
// pixel (or one pooled pixel: the max of A over its p x p window, the fused pool of Sec. 2.1)
// for every channel, then compares sign*A with the integer thresholds.
#pragma once
#include <cstdint>

#include "conv_common.cuh"   // FastDiv

namespace ifq {

constexpr int kDirectMaxCout = 32;   // channels per thread (16 pairs)
constexpr int kDirectMaxK = 257;
constexpr int kDirectThreads = 128;

struct DirectArgs {
  const uint8_t* x;        // 8-bit values NHWC [n][h][w][cin]
  const uint32_t* wmask;   // [K] bit n: filter n is +1 at tap k ((dy, dx, c) order)
  const int32_t* thr;      // [cout][lvl]
  const int8_t* sign;      // [cout]
  uint8_t* y_codes;        // packed codes [n][pho][pwo][cout*sbo/8] or nullptr
  int32_t* y_acc;          // int32 [n][ho][wo][cout] or nullptr (no pool)
  int n, h, w, cin, cout, kh, kw, stride, pad, ho, wo;
  int K, lvl, sbo, pool, pho, pwo;
  int total;               // n * pho * pwo
  FastDiv div_pwo, div_pho;
};

// NP = channel pairs per thread (4, 8 or 16: cout <= 8, 16, 32).
template <int NP>
__global__ void __launch_bounds__(kDirectThreads) conv_direct_kernel(const DirectArgs a) {
  __shared__ uint32_t sM[kDirectMaxK * NP];   // pair masks [k][j]
  __shared__ int32_t sT[2 * NP * 15];
  __shared__ int32_t sS[2 * NP];
  grid_dep_launch();
  grid_dep_wait();
  constexpr int np = NP;
  for (int i = threadIdx.x; i < a.K * np; i += blockDim.x) {
    const int k = i / np, j = i - k * np;
    const uint32_t mk = a.wmask[k];
    sM[i] = ((mk >> (2 * j)) & 1u) | (((mk >> (2 * j + 1)) & 1u) << 16);
  }
  if (a.thr)
    for (int i = threadIdx.x; i < a.cout * a.lvl; i += blockDim.x) sT[i] = a.thr[i];
  if (a.sign)
    for (int i = threadIdx.x; i < a.cout; i += blockDim.x) sS[i] = a.sign[i];
  __syncthreads();
  const int rowb = a.w * a.cin;
  for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < a.total; it += gridDim.x * blockDim.x) {
    const int t = (int)fdiv((uint32_t)it, a.div_pwo);
    const int px = it - t * a.pwo;
    const int b = (int)fdiv((uint32_t)t, a.div_pho);
    const int py = t - b * a.pho;
    int amax[2 * NP];
#pragma unroll
    for (int n = 0; n < 2 * NP; ++n) amax[n] = INT32_MIN;
    for (int wy = 0; wy < a.pool; ++wy)
      for (int wx = 0; wx < a.pool; ++wx) {
        const int oy = py * a.pool + wy, ox = px * a.pool + wx;
        uint32_t P[NP];
#pragma unroll
        for (int j = 0; j < NP; ++j) P[j] = 0;
        int S = 0;
        int k = 0;
        for (int dy = 0; dy < a.kh; ++dy) {
          const int iy = oy * a.stride + dy - a.pad;
          for (int dx = 0; dx < a.kw; ++dx, k += a.cin) {
            const int ix = ox * a.stride + dx - a.pad;
            if ((unsigned)iy >= (unsigned)a.h || (unsigned)ix >= (unsigned)a.w) continue;   // zero padding
            const uint32_t* px4 = (const uint32_t*)(a.x + (size_t)b * a.h * rowb + (size_t)iy * rowb + (size_t)ix * a.cin);
            for (int c4 = 0; c4 < a.cin; c4 += 4) {
              const uint32_t v = __ldg(px4 + (c4 >> 2));
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const uint32_t xv = (v >> (8 * q)) & 0xFFu;
                S += (int)xv;
                const uint32_t* m = sM + (size_t)(k + c4 + q) * np;
#pragma unroll
                for (int j = 0; j < NP; ++j) P[j] += xv * m[j];
              }
            }
          }
        }
#pragma unroll
        for (int j = 0; j < NP; ++j) {
          const int A0 = 2 * (int)(P[j] & 0xFFFFu) - S, A1 = 2 * (int)(P[j] >> 16) - S;
          amax[2 * j] = max(amax[2 * j], A0);
          amax[2 * j + 1] = max(amax[2 * j + 1], A1);
        }
        if (a.y_acc && a.pool == 1) {
          int32_t* dst = a.y_acc + ((size_t)(b * a.ho + oy) * a.wo + ox) * a.cout;
#pragma unroll
          for (int n = 0; n < 2 * NP; ++n)
            if (n < a.cout) dst[n] = amax[n];
        }
      }
    if (a.y_codes) {
      // codes of the (pooled) accumulator, 8/sbo per byte, stored byte by byte (a pixel's
      // cout*sbo/8 bytes need not be word-aligned); cout % 4 == 0 fills the last byte
      uint8_t* dst = a.y_codes + (size_t)it * (a.cout * a.sbo / 8);
      uint32_t byte = 0;
      int nbits = 0, bi = 0;
#pragma unroll
      for (int n = 0; n < 2 * NP; ++n) {
        if (n < a.cout) {
          const int sv = sS[n] * amax[n];
          uint32_t code = 0;
          for (int i = 0; i < a.lvl; ++i) code += (uint32_t)(sv > sT[n * a.lvl + i]);
          byte |= code << nbits;
          nbits += a.sbo;
          if (nbits == 8) {
            dst[bi++] = (uint8_t)byte;
            byte = 0;
            nbits = 0;
          }
        }
      }
    }
  }
}

// a . b + c over four byte lanes, a unsigned (pixel values), b signed (+-1 weights).
__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
  int d;
  asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// The common first layer: cin = 4 (RGB and a zero channel: one 32-bit word per pixel), 3x3,
// stride 1, pool P = 1 or 2.  A tap is one word of four 8-bit values, so A[n] is nine dp4a of the
// pixel words with filter n's +-1 byte words (0x01 / 0xFF).  The (P + 2)^2 input words of a
// thread's window are loaded first, and the loop runs over the 9 taps outermost, so each tap's
// weight words are read once for the P^2 conv pixels.
template <int NC, int P>
__global__ void __launch_bounds__(kDirectThreads) conv_direct_rgb3_kernel(const DirectArgs a) {
  constexpr int KS = 3, WIN = P + KS - 1, TAPS = KS * KS;
  __shared__ __align__(16) uint32_t sW[TAPS * NC];   // [tap][n] +-1 byte words
  __shared__ int32_t sT[NC * 15];
  __shared__ int32_t sS[NC];
  __shared__ int4 sT3[NC];                            // lvl = 3: {T1, T2, T3, sign} per channel
  grid_dep_launch();
  grid_dep_wait();
  for (int i = threadIdx.x; i < TAPS * NC; i += blockDim.x) {
    const int t = i / NC, n = i - t * NC;
    uint32_t wv = 0;
#pragma unroll
    for (int c = 0; c < 4; ++c) wv |= (((a.wmask[4 * t + c] >> n) & 1u) ? 0x01u : 0xFFu) << (8 * c);
    sW[i] = wv;
  }
  if (a.thr)
    for (int i = threadIdx.x; i < a.cout * a.lvl; i += blockDim.x) sT[i] = a.thr[i];
  if (a.sign)
    for (int i = threadIdx.x; i < a.cout; i += blockDim.x) sS[i] = a.sign[i];
  if (a.thr && a.sign && a.lvl == 3)
    for (int i = threadIdx.x; i < a.cout; i += blockDim.x)
      sT3[i] = make_int4(a.thr[3 * i], a.thr[3 * i + 1], a.thr[3 * i + 2], a.sign[i]);
  __syncthreads();
  const uint32_t* x32 = (const uint32_t*)a.x;
  for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < a.total; it += gridDim.x * blockDim.x) {
    const int t = (int)fdiv((uint32_t)it, a.div_pwo);
    const int px = it - t * a.pwo;
    const int b = (int)fdiv((uint32_t)t, a.div_pho);
    const int py = t - b * a.pho;
    const int iy0 = py * P - a.pad, ix0 = px * P - a.pad;
    uint32_t win[WIN * WIN];
    if (iy0 >= 0 && ix0 >= 0 && iy0 + WIN <= a.h && ix0 + WIN <= a.w) {
      // the whole window inside the image (all but the border pixels): one address, no checks
      const uint32_t* p0 = x32 + ((size_t)b * a.h + iy0) * a.w + ix0;
#pragma unroll
      for (int wy = 0; wy < WIN; ++wy)
#pragma unroll
        for (int wx = 0; wx < WIN; ++wx) win[wy * WIN + wx] = __ldg(p0 + (size_t)wy * a.w + wx);
    } else {
#pragma unroll
      for (int wy = 0; wy < WIN; ++wy)
#pragma unroll
        for (int wx = 0; wx < WIN; ++wx) {
          const int iy = iy0 + wy, ix = ix0 + wx;
          const bool in = (unsigned)iy < (unsigned)a.h && (unsigned)ix < (unsigned)a.w;   // else zero padding
          win[wy * WIN + wx] = in ? __ldg(x32 + ((size_t)b * a.h + iy) * a.w + ix) : 0u;
        }
    }
    int acc[P * P][NC];
#pragma unroll
    for (int q = 0; q < P * P; ++q)
#pragma unroll
      for (int n = 0; n < NC; ++n) acc[q][n] = 0;
#pragma unroll
    for (int dy = 0; dy < KS; ++dy)
#pragma unroll
      for (int dx = 0; dx < KS; ++dx) {
        const uint32_t* wt = sW + (dy * KS + dx) * NC;
#pragma unroll
        for (int n = 0; n < NC; ++n) {
          const uint32_t wv = wt[n];
#pragma unroll
          for (int q = 0; q < P * P; ++q) acc[q][n] = dp4a_us(win[(q / P + dy) * WIN + (q % P + dx)], wv, acc[q][n]);
        }
      }
    int amax[NC];
#pragma unroll
    for (int n = 0; n < NC; ++n) {
      int m = acc[0][n];
#pragma unroll
      for (int q = 1; q < P * P; ++q) m = max(m, acc[q][n]);
      amax[n] = m;
    }
    if (P == 1 && a.y_acc) {
      int32_t* dst = a.y_acc + (size_t)it * a.cout;
#pragma unroll
      for (int n = 0; n < NC; ++n)
        if (n < a.cout) dst[n] = amax[n];
    }
    if (a.y_codes && a.lvl == 3 && a.sbo == 2 && (a.cout & 3) == 0) {
      // 2-bit codes: thresholds and sign of a channel in one 16-byte load, the codes of 4 channels
      // a byte
      uint8_t* dst = a.y_codes + (size_t)it * (a.cout >> 2);
#pragma unroll
      for (int n4 = 0; n4 < NC; n4 += 4) {
        if (n4 < a.cout) {
          uint32_t byte = 0;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int4 t = sT3[n4 + q];
            const int sv = t.w * amax[n4 + q];
            byte |= ((uint32_t)(sv > t.x) + (uint32_t)(sv > t.y) + (uint32_t)(sv > t.z)) << (2 * q);
          }
          dst[n4 >> 2] = (uint8_t)byte;
        }
      }
    } else if (a.y_codes) {
      uint8_t* dst = a.y_codes + (size_t)it * (a.cout * a.sbo / 8);
      uint32_t byte = 0;
      int nbits = 0, bi = 0;
#pragma unroll
      for (int n = 0; n < NC; ++n) {
        if (n < a.cout) {
          const int sv = sS[n] * amax[n];
          uint32_t code = 0;
          for (int i = 0; i < a.lvl; ++i) code += (uint32_t)(sv > sT[n * a.lvl + i]);
          byte |= code << nbits;
          nbits += a.sbo;
          if (nbits == 8) {
            dst[bi++] = (uint8_t)byte;
            byte = 0;
            nbits = 0;
          }
        }
      }
    }
  }
}

// Filter sign words [cout][kwords] -> per-tap masks [K] (bit n = +1 for filter n < min(cout, 32)).
__global__ void prep_direct_masks_kernel(const uint32_t* bits, uint32_t* masks, int cout, int K, int kwords) {
  for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < K; k += gridDim.x * blockDim.x) {
    uint32_t m = 0;
    for (int n = 0; n < cout && n < 32; ++n) m |= ((bits[(size_t)n * kwords + (k >> 5)] >> (k & 31)) & 1u) << n;
    masks[k] = m;
  }
}

}  // namespace ifq
