// Tensor-core path of the quantized convolution (Eq. (1) integer core with the
// thresholds of Eq. (7) fused as the epilogue), for sm_103a.
//
// GEMM view: D[m][n] = sum_k A[m][k] * B[n][k] with m = output pixel
// (b, oy, ox), n = output channel, k = (dy, dx, c) -- an implicit GEMM whose
// A rows are gathered on the fly from the packed 2-bit NHWC input.
//
// Exact integer arithmetic on the fp8 tensor cores (sm_103a has no tcgen05
// integer MMA):
//   * A: code c in {0,1,2,3} is stored as the e4m3 byte c, i.e. the subnormal
//     value c * 2^-9; the 2-bit -> 8-bit expansion is a mask per byte lane.
//   * B: +1 / -1 are the e4m3 bytes 0x38 / 0xB8 (+-1.0).
//   * Every product is c * 2^-9 exactly; every partial sum is an integer
//     multiple of 2^-9 of magnitude <= 3K * 2^-9; with 3K < 2^15 it needs at
//     most 24 significant bits, so the fp32 accumulator in tensor memory holds
//     it exactly and A = D * 512 recovers the integer.
//
// K ordering inside each 16-element chunk: the expansion of one 32-bit word
// of 16 packed codes produces byte p = 4q + t from code 4t + q (a 4x4
// transpose).  The prepared filter rows use the same order, so the dot
// product over K is unchanged.
//
// CTA: 128 output pixels x BN output channels; 6 warps:
//   warps 0-3  gather: im2col of packed codes (cp.async, zero fill for
//              padding), expansion into the 128B-swizzled K-major A tile,
//              then the epilogue (tcgen05.ld, thresholds, 2-bit packing);
//   warp 4     TMA producer of the prepared filter tile (B);
//   warp 5     TMEM allocation and the single-thread tcgen05.mma issue.
#pragma once
#include <cuda.h>

#include <cstdint>

#include "ptx.cuh"

namespace ifq {

struct ConvArgs {
  const uint8_t* x;      // packed input codes, NHWC
  const int32_t* thr;    // [cout][3]
  const int8_t* sign;    // [cout]
  uint8_t* y_codes;      // packed output codes or nullptr
  int32_t* y_acc;        // int32 accumulators or nullptr
  int n, h, w, cin, cout, kh, kw, stride, pad, ho, wo;
  int M;                 // n*ho*wo
  int K;                 // kh*kw*cin
  int nk;                // number of 128-wide K stages (Kpad / 128)
};

constexpr int kBM = 128;      // output pixels per CTA (MMA M)
constexpr int kBK = 128;      // K elements (= bytes) per pipeline stage
constexpr int kRawRow = 32;   // packed bytes of one A row per stage (128 codes)
constexpr int kTcThreads = 192;

// Byte offset of element (row r, byte k) inside a K-major 128B-swizzled tile.
__device__ __forceinline__ uint32_t sw128_chunk(int r, int chunk) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((chunk ^ (r & 7)) << 4));
}
// Raw staging: row r, 32 bytes, 16-byte halves swapped on alternate groups of 4 rows.
__device__ __forceinline__ uint32_t raw_off(int r, int byte) {
  return (uint32_t)(r * kRawRow + ((((byte >> 4) ^ (r >> 2)) & 1) << 4) + (byte & 15));
}

template <int BN, int STAGES, int RAW>
struct TcSmem {
  static constexpr int kA = kBM * kBK;   // 16 KB per stage
  static constexpr int kB = BN * kBK;
  static constexpr int kRaw = kBM * kRawRow;
  static constexpr int offA = 0;
  static constexpr int offB = offA + STAGES * kA;
  static constexpr int offRaw = offB + STAGES * kB;
  static constexpr int offThr = offRaw + RAW * kRaw;
  static constexpr int offBar = offThr + BN * 16;
  static constexpr int nBar = 3 * STAGES + 1;
  static constexpr int offTmem = offBar + nBar * 8;
  static constexpr int bytes = offTmem + 16 + 1024;  // + alignment slack
};

__device__ __forceinline__ void expand_store(uint32_t dstA, int r, int chunk, uint32_t u) {
  // 16 codes -> 16 e4m3 bytes; byte t of word q holds code 4t + q
  const uint32_t o0 = u & 0x03030303u, o1 = (u >> 2) & 0x03030303u;
  const uint32_t o2 = (u >> 4) & 0x03030303u, o3 = (u >> 6) & 0x03030303u;
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(dstA + sw128_chunk(r, chunk)), "r"(o0), "r"(o1),
               "r"(o2), "r"(o3)
               : "memory");
}

// GB: bytes per gathered granule: 16 (cin % 64 == 0), 4 (cin % 16 == 0), 1 (cin % 4 == 0).
template <int BN, int STAGES, int RAW, int GB>
__global__ void __launch_bounds__(kTcThreads, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap tmap_w, const ConvArgs args) {
  using L = TcSmem<BN, STAGES, RAW>;
  extern __shared__ uint8_t smem_raw_[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw_ + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sA = sbase + L::offA, sB = sbase + L::offB, sRaw = sbase + L::offRaw;
  int4* sThr = (int4*)(smem + L::offThr);
  const uint32_t barBase = sbase + L::offBar;
  auto full_a = [&](int s) { return barBase + 8u * s; };
  auto full_b = [&](int s) { return barBase + 8u * (STAGES + s); };
  auto empty = [&](int s) { return barBase + 8u * (2 * STAGES + s); };
  const uint32_t acc_full = barBase + 8u * (3 * STAGES);
  uint32_t* tmem_slot = (uint32_t*)(smem + L::offTmem);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.x * kBM, n0 = blockIdx.y * BN;
  constexpr uint32_t kCols = BN < 32 ? 32 : BN;

  // ---- setup
  if (warp == 5) {
    tmem_alloc(smem_u32(tmem_slot), kCols);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_a(s), 128);
      mbar_init(full_b(s), 1);
      mbar_init(empty(s), 1);
    }
    mbar_init(acc_full, 1);
    fence_mbar_init();
  }
  if (warp == 4 && lane == 0) prefetch_tmap(&tmap_w);
  for (int c = tid; c < BN; c += kTcThreads) {
    const int nn = n0 + c;
    int4 t = make_int4(0, 0, 0, 1);
    if (nn < args.cout && args.thr) t = make_int4(args.thr[3 * nn], args.thr[3 * nn + 1], args.thr[3 * nn + 2], args.sign[nn]);
    sThr[c] = t;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int nk = args.nk;
  bool ok = true;

  if (warp < 4) {
    // =================== gather (im2col + expansion) ===================
    const int r = tid;              // A row of this thread
    const int m = m0 + r;
    const bool row_ok = m < args.M;
    int iy0 = 0, ix0 = 0;
    const uint8_t* img = args.x;
    if (row_ok) {
      const int hw = args.ho * args.wo;
      const int b = m / hw, rem = m - b * hw;
      const int oy = rem / args.wo, ox = rem - oy * args.wo;
      iy0 = oy * args.stride - args.pad;
      ix0 = ox * args.stride - args.pad;
      img = args.x + (size_t)b * args.h * args.w * (args.cin >> 2);
    }
    const int cinb = args.cin >> 2;
    // issue cursor over the K axis: channel c (codes) within tap (dy, dx)
    int cc = 0, dx = 0, dy = 0;

    if constexpr (GB >= 4) {
      constexpr int kGran = kRawRow / GB;  // granules per stage
      auto issue = [&](int stage) {
        const uint32_t dst = sRaw + (uint32_t)((stage % RAW) * L::kRaw);
#pragma unroll
        for (int g = 0; g < kGran; ++g) {
          const int iy = iy0 + dy, ix = ix0 + dx;
          const bool inb = row_ok && dy < args.kh && (unsigned)iy < (unsigned)args.h && (unsigned)ix < (unsigned)args.w;
          const uint8_t* src = inb ? img + ((size_t)iy * args.w + ix) * cinb + (cc >> 2) : args.x;
          if constexpr (GB == 16)
            cp_async_16(dst + raw_off(r, g * 16), src, inb ? 16u : 0u);
          else
            cp_async_4(dst + raw_off(r, g * 4), src, inb ? 4u : 0u);
          cc += 4 * GB;
          if (cc == args.cin) {
            cc = 0;
            if (++dx == args.kw) { dx = 0; ++dy; }
          }
        }
      };
      constexpr int D = RAW - 1;
#pragma unroll 1
      for (int d = 0; d < D; ++d) {
        if (d < nk) issue(d);
        cp_async_commit();
      }
#pragma unroll 1
      for (int i = 0; i < nk; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (uint32_t)(i / STAGES) & 1u;
        if (i + D < nk) issue(i + D);
        cp_async_commit();
        cp_async_wait<D>();
        if (!mbar_wait(empty(s), ph ^ 1u)) { ok = false; break; }
        const uint32_t src = sRaw + (uint32_t)((i % RAW) * L::kRaw);
        const uint32_t dstA = sA + (uint32_t)(s * L::kA);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t u0, u1, u2, u3;
          asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];"
                       : "=r"(u0), "=r"(u1), "=r"(u2), "=r"(u3)
                       : "r"(src + raw_off(r, half * 16)));
          expand_store(dstA, r, half * 4 + 0, u0);
          expand_store(dstA, r, half * 4 + 1, u1);
          expand_store(dstA, r, half * 4 + 2, u2);
          expand_store(dstA, r, half * 4 + 3, u3);
        }
        fence_proxy_async_smem();
        mbar_arrive(full_a(s));
      }
      cp_async_wait<0>();
    } else {
      // narrow channels (cin % 16 != 0): byte-wise gather, 4 codes per byte
#pragma unroll 1
      for (int i = 0; i < nk; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (uint32_t)(i / STAGES) & 1u;
        uint32_t word[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          uint32_t u = 0;
#pragma unroll
          for (int bq = 0; bq < 4; ++bq) {
            const int iy = iy0 + dy, ix = ix0 + dx;
            const bool inb =
                row_ok && dy < args.kh && (unsigned)iy < (unsigned)args.h && (unsigned)ix < (unsigned)args.w;
            uint32_t v = 0;
            if (inb) v = __ldg(img + ((size_t)iy * args.w + ix) * cinb + (cc >> 2));
            u |= v << (8 * bq);
            cc += 4;
            if (cc == args.cin) {
              cc = 0;
              if (++dx == args.kw) { dx = 0; ++dy; }
            }
          }
          word[q] = u;
        }
        if (!mbar_wait(empty(s), ph ^ 1u)) { ok = false; break; }
        const uint32_t dstA = sA + (uint32_t)(s * L::kA);
#pragma unroll
        for (int q = 0; q < 8; ++q) expand_store(dstA, r, q, word[q]);
        fence_proxy_async_smem();
        mbar_arrive(full_a(s));
      }
    }

    // =================== epilogue ===================
    if (ok) ok = mbar_wait(acc_full, 0);
    tc_fence_after();
    if (ok) {
      const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
      uint32_t packed[BN / 16];
#pragma unroll
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(trow + c0, v);
        tmem_ld_wait();
        int a[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) a[j] = __float2int_rn(__uint_as_float(v[j]) * 512.0f);
        uint32_t w0 = 0, w1 = 0;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int4 t = sThr[c0 + j];
          const int sv = t.w * a[j];
          const uint32_t code = (uint32_t)(sv > t.x) + (uint32_t)(sv > t.y) + (uint32_t)(sv > t.z);
          if (j < 16) w0 |= code << (2 * j);
          else w1 |= code << (2 * (j - 16));
        }
        packed[c0 / 16] = w0;
        packed[c0 / 16 + 1] = w1;
        if (args.y_acc && row_ok) {
          int32_t* dst = args.y_acc + (size_t)m * args.cout + n0 + c0;
          if (n0 + c0 + 32 <= args.cout && (args.cout & 3) == 0) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) *(int4*)(dst + j) = make_int4(a[j], a[j + 1], a[j + 2], a[j + 3]);
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (n0 + c0 + j < args.cout) dst[j] = a[j];
          }
        }
      }
      if (args.y_codes && row_ok) {
        const int rowb = args.cout >> 2;  // bytes per output pixel
        uint8_t* dst = args.y_codes + (size_t)m * rowb + (n0 >> 2);
        if (n0 + BN <= args.cout && (rowb & 15) == 0 && BN >= 64) {
#pragma unroll
          for (int q = 0; q < BN / 64; ++q)
            *(uint4*)(dst + 16 * q) = make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
        } else if (n0 + BN <= args.cout && (rowb & 3) == 0) {
#pragma unroll
          for (int q = 0; q < BN / 16; ++q) *(uint32_t*)(dst + 4 * q) = packed[q];
        } else {
          const int nbytes = min(BN, args.cout - n0) >> 2;
          for (int q = 0; q < nbytes; ++q) dst[q] = (uint8_t)(packed[q >> 2] >> (8 * (q & 3)));
        }
      }
    }
  } else if (warp == 4) {
    // =================== TMA producer (filters) ===================
    if (lane == 0) {
      int issued = 0;
#pragma unroll 1
      for (int i = 0; i < nk; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (uint32_t)(i / STAGES) & 1u;
        if (!mbar_wait(empty(s), ph ^ 1u)) break;
        mbar_arrive_expect_tx(full_b(s), (uint32_t)L::kB);
        tma_load_2d(sB + (uint32_t)(s * L::kB), &tmap_w, full_b(s), i * kBK, n0);
        ++issued;
      }
      // drain: the last loads into each slot have landed before the CTA may exit
      for (int i = issued - STAGES < 0 ? 0 : issued - STAGES; i < issued; ++i)
        mbar_wait(full_b(i % STAGES), (uint32_t)(i / STAGES) & 1u);
    }
    __syncwarp();
  } else {
    // =================== MMA issue ===================
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_e4m3_f32(kBM, BN);
#pragma unroll 1
      for (int i = 0; i < nk; ++i) {
        const int s = i % STAGES;
        const uint32_t ph = (uint32_t)(i / STAGES) & 1u;
        if (!mbar_wait(full_a(s), ph)) break;
        if (!mbar_wait(full_b(s), ph)) break;
        tc_fence_after();
        const uint32_t a0 = sA + (uint32_t)(s * L::kA), b0 = sB + (uint32_t)(s * L::kB);
#pragma unroll
        for (int kk = 0; kk < kBK / 32; ++kk)
          mma_e4m3(tmem, sdesc_sw128(a0 + 32 * kk), sdesc_sw128(b0 + 32 * kk), idesc, (i | kk) != 0 ? 1u : 0u);
        mma_commit(empty(s));
      }
      mma_commit(acc_full);  // also fires if the loop broke: no MMA stays in flight
    }
    __syncwarp();
  }

  // ---- teardown: all MMAs are complete (acc_full) before TMEM is released
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    mbar_wait(acc_full, 0);
    tmem_dealloc(tmem, kCols);
  }
}

}  // namespace ifq
