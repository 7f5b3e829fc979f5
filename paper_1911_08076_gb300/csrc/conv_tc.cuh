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
//     it exactly: D = A / 512.
//   * Thresholds: sign*A > T  <=>  sign*D > T/512, and T/512 is exact in fp32
//     (|T| < 2^24), so the epilogue compares the accumulator in fp32 directly.
//
// K ordering inside each 16-element chunk: the expansion of one 32-bit word
// of 16 packed codes produces byte p = 4q + t from code 4t + q (a 4x4
// transpose).  The prepared filter rows use the same order, so the dot
// product over K is unchanged.
//
// Persistent, warp-specialized CTA (one per SM).  A tile is SUB x 128 output
// pixels by BN output channels; with SUB = 2 the two 128-row halves have their
// own accumulators and their MMAs interleave, so consecutive MMAs do not wait
// on each other.  18 warps:
//   warps 0-7    gather: each thread owns one 16-byte unit (64 codes) of a
//                row per K stage, fetched with cp.async several stages ahead
//                (zero fill for padding) and expanded into the 128B-swizzled
//                K-major A tile;
//   warp 8       TMA producer of the prepared filter tile (B);
//   warp 9       TMEM allocation and the single-thread tcgen05.mma issue;
//   warps 10-17  epilogue: tcgen05.ld of the finished accumulator buffer
//                (two buffers, so it overlaps the next tile's mainloop),
//                thresholds, 2-bit packing, stores.
// The K-stage pipeline runs continuously across a CTA's tiles.
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
  int nt;                // number of BN-wide output-channel tiles
  int ntiles;            // M tiles * nt
  int ntab;              // entries of the K-granule table (Kpad / codes per granule)
};

constexpr int kBK = 128;         // K elements (= bytes) per pipeline stage
constexpr int kRawRow = 32;      // packed bytes of one A row per stage (128 codes)
constexpr int kGatherWarps = 8;
constexpr int kEpiWarps = 8;
constexpr int kTcThreads = 32 * (kGatherWarps + 2 + kEpiWarps);   // 576
constexpr int kWarpTma = kGatherWarps, kWarpMma = kGatherWarps + 1, kWarpEpi0 = kGatherWarps + 2;
constexpr int kMaxTab = 1024;    // K-granule table entries

// Byte offset of 16-byte chunk `chunk` of row r inside a K-major 128B-swizzled tile.
__device__ __forceinline__ uint32_t sw128_chunk(int r, int chunk) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((chunk ^ (r & 7)) << 4));
}
// Raw staging: row r, 32 bytes; 16-byte halves swapped on alternate groups of 4 rows.
__device__ __forceinline__ uint32_t raw_off(int r, int half) {
  return (uint32_t)(r * kRawRow + (((half ^ (r >> 2)) & 1) << 4));
}

template <int BN, int SUB, int STAGES, int RAW>
struct TcSmem {
  static constexpr int kRows = 128 * SUB;
  static constexpr int kA = kRows * kBK;          // expanded A per stage
  static constexpr int kB = BN * kBK;
  static constexpr int kRaw = kRows * kRawRow;    // packed A per stage
  static constexpr int offA = 0;
  static constexpr int offB = offA + STAGES * kA;
  static constexpr int offRaw = offB + STAGES * kB;
  static constexpr int offThr = offRaw + RAW * kRaw;       // 2 buffers of BN float4
  static constexpr int offTab = offThr + 2 * BN * 16;      // kMaxTab x int2
  static constexpr int offBar = offTab + kMaxTab * 8;
  static constexpr int nBar = 3 * STAGES + 5;              // full_a, full_b, empty, acc_full[2], acc_empty[2], done
  static constexpr int offTmem = offBar + nBar * 8;
  static constexpr int bytes = offTmem + 16 + 1024;        // + alignment slack
};

__device__ __forceinline__ void expand_store(uint32_t addr, uint32_t u) {
  // 16 codes -> 16 e4m3 bytes; byte t of word q holds code 4t + q
  const uint32_t o0 = u & 0x03030303u, o1 = (u >> 2) & 0x03030303u;
  const uint32_t o2 = (u >> 4) & 0x03030303u, o3 = (u >> 6) & 0x03030303u;
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(o0), "r"(o1), "r"(o2), "r"(o3) : "memory");
}

// The input row (output pixel) that a gather unit reads in one tile: a base
// pointer for tap (0,0) (possibly outside the image; dereferenced only when
// valid) and bitmasks of the taps dy / dx that fall inside the image.
struct RowGeom {
  const uint8_t* base;
  uint32_t vy, vx;
};

__device__ __forceinline__ RowGeom row_geom(const ConvArgs& a, int m) {
  RowGeom g;
  g.base = a.x;
  g.vy = g.vx = 0;
  if (m < a.M) {
    const int hw = a.ho * a.wo;
    const int b = m / hw, rem = m - b * hw;
    const int oy = rem / a.wo, ox = rem - oy * a.wo;
    const int iy0 = oy * a.stride - a.pad, ix0 = ox * a.stride - a.pad;
    const int cinb = a.cin >> 2;
    g.base = a.x + ((long long)b * a.h * a.w + (long long)iy0 * a.w + ix0) * cinb;
    for (int d = 0; d < a.kh; ++d)
      if ((unsigned)(iy0 + d) < (unsigned)a.h) g.vy |= 1u << d;
    for (int d = 0; d < a.kw; ++d)
      if ((unsigned)(ix0 + d) < (unsigned)a.w) g.vx |= 1u << d;
  }
  return g;
}

// GB: bytes per gathered granule: 16 (cin % 64 == 0), 4 (cin % 16 == 0), 1 (cin % 4 == 0).
template <int BN, int SUB, int STAGES, int RAW, int GB>
__global__ void __launch_bounds__(kTcThreads, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap tmap_w, const ConvArgs args) {
  using L = TcSmem<BN, SUB, STAGES, RAW>;
  constexpr int kRows = L::kRows;
  extern __shared__ uint8_t smem_raw_[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw_ + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sA = sbase + L::offA, sB = sbase + L::offB, sRaw = sbase + L::offRaw;
  float4* sThr = (float4*)(smem + L::offThr);
  int2* sTab = (int2*)(smem + L::offTab);
  const uint32_t barBase = sbase + L::offBar;
  auto full_a = [&](int s) { return barBase + 8u * s; };
  auto full_b = [&](int s) { return barBase + 8u * (STAGES + s); };
  auto empty = [&](int s) { return barBase + 8u * (2 * STAGES + s); };
  auto acc_full = [&](int b) { return barBase + 8u * (3 * STAGES + b); };
  auto acc_empty = [&](int b) { return barBase + 8u * (3 * STAGES + 2 + b); };
  const uint32_t done_bar = barBase + 8u * (3 * STAGES + 4);
  uint32_t* tmem_slot = (uint32_t*)(smem + L::offTmem);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr uint32_t kCols = 2 * SUB * BN;   // two buffers x SUB accumulators
  const int G = gridDim.x;
  const int n_local = (args.ntiles - (int)blockIdx.x + G - 1) / G;
  const int nk = args.nk;

  // ---- setup (reads no global memory, so it may overlap the previous grid)
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(tmem_slot), kCols);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_a(s), kGatherWarps);
      mbar_init(full_b(s), 1);
      mbar_init(empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), kEpiWarps);
    }
    mbar_init(done_bar, 1);
    fence_mbar_init();
  }
  if (warp == kWarpTma && lane == 0) prefetch_tmap(&tmap_w);
  // K-granule table: byte offset of each granule from the row's tap-(0,0)
  // pointer, and its tap (dy, dx); dy = 0xFF past K.
  {
    const int cinb = args.cin >> 2;
    for (int gk = tid; gk < args.ntab; gk += kTcThreads) {
      const int k0 = gk * 4 * GB;
      const int tap = k0 / args.cin, cc = k0 - tap * args.cin;
      int2 e = make_int2(0, 0xFF << 8);
      if (tap < args.kh * args.kw) {
        const int dy = tap / args.kw, dx = tap - dy * args.kw;
        e = make_int2((dy * args.w + dx) * cinb + (cc >> 2), (dy << 8) | dx);
      }
      sTab[gk] = e;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_launch();
  grid_dep_wait();

  if (warp < kGatherWarps) {
    // =================== gather (im2col + expansion) ===================
    // unit u = tid + 256*i (i < SUB): row u % kRows, half (64 codes) u / kRows
    constexpr int kUnits = SUB;
    int urow[kUnits], uhalf[kUnits];
#pragma unroll
    for (int i = 0; i < kUnits; ++i) {
      const int u = tid + 256 * i;
      urow[i] = u % kRows;
      uhalf[i] = u / kRows;
    }
    const int total = n_local * nk;
    auto geom = [&](int jt, RowGeom (&g)[kUnits]) {
      const int t = (int)blockIdx.x + jt * G;
      const int mt = t / args.nt;
#pragma unroll
      for (int i = 0; i < kUnits; ++i) g[i] = row_geom(args, mt * kRows + urow[i]);
    };
    auto gather_unit = [&](const RowGeom& g, int stage_k, int half, uint32_t dst) {
      // 16 bytes of packed codes for K positions stage_k*128 + half*64 .. +64
      if constexpr (GB == 16) {
        const int2 e = sTab[stage_k * 2 + half];
        const int dy = e.y >> 8, dx = e.y & 0xFF;
        const bool ok = dy != 0xFF && ((g.vy >> dy) & (g.vx >> dx) & 1u);
        cp_async_16(dst, ok ? g.base + e.x : args.x, ok ? 16u : 0u);
      } else if constexpr (GB == 4) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int2 e = sTab[stage_k * 8 + half * 4 + q];
          const int dy = e.y >> 8, dx = e.y & 0xFF;
          const bool ok = dy != 0xFF && ((g.vy >> dy) & (g.vx >> dx) & 1u);
          cp_async_4(dst + 4 * q, ok ? g.base + e.x : args.x, ok ? 4u : 0u);
        }
      }
    };
    if constexpr (GB >= 4) {
      constexpr int D = RAW - 1;   // stages in flight ahead of the expansion
      int i_tile = 0, i_k = 0;
      RowGeom g[kUnits];
      geom(0, g);
      auto issue = [&](int it) {
        const uint32_t slot = sRaw + (uint32_t)((it % RAW) * L::kRaw);
#pragma unroll
        for (int i = 0; i < kUnits; ++i) gather_unit(g[i], i_k, uhalf[i], slot + raw_off(urow[i], uhalf[i]));
        if (++i_k == nk) {
          i_k = 0;
          if (++i_tile < n_local) geom(i_tile, g);
        }
      };
#pragma unroll 1
      for (int d = 0; d < D; ++d) {
        if (d < total) issue(d);
        cp_async_commit();
      }
#pragma unroll 1
      for (int it = 0; it < total; ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
        if (it + D < total) issue(it + D);
        cp_async_commit();
        cp_async_wait<D>();
        if (!mbar_wait(empty(s), ph ^ 1u)) break;
        const uint32_t slot = sRaw + (uint32_t)((it % RAW) * L::kRaw);
        const uint32_t dstA = sA + (uint32_t)(s * L::kA);
#pragma unroll
        for (int i = 0; i < kUnits; ++i) {
          uint32_t u0, u1, u2, u3;
          asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];"
                       : "=r"(u0), "=r"(u1), "=r"(u2), "=r"(u3)
                       : "r"(slot + raw_off(urow[i], uhalf[i])));
          const int r = urow[i] & 127, c0 = uhalf[i] * 4;
          const uint32_t rowA = dstA + (uint32_t)((urow[i] >> 7) * 16384);
          expand_store(rowA + sw128_chunk(r, c0 + 0), u0);
          expand_store(rowA + sw128_chunk(r, c0 + 1), u1);
          expand_store(rowA + sw128_chunk(r, c0 + 2), u2);
          expand_store(rowA + sw128_chunk(r, c0 + 3), u3);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(full_a(s));
      }
      cp_async_wait<0>();
    } else {
      // narrow channels (cin % 16 != 0): byte loads, 4 codes per byte, 16 bytes per unit
      int it = 0;
      bool ok = true;
#pragma unroll 1
      for (int jt = 0; jt < n_local && ok; ++jt) {
        RowGeom g[kUnits];
        geom(jt, g);
#pragma unroll 1
        for (int k = 0; k < nk; ++k, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
          uint32_t word[kUnits][4];
#pragma unroll
          for (int i = 0; i < kUnits; ++i)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              uint32_t v = 0;
#pragma unroll
              for (int bq = 0; bq < 4; ++bq) {
                const int2 e = sTab[k * 32 + uhalf[i] * 16 + q * 4 + bq];
                const int dy = e.y >> 8, dx = e.y & 0xFF;
                const bool okb = dy != 0xFF && ((g[i].vy >> dy) & (g[i].vx >> dx) & 1u);
                if (okb) v |= (uint32_t)__ldg(g[i].base + e.x) << (8 * bq);
              }
              word[i][q] = v;
            }
          if (!mbar_wait(empty(s), ph ^ 1u)) { ok = false; break; }
          const uint32_t dstA = sA + (uint32_t)(s * L::kA);
#pragma unroll
          for (int i = 0; i < kUnits; ++i) {
            const int r = urow[i] & 127, c0 = uhalf[i] * 4;
            const uint32_t rowA = dstA + (uint32_t)((urow[i] >> 7) * 16384);
#pragma unroll
            for (int q = 0; q < 4; ++q) expand_store(rowA + sw128_chunk(r, c0 + q), word[i][q]);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(full_a(s));
        }
      }
    }
  } else if (warp == kWarpTma) {
    // =================== TMA producer (filters) ===================
    if (lane == 0) {
      int it = 0;
      bool ok = true;
#pragma unroll 1
      for (int jt = 0; jt < n_local && ok; ++jt) {
        const int t = (int)blockIdx.x + jt * G;
        const int n0 = (t % args.nt) * BN;
#pragma unroll 1
        for (int k = 0; k < nk; ++k, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
          if (!mbar_wait(empty(s), ph ^ 1u)) { ok = false; break; }
          mbar_arrive_expect_tx(full_b(s), (uint32_t)L::kB);
          tma_load_2d(sB + (uint32_t)(s * L::kB), &tmap_w, full_b(s), k * kBK, n0);
        }
      }
      // drain: the last load into each slot has landed before the CTA may exit
      for (int i = it - STAGES < 0 ? 0 : it - STAGES; i < it; ++i)
        mbar_wait(full_b(i % STAGES), (uint32_t)(i / STAGES) & 1u);
    }
    __syncwarp();
  } else if (warp == kWarpMma) {
    // =================== MMA issue ===================
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_e4m3_f32(128, BN);
      int it = 0;
      bool ok = true;
#pragma unroll 1
      for (int jt = 0; jt < n_local && ok; ++jt) {
        const int ab = jt & 1;
        if (!mbar_wait(acc_empty(ab), ((uint32_t)(jt >> 1) & 1u) ^ 1u)) break;
        tc_fence_after();
        const uint32_t dacc = tmem + (uint32_t)(ab * SUB * BN);
#pragma unroll 1
        for (int k = 0; k < nk; ++k, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
          if (!mbar_wait(full_a(s), ph) || !mbar_wait(full_b(s), ph)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = sA + (uint32_t)(s * L::kA), b0 = sB + (uint32_t)(s * L::kB);
#pragma unroll
          for (int kk = 0; kk < kBK / 32; ++kk)
#pragma unroll
            for (int sub = 0; sub < SUB; ++sub)
              mma_e4m3(dacc + (uint32_t)(sub * BN), sdesc_sw128(a0 + sub * 16384 + 32 * kk),
                       sdesc_sw128(b0 + 32 * kk), idesc, (k | kk) != 0 ? 1u : 0u);
          mma_commit(empty(s));
        }
        if (ok) mma_commit(acc_full(ab));
      }
      mma_commit(done_bar);   // fires once every MMA issued above has completed
    }
    __syncwarp();
  } else {
    // =================== epilogue ===================
    // SUB = 2: warp pair e, e+4 covers lane quarter (warp % 4) of accumulators 0 and 1, all columns.
    // SUB = 1: warp pair e, e+4 covers lane quarter (warp % 4), column halves 0 and 1.
    constexpr int CW = SUB == 2 ? BN : BN / 2;   // columns per thread
    const int e = warp - kWarpEpi0;             // 0..7
    const int et = tid - kWarpEpi0 * 32;        // 0..255
    const int quarter = warp & 3;
    const int sub = SUB == 2 ? (e >> 2) : 0;
    const int c_lo = SUB == 2 ? 0 : (e >> 2) * CW;
    const int row = sub * 128 + quarter * 32 + lane;   // row of the tile
    bool ok = true;   // after a timed-out wait, keep only the named barriers (uniform over the 8 warps)
#pragma unroll 1
    for (int jt = 0; jt < n_local; ++jt) {
      const int t = (int)blockIdx.x + jt * G;
      const int n0 = (t % args.nt) * BN;
      const int m = (t / args.nt) * kRows + row;
      const int tb = args.nt > 1 ? (jt & 1) : 0;
      if (jt == 0 || args.nt > 1) {
        for (int c = et; c < BN; c += 256) {
          const int nn = n0 + c;
          float4 v = make_float4(0.f, 0.f, 0.f, 1.f);
          if (nn < args.cout && args.thr) {
            // sign*A > T  <=>  sign*D > T/512 with D = A/512 (exact in fp32)
            v = make_float4((float)args.thr[3 * nn] * (1.0f / 512.0f), (float)args.thr[3 * nn + 1] * (1.0f / 512.0f),
                            (float)args.thr[3 * nn + 2] * (1.0f / 512.0f), (float)args.sign[nn]);
          }
          sThr[tb * BN + c] = v;
        }
        named_bar(1, kEpiWarps * 32);
      }
      const int ab = jt & 1;
      if (ok) ok = mbar_wait(acc_full(ab), (uint32_t)(jt >> 1) & 1u);
      if (!ok) continue;
      tc_fence_after();
      const uint32_t tacc = tmem + (uint32_t)((ab * SUB + sub) * BN + c_lo) + ((uint32_t)(quarter * 32) << 16);
      const float4* th = sThr + tb * BN + c_lo;
      uint32_t packed[CW / 16];
#pragma unroll
      for (int c0 = 0; c0 < CW; c0 += 16) {
        uint32_t v[16];
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
              "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
            : "r"(tacc + c0)
            : "memory");
        tmem_ld_wait();
        uint32_t wd = 0;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float4 tq = th[c0 + j];
          const float sv = __uint_as_float(v[j]) * tq.w;
          const uint32_t code = (uint32_t)(sv > tq.x) + (uint32_t)(sv > tq.y) + (uint32_t)(sv > tq.z);
          wd |= code << (2 * j);
        }
        packed[c0 / 16] = wd;
        if (args.y_acc && m < args.M) {
          const int cbase = n0 + c_lo + c0;
          int32_t* dst = args.y_acc + (size_t)m * args.cout + cbase;
          if (cbase + 16 <= args.cout && (args.cout & 3) == 0) {
#pragma unroll
            for (int j = 0; j < 16; j += 4)
              *(int4*)(dst + j) = make_int4(__float2int_rn(__uint_as_float(v[j]) * 512.0f),
                                            __float2int_rn(__uint_as_float(v[j + 1]) * 512.0f),
                                            __float2int_rn(__uint_as_float(v[j + 2]) * 512.0f),
                                            __float2int_rn(__uint_as_float(v[j + 3]) * 512.0f));
          } else {
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (cbase + j < args.cout) dst[j] = __float2int_rn(__uint_as_float(v[j]) * 512.0f);
          }
        }
      }
      // the accumulator buffer may be refilled once every epilogue warp has read it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty(ab));
      if (args.y_codes && m < args.M) {
        const int rowb = args.cout >> 2;        // bytes per output pixel
        const int cb = n0 + c_lo;               // first channel of this thread
        uint8_t* dst = args.y_codes + (size_t)m * rowb + (cb >> 2);
        if (cb + CW <= args.cout && CW >= 64 && (rowb & 15) == 0 && (cb & 63) == 0) {
#pragma unroll
          for (int q = 0; q < CW / 64; ++q)
            *(uint4*)(dst + 16 * q) =
                make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
        } else if (cb + CW <= args.cout && (rowb & 3) == 0 && (cb & 15) == 0) {
#pragma unroll
          for (int q = 0; q < CW / 16; ++q) *(uint32_t*)(dst + 4 * q) = packed[q];
        } else {
          const int nbytes = max(0, min(CW, args.cout - cb)) >> 2;
          for (int q = 0; q < nbytes; ++q) dst[q] = (uint8_t)(packed[q >> 2] >> (8 * (q & 3)));
        }
      }
    }
  }

  // ---- teardown: every MMA has completed (done_bar) before TMEM is released
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    mbar_wait(done_bar, 0);
    tmem_dealloc(tmem, kCols);
  }
}

}  // namespace ifq
