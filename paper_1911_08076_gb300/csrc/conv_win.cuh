// Window path of the quantized convolution (Eq. (1) integer core, Eq. (7)
// thresholds fused as the epilogue) for stride-1 k x k layers with "same"
// padding, on the sm_103a tensor cores.
//
// GEMM view with the output pixels on the MMA's N side:
//   D[m][j] = sum_K A[m][K] * B[j][K],   m = (sy, n): output row offset sy and
//   output channel n of the tile; j = an anchor pixel of the tile's band.
//
// B is the input itself.  A tile's input rows are copied to shared memory by
// the copy engine (cp.async.bulk: an image row of packed codes is contiguous)
// and expanded once into a band of e4m3 bytes (a 2-bit code c is the e4m3
// byte c, c * 2^-9): one 16-byte slot per pixel and 16-channel plane, zero
// slots for the padding.  The MMA's B operand for one tap (dy, dx) is that band
// read at an offset of dy rows and dx slots: in the non-swizzled K-major layout
// a core matrix is 8 rows of 16 bytes, 16 bytes apart, so consecutive anchors
// are consecutive slots and every tap is just another descriptor over the same
// bytes.  No im2col copy is ever made.
//
// A is the filter bank, made resident in shared memory once per CTA as a
// block-Toeplitz matrix: row (sy, n) holds w[n][iy - sy][ix][c] at K position
// (iy, ix, c) for 0 <= iy - sy < k, zero elsewhere.  So accumulator row
// (sy, n) computes output row sy of the anchor's row band for channel n, and
// with 128 / cout output rows stacked along M a layer with few channels still
// fills the 128 lanes of the MMA.  The prepared filter rows (ifq_pack_weights:
// e4m3 +-1, natural (dy, dx, c) order with the intra-word order of the code
// expansion) are its source: the rows of one sy are the filters shifted along K
// by sy k cin bytes, so the copy engine loads them as 128-byte-swizzled boxes.
//
// Anchors.  With one output row per M row (cout >= 128) the tile's R anchor
// rows are consecutive output rows and share the band's input rows (R + k - 1
// of them, `seg_pitch` = pitch slots apart).  With rows stacked along M, a
// tile is R row bands of `ry` output rows side by side along N: band row iy
// holds input row iy of each of the R bands, `pitch` slots each, so a tap's
// offset is the same for every anchor.  Either way anchor j is (r, x) =
// (j / pitch, j % pitch), and columns with x >= w are computed and dropped.
//
// Exactness is that of the main path: every product is +-c * 2^-9 and every
// partial sum an integer multiple of 2^-9 far inside the fp32 significand
// (the planner admits 3 K <= 196608), so D = A_int / 512 exactly.
//
// Epilogue: tensor-memory lane m is one output channel of one output row, so
// its three thresholds and its sign are per-thread constants.  Each step
// [sign * A > T_i] is an exact saturated fma of D (see sat_fma), the sign
// folded into the multiplier.  The codes of 32 channels of one pixel are
// gathered with two warp ballots (bit 1 and bit 0 of the code) and packed into
// the 8 bytes those channels occupy in the NHWC output.  The fused 2 x 2 pool (Sec. 2.1: on
// Y^conv, before BN and the quantizer) takes the max of A over the
// horizontal pair in registers; the vertical pair is either two anchor rows
// of the same thread (one output row per M row) or two warps (stacked output
// rows), which swap halves of their horizontal maxima through shared memory,
// so each thresholds the window maximum of half the pooled columns.
//
// Warps: 0-15 epilogue (lane quadrant = warp % 4, four warps a quadrant on
// interleaved column groups), 16 TMEM allocation and MMA issue, 17-20
// producers (one lane of warp 17 issues the bulk copies).  Two
// staging buffers, two bands and two accumulators, so the copy of tile i+2,
// the expansion of tile i+1, the MMAs of tile i and the epilogue of tile i-1
// overlap.  Every wait is bounded (IFQ_ETIMEOUT, then the roles leave their
// loops; warps sharing a named barrier keep reaching it).
#pragma once
#include "conv_common.cuh"

namespace ifq {

constexpr int kWinEpiPerQ = 4;         // epilogue warps per tensor-memory lane quadrant
constexpr int kWinEpiWarps = 4 * kWinEpiPerQ;
constexpr int kWinMmaWarp = kWinEpiWarps;
constexpr int kWinProd0 = kWinEpiWarps + 1;
constexpr int kWinProdWarps = 4;
constexpr int kWinThreads = 32 * (kWinEpiWarps + 1 + kWinProdWarps);   // 672
constexpr int kWinPoolGroups = 4;      // groups of 32 pooled columns a tile can have (N <= 256)
constexpr int kWinGpw = (kWinPoolGroups + kWinEpiPerQ - 1) / kWinEpiPerQ;   // of them per epilogue warp
constexpr int kWinProdBar = 1 + 2 * kWinEpiPerQ;   // producers' named barrier (1..2 kWinEpiPerQ: row pairs)
constexpr int kWinXchgBytes = 3 * kWinEpiWarps * 2048;   // horizontal maxima of the row pairs (stacked rows, pooled)
constexpr int kWinMaxMma = 64;         // MMAs per tile (K' / 32)
constexpr int kWinTabBytes = 8 * kWinMaxMma;
constexpr int kWinStashBytes = kWinEpiWarps * 32 * 8;   // per epilogue warp, 32 pairs of ballots
constexpr int kWinMaxSmem = 232448;    // dynamic shared memory per CTA

struct WinArgs {
  const uint8_t* x;        // packed 2-bit NHWC input codes
  const uint8_t* w_prep;   // prepared e4m3 filter rows [cout][Kpad]
  const int32_t* thr;      // [cout][3]
  const int8_t* sign;      // [cout]
  uint8_t* y_codes;        // packed 2-bit output codes (after the fused pool) or nullptr
  int32_t* y_acc;          // int32 accumulators or nullptr (never with a fused pool)
  int n, h, w, cin, cout, k, pad, Kpad;
  int planes;       // cin / 16
  int ct;           // output channels of a tile; M = ry * ct = 128
  int ry;           // output rows stacked along M
  int nct;          // channel tiles, cout / ct
  int R;            // anchor rows of a tile
  int rows;         // output rows a tile covers: ry * R
  int pitch;        // slots of one anchor row
  int seg_pitch;    // slots between band rows: pitch (ry = 1) or R * pitch (ry > 1)
  int nseg;         // row bands staged per tile: 1 (ry = 1) or R
  int N;            // MMA N: anchors per tile, a multiple of 16, <= 256
  int rb;           // band rows: R + k - 1 (ry = 1) or ry + k - 1
  int kc;           // 16-byte core columns of the Toeplitz K (even)
  int kc_real;      // of which carry filter bytes: (ry + k - 1) * k * planes
  int bands;        // tiles per image and channel tile
  int ntiles;       // n * bands (per channel tile)
  int row_bytes;    // packed bytes of one input row (a multiple of 16)
  uint32_t plane_stride;   // bytes between the planes of a band buffer
  uint32_t band_bytes;     // bytes of one band buffer
  uint32_t stage_bytes;    // bytes of one staging buffer (nseg * rb * row_bytes, rounded)
  uint32_t a_bytes;        // bytes of the resident A operand: 16 KB per 128-byte K stage of the Toeplitz K
  uint32_t xchg_bytes;     // row-pair exchange buffers: kWinXchgBytes with stacked rows and a pool, else 0
  int early;               // 1: no kernel before this one in the stream writes the filters
  FastDiv div_planes, div_pitch, div_seg, div_bands, div_chunks, div_rb;
};

// Shared-memory descriptor of a K-major operand in the non-swizzled layout: core matrices of
// 8 rows x 16 bytes, `lbo` bytes apart along K and `sbo` bytes apart along M/N.
__device__ __forceinline__ uint64_t sdesc_none(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46);
}

// 32 lanes x 32 consecutive columns of tensor memory -> 32 registers, with the wait in the same
// asm statement (the destination registers are written asynchronously until the wait).
__device__ __forceinline__ void tmem_ld32_sync(uint32_t t0, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(t0)
      : "memory");
}

// Two loads of 32 columns (at t0 and t1) in flight together, one wait: 64 registers.
__device__ __forceinline__ void tmem_ld2x32_sync(uint32_t t0, uint32_t t1, uint32_t (&v)[64]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%64];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%65];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31]), "=r"(v[32]), "=r"(v[33]), "=r"(v[34]), "=r"(v[35]), "=r"(v[36]), "=r"(v[37]), "=r"(v[38]), "=r"(v[39]), "=r"(v[40]), "=r"(v[41]), "=r"(v[42]), "=r"(v[43]), "=r"(v[44]), "=r"(v[45]), "=r"(v[46]), "=r"(v[47]), "=r"(v[48]), "=r"(v[49]), "=r"(v[50]), "=r"(v[51]), "=r"(v[52]), "=r"(v[53]), "=r"(v[54]), "=r"(v[55]), "=r"(v[56]), "=r"(v[57]), "=r"(v[58]), "=r"(v[59]), "=r"(v[60]), "=r"(v[61]), "=r"(v[62]), "=r"(v[63])
      : "r"(t0), "r"(t1)
      : "memory");
}

// Two loads of 16 columns (at t0 and t1) in flight together, one wait: 32 registers.
__device__ __forceinline__ void tmem_ld2x16_sync(uint32_t t0, uint32_t t1, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%32];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%33];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
        "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(t0), "r"(t1)
      : "memory");
}

// 32 bits -> 64 bits with bit i at bit 2i.
__device__ __forceinline__ uint64_t spread_bits(uint32_t x) {
  uint64_t v = x;
  v = (v | (v << 16)) & 0x0000FFFF0000FFFFull;
  v = (v | (v << 8)) & 0x00FF00FF00FF00FFull;
  v = (v | (v << 4)) & 0x0F0F0F0F0F0F0F0Full;
  v = (v | (v << 2)) & 0x3333333333333333ull;
  v = (v | (v << 1)) & 0x5555555555555555ull;
  return v;
}

// Byte offset in a band buffer of 16-byte core column c = (iy, ix, p) of the Toeplitz K, for
// anchor 0.
__device__ __forceinline__ uint32_t win_col_offset(const WinArgs& a, int c) {
  const int p = c % a.planes, t = c / a.planes;
  const int iy = t / a.k, ix = t - iy * a.k;
  return (uint32_t)p * a.plane_stride + 16u * (uint32_t)(iy * a.seg_pitch + ix);
}

// First output row of tile t's anchor row r (rows of a tile: R anchor rows of ry output rows).
__device__ __forceinline__ int win_row(const WinArgs& a, int y0, int r) { return y0 + r * a.ry; }

template <int POOL, int ACC>
__global__ void __launch_bounds__(kWinThreads, 1)
    conv_win_kernel(const __grid_constant__ CUtensorMap tmap_a, const WinArgs a) {
  extern __shared__ uint8_t smem_raw_[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw_ + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sA = sbase;
  const uint32_t sBand = sbase + a.a_bytes;
  const uint32_t oStage = a.a_bytes + 2 * a.band_bytes;
  const uint32_t sStage = sbase + oStage;
  const uint32_t oXchg = oStage + 2 * a.stage_bytes;
  float4* xchg4 = (float4*)(smem + oXchg);
  uint64_t* mtab = (uint64_t*)(smem + oXchg + a.xchg_bytes);   // B descriptors of band 0, per MMA
  const uint32_t barBase = sbase + oXchg + a.xchg_bytes + kWinTabBytes;
  auto band_full = [&](int b) { return barBase + 8u * b; };
  auto band_empty = [&](int b) { return barBase + 16u + 8u * b; };
  auto acc_full = [&](int b) { return barBase + 32u + 8u * b; };
  auto acc_empty = [&](int b) { return barBase + 48u + 8u * b; };
  auto stage_full = [&](int b) { return barBase + 64u + 8u * b; };
  const uint32_t done_bar = barBase + 80u;
  const uint32_t a_full = barBase + 88u;   // the resident A operand has landed
  uint32_t* tmem_slot = (uint32_t*)(smem + oXchg + a.xchg_bytes + kWinTabBytes + 104);
  uint2* win_stash = (uint2*)(smem + oXchg + a.xchg_bytes + kWinTabBytes + 128);   // 32 ballot pairs a warp

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // CTA c takes channel tile c % nct and the band tiles c / nct, c / nct + G / nct, ... of it
  const int ctile = (int)blockIdx.x % a.nct;
  const int first = (int)blockIdx.x / a.nct, step = (int)gridDim.x / a.nct;
  const int n_local = first < a.ntiles ? (a.ntiles - first + step - 1) / step : 0;
  const int nmma = a.kc >> 1;

  if (warp == kWinMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), 512);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(band_full(b), kWinProdWarps);
      mbar_init(band_empty(b), 1);
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), kWinEpiWarps);
      mbar_init(stage_full(b), 1);
    }
    mbar_init(done_bar, 1);
    mbar_init(a_full, 1);
    fence_mbar_init();
  }
  // B descriptors of band buffer 0, one per MMA: the pair of core columns (2q, 2q + 1); past the
  // filter bytes (where A is zero) the second one is the slot after the first
  if (tid < nmma) {
    const int c0 = 2 * tid;
    const uint32_t b0 = win_col_offset(a, c0);
    const uint32_t b1 = c0 + 1 < a.kc_real ? win_col_offset(a, c0 + 1) : b0 + 16u;
    mtab[tid] = sdesc_none(sBand + b0, b1 - b0, 128u);
  }
  grid_dep_wait();
  // both band buffers start as zeros: padding slots and the tail past the band stay zero
  for (uint32_t o = (uint32_t)tid * 16u; o < 2u * a.band_bytes; o += kWinThreads * 16u)
    *(uint4*)(smem + a.a_bytes + o) = make_uint4(0u, 0u, 0u, 0u);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_launch();

  if (warp >= kWinProd0) {
    // =================== producers: bulk copy of packed rows, expansion into the band ===================
    const int pt = tid - kWinProd0 * 32;   // 0..127
    const int cinb = a.cin >> 2;           // packed bytes per pixel
    const bool issuer = pt == 0;
    // rows of tile i staged in buffer i & 1: segment s (row band of ry * s output rows below y0)
    // holds input rows y0 + s ry - pad + iy, iy < rb, at (s rb + iy) row_bytes; rows outside the
    // image are not copied (their slots expand to zeros)
    auto issue = [&](int i) {
      const int t = first + i * step;
      const int b = (int)fdiv((uint32_t)t, a.div_bands);
      const int y0 = (t - b * a.bands) * a.rows;
      const uint8_t* img = a.x + (size_t)b * a.h * a.row_bytes;
      const uint32_t dst = sStage + (uint32_t)(i & 1) * a.stage_bytes;
      uint32_t total = 0;
      for (int s = 0; s < a.nseg; ++s) {
        const int top = win_row(a, y0, s) - a.pad;
        const int r0 = max(0, top), r1 = min(a.h, top + a.rb);
        if (r1 > r0) total += (uint32_t)((r1 - r0) * a.row_bytes);
      }
      mbar_arrive_expect_tx(stage_full(i & 1), total);
      for (int s = 0; s < a.nseg; ++s) {
        const int top = win_row(a, y0, s) - a.pad;
        const int r0 = max(0, top), r1 = min(a.h, top + a.rb);
        if (r1 > r0)
          bulk_copy_g2s(dst + (uint32_t)((s * a.rb + (r0 - top)) * a.row_bytes), img + (size_t)r0 * a.row_bytes,
                        (uint32_t)((r1 - r0) * a.row_bytes), stage_full(i & 1));
      }
    };
    int issued = 0, waited = 0;   // tiles whose copies were issued / were waited for
    if (issuer && n_local > 0) {
      issue(0);
      issued = 1;
    }
    bool ok = true;
#pragma unroll 1
    for (int i = 0; i < n_local; ++i) {
      const int bb = i & 1;
      if (ok) {
        if (issuer && i + 1 < n_local) {   // stage (i + 1) & 1 was read in iteration i - 1, fenced by the barrier
          issue(i + 1);
          issued = i + 2;
        }
        bool got = mbar_wait(stage_full(bb), (uint32_t)(i >> 1) & 1u);
        if (got) waited = i + 1;
        got = got && mbar_wait_backoff(band_empty(bb), ((uint32_t)(i >> 1) & 1u) ^ 1u, 64);
        ok = __all_sync(0xffffffffu, got);
      }
      if (ok) {
        const int t = first + i * step;
        const int b = (int)fdiv((uint32_t)t, a.div_bands);
        const int y0 = (t - b * a.bands) * a.rows;
        const uint8_t* stg = smem + oStage + (size_t)bb * a.stage_bytes;
        const uint32_t dst0 = a.a_bytes + (uint32_t)bb * a.band_bytes;   // byte offset from smem
        // Row items: band row iy of row band s, 16 staged bytes (4 words) a thread.  A row inside
        // the image expands its words into their slots; a row outside it writes zeros into the
        // slots of its w pixels (the padding slots beside the rows are never written and stay
        // zero from the start).
        const int chunks = a.row_bytes >> 4;
        const int total = a.nseg * a.rb * chunks;
#pragma unroll 2
        for (int it = pt; it < total; it += 128) {
          const int row = (int)fdiv((uint32_t)it, a.div_chunks);   // staged row s rb + iy
          const int ch = it - row * chunks;
          const int s = (int)fdiv((uint32_t)row, a.div_rb);
          const int iy = row - s * a.rb;
          const int yy = win_row(a, y0, s) - a.pad + iy;
          uint4 w4 = make_uint4(0u, 0u, 0u, 0u);
          if (yy >= 0 && yy < a.h) w4 = *(const uint4*)(stg + (size_t)row * a.row_bytes + 16 * ch);
          const uint32_t ws[4] = {w4.x, w4.y, w4.z, w4.w};
          const uint32_t rowo = dst0 + 16u * (uint32_t)(iy * a.seg_pitch + s * a.pitch + a.pad);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int qw = 4 * ch + e;                               // word of the row
            const int xx = (int)fdiv((uint32_t)qw, a.div_planes);   // its pixel
            const int pl = qw - xx * a.planes;                      // and plane
            const uint32_t v = ws[e];
            *(uint4*)(smem + rowo + (uint32_t)pl * a.plane_stride + 16u * (uint32_t)xx) =
                make_uint4(v & 0x03030303u, v & 0x0C0C0C0Cu, (v >> 4) & 0x03030303u, (v >> 4) & 0x0C0C0C0Cu);
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(band_full(bb));
      }
      // every producer warp is done with staging buffer bb before a copy into it is issued
      named_bar(kWinProdBar, kWinProdWarps * 32);
    }
    // copies issued but never waited for (after a timed-out wait) land before the CTA may exit
    if (issuer) {
      for (int i = waited; i < issued; ++i) mbar_wait(stage_full(i & 1), (uint32_t)(i >> 1) & 1u);
    }
  } else if (warp == kWinMmaWarp) {
    // =================== MMA issue (one elected lane; the warp runs the loop) ===================
    const uint32_t idesc = idesc_e4m3_f32(128, a.N);
    // The resident A operand, loaded by the copy engine in 128-byte-swizzled K stages of 128 rows
    // x 128 bytes (the layout of a TMA box with 128B swizzle).  Row (sy, n) of the Toeplitz block
    // is filter n shifted by sy k cin bytes along K (tap row iy = dy + sy), so the rows of one sy
    // in K stage j are one box of the prepared filters at K = 128 j - sy k cin; the zeros before
    // and after the filter come from the box reading outside the rows (zero fill).
    if (!a.early) grid_dep_wait();
    if (lane == 0) mbar_arrive_expect_tx(a_full, a.a_bytes);
    __syncwarp();
    const int nst = (int)(a.a_bytes >> 14);
    for (int bx = lane; bx < nst * a.ry; bx += 32) {
      const int j = bx / a.ry, sy = bx - j * a.ry;
      tma_load_2d(sA + (uint32_t)j * 16384u + (uint32_t)(sy * a.ct) * 128u, &tmap_a, a_full,
                  128 * j - sy * a.k * a.cin, ctile * a.ct);
    }
    bool ok = __all_sync(0xffffffffu, mbar_wait(a_full, 0));
#pragma unroll 1
    for (int i = 0; i < n_local && ok; ++i) {
      const int bb = i & 1;
      const uint32_t ph = (uint32_t)(i >> 1) & 1u;
      bool got = mbar_wait(band_full(bb), ph);
      got = got && mbar_wait(acc_empty(bb), ph ^ 1u);
      if (!__all_sync(0xffffffffu, got)) {
        ok = false;
        break;
      }
      tc_fence_after();
      if (elect_one()) {
        const uint32_t dacc = tmem + (uint32_t)(bb * 256);
        const uint64_t boff = (uint64_t)(((uint32_t)bb * a.band_bytes) >> 4);
#pragma unroll 1
        for (int q = 0; q < nmma; ++q)
          mma_e4m3(dacc, sdesc_sw128(sA + (uint32_t)(q >> 2) * 16384u + (uint32_t)(q & 3) * 32u), mtab[q] + boff,
                   idesc, q > 0 ? 1u : 0u);
        mma_commit(band_empty(bb));
        mma_commit(acc_full(bb));
      }
      __syncwarp();
    }
    if (elect_one()) mma_commit(done_bar);
    __syncwarp();
  } else {
    // =================== epilogue: thresholds, code packing, fused pool, stores ===================
    // Warps q, q + 4, q + 8, ... share lane quadrant q (warp % 4) and take every kWinEpiPerQ-th
    // 32-column (pooled: 32 pooled-column) group, so each quadrant has several warps hiding each
    // other's latencies.
    const int q = warp & 3;                      // lane quadrant
    const int sub = warp >> 2;                   // which of the quadrant's column groups
    const int sy = (32 * q) / a.ct;              // output row offset of this quadrant
    const int cg = ((32 * q) % a.ct) >> 5;       // 32-channel group within the channel tile
    const int n = ctile * a.ct + cg * 32 + lane;
    // this lane's channel: -T1, -T2, -T3 and 512 s, so that sat_fma(D, 512 s, -T_i) = [s A > T_i]
    // exactly (D = A / 512; the FMA pipe, not the ALU pipe the compares would take)
    float nt1 = 0.f, nt2 = 0.f, nt3 = 0.f, s512 = 512.f;
    if (a.thr) {
      nt1 = -(float)a.thr[3 * n];
      nt2 = -(float)a.thr[3 * n + 1];
      nt3 = -(float)a.thr[3 * n + 2];
      s512 = 512.f * (float)a.sign[n];
    }
    // ballots of a column group, kept by lane 0 at [column] and read back by the column's lane
    const uint32_t stash = smem_u32(win_stash) + (uint32_t)warp * 256u;
    const int rowb = a.cout >> 2;                                  // output bytes per pixel
    const int chb = (ctile * a.ct + cg * 32) >> 2;                 // this warp's byte within a pixel
    const uint32_t lane_off = (uint32_t)(32 * q) << 16;
    // row pairs of stacked output rows (ry > 1, pooled): the odd row's warp hands its codes over
    const int pair = a.ct == 32 ? (q >> 1) : (q & 1);
    const bool odd_row = (sy & 1) != 0;
    // The code of one value is x1 + x2 + x3 with x_i = [s A > T_i] in {0, 1}, x1 >= x2 >= x3 (the
    // thresholds ascend): bit 1 is x2 and bit 0 is x1 - x2 + x3.  Their two warp ballots (the codes of
    // this warp's 32 channels for one pixel) go to the stash at the column's index (lane 0 stores,
    // one shared-memory store instead of a per-lane select), and packed() hands the column's lane its
    // pair: the 8 bytes those channels occupy in the NHWC output.  Warp-uniform calls only.
    auto code_ballot = [&](float f, int col, uint32_t&, uint32_t&) {
      const float x1 = sat_fma(f, s512, nt1), x2 = sat_fma(f, s512, nt2), x3 = sat_fma(f, s512, nt3);
      const uint32_t m1 = __ballot_sync(0xffffffffu, x2 > 0.5f);
      const uint32_t m0 = __ballot_sync(0xffffffffu, x1 - x2 + x3 > 0.5f);
      if (lane == 0)
        asm volatile("st.shared.v2.u32 [%0], {%1, %2};" ::"r"(stash + 8u * (uint32_t)col), "r"(m0), "r"(m1) : "memory");
    };
    auto packed = [&](uint32_t, uint32_t) {
      __syncwarp();
      uint32_t m0, m1;
      asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(m0), "=r"(m1) : "r"(stash + 8u * (uint32_t)lane) : "memory");
      __syncwarp();
      return spread_bits(m0) | (spread_bits(m1) << 1);
    };
    bool ok = true;
#pragma unroll 1
    for (int i = 0; i < n_local; ++i) {
      const int ab = i & 1;
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait_backoff(acc_full(ab), (uint32_t)(i >> 1) & 1u, 64));
      const int t = first + i * step;
      const int b = (int)fdiv((uint32_t)t, a.div_bands);
      const int y0 = (t - b * a.bands) * a.rows;
      const uint32_t tacc = tmem + (uint32_t)(ab * 256) + lane_off;
      if (ok) tc_fence_after();
      if constexpr (POOL == 0) {
        if (ok) {
#pragma unroll 1
          for (int g = sub; g * 32 < a.N; g += kWinEpiPerQ) {
            uint32_t v[32];
            tmem_ld32_sync(tacc + (uint32_t)(32 * g), v);
            uint32_t k0 = 0, k1 = 0;
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const float f = __uint_as_float(v[c]);
              code_ballot(f, c, k0, k1);
              if constexpr (ACC != 0) {
                const int j = 32 * g + c;
                const int r = (int)fdiv((uint32_t)j, a.div_pitch), xx = j - r * a.pitch;
                const int yy = win_row(a, y0, r) + sy;
                if (r < a.R && xx < a.w && yy < a.h)
                  a.y_acc[(((size_t)b * a.h + yy) * a.w + xx) * a.cout + n] = __float2int_rn(f * 512.0f);
              }
            }
            const int j = 32 * g + lane;
            const int r = (int)fdiv((uint32_t)j, a.div_pitch), xx = j - r * a.pitch;
            const int yy = win_row(a, y0, r) + sy;
            const uint64_t pk = packed(k0, k1);
            if (a.y_codes && r < a.R && xx < a.w && yy < a.h)
              *(uint64_t*)(a.y_codes + (((size_t)b * a.h + yy) * a.w + xx) * rowb + chb) = pk;
          }
        }
      } else {
        // pooled output map: (h / 2) x (w / 2); groups of 32 pooled columns, alternate ones per warp
        const int pw = a.w >> 1, ph = a.h >> 1;
        const int halfw = a.pitch >> 1;
        const int npool = a.ry > 1 ? (a.N >> 1) : (a.R >> 1) * halfw;
        if (a.ry > 1) {
          // Rows sy (even) and sy + 1 of each pooled window live in the two warps of a row pair.
          // Each warp takes the horizontal maxima of its 32 pooled columns, hands the half the
          // partner thresholds to it through shared memory (four 16-byte stores a lane), takes the
          // vertical max of the half it keeps (the even row keeps pooled columns 0..15 of the group,
          // the odd row 16..31) and thresholds only that: the quantizer sees max A over the whole
          // 2 x 2 window, as Sec. 2.1 places the pool.  Buffers alternate with the tile parity, so a
          // warp never overwrites a half its partner has not read yet.
          const int g = sub;   // kWinGpw == 1: one group of 32 pooled columns per warp
          const bool act = ok && 32 * g < npool;
          // slots of 128 float4 ([e4][lane]): one per epilogue warp for the half it keeps (read back
          // by the same lane), then one per tile parity and warp for the half it hands over; the
          // partner is the warp of the other row of the pair: quadrant q ^ (ct / 32), same sub
          float4* mine = xchg4 + (size_t)warp * 128;
          float4* give = xchg4 + (size_t)(kWinEpiWarps + (i & 1) * kWinEpiWarps + warp) * 128;
          const float4* take = xchg4 + (size_t)(kWinEpiWarps + (i & 1) * kWinEpiWarps + (warp ^ (a.ct >> 5))) * 128;
          auto half = [&](auto kept_c) {
            constexpr int kKept = decltype(kept_c)::value, kGive = 16 - kKept;
            // pooled columns [c, c + 16) come from accumulator columns [2 c, 2 c + 32); both halves
            // of this row's horizontal maxima go to shared memory (the kept one to this warp's own
            // slot), so nothing stays in registers across the barrier
            if (act) {
#pragma unroll
              for (int hh = 0; hh < 2; ++hh) {
                uint32_t v[32];
                tmem_ld32_sync(tacc + (uint32_t)(64 * g + 32 * hh), v);
                float4* dst = (hh == 0) == (kKept == 0) ? mine : give;
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                  float m4[4];
#pragma unroll
                  for (int j = 0; j < 4; ++j)
                    m4[j] = fmaxf(__uint_as_float(v[8 * q4 + 2 * j]), __uint_as_float(v[8 * q4 + 2 * j + 1]));
                  dst[q4 * 32 + lane] = make_float4(m4[0], m4[1], m4[2], m4[3]);
                }
              }
            }
            named_bar(1 + pair + 2 * sub, 64);
            if (act) {
              uint32_t k0 = 0, k1 = 0;
#pragma unroll
              for (int q4 = 0; q4 < 4; ++q4) {
                const float4 o = take[q4 * 32 + lane], m = mine[q4 * 32 + lane];
                code_ballot(fmaxf(m.x, o.x), 4 * q4, k0, k1);
                code_ballot(fmaxf(m.y, o.y), 4 * q4 + 1, k0, k1);
                code_ballot(fmaxf(m.z, o.z), 4 * q4 + 2, k0, k1);
                code_ballot(fmaxf(m.w, o.w), 4 * q4 + 3, k0, k1);
              }
              const int pi = 32 * g + kKept + lane;
              const int r = (int)fdiv((uint32_t)(2 * pi), a.div_pitch), xx = 2 * pi - r * a.pitch;
              const int py = (win_row(a, y0, r) + sy) >> 1, px = xx >> 1;
              const uint64_t pk = packed(k0, k1);
              if (a.y_codes && lane < 16 && pi < npool && r < a.R && px < pw && py < ph)
                *(uint64_t*)(a.y_codes + (((size_t)b * ph + py) * pw + px) * rowb + chb) = pk;
            }
          };
          if (odd_row) half(std::integral_constant<int, 16>{});
          else half(std::integral_constant<int, 0>{});
        } else {
        uint64_t own[kWinGpw];
#pragma unroll
        for (int gi = 0; gi < kWinGpw; ++gi) own[gi] = 0ull;
        if (ok) {
#pragma unroll
          for (int gi = 0; gi < kWinGpw; ++gi) {
            const int g = kWinEpiPerQ * gi + sub;
            if (32 * g < npool) {
              uint32_t k0 = 0, k1 = 0;
              {
                // pooled column (pr, px) <- columns 2 px, 2 px + 1 of anchor rows 2 pr and 2 pr + 1
                // (pitch % 16 == 0, so 8 pooled columns are 16 aligned columns of each row)
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                  uint32_t col[2];
#pragma unroll
                  for (int u = 0; u < 2; ++u) {
                    const int pi0 = 32 * g + 16 * hh + 8 * u;
                    const int pr = pi0 / halfw, px0 = pi0 - pr * halfw;
                    col[u] = pi0 < npool ? (uint32_t)(2 * pr * a.pitch + 2 * px0) : 0u;
                  }
#pragma unroll
                  for (int u = 0; u < 2; ++u) {
                    uint32_t v[32];   // 16 columns of the top row, then of the bottom row
                    tmem_ld2x16_sync(tacc + col[u], tacc + col[u] + (uint32_t)a.pitch, v);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                      const float top = fmaxf(__uint_as_float(v[2 * e]), __uint_as_float(v[2 * e + 1]));
                      const float bot = fmaxf(__uint_as_float(v[16 + 2 * e]), __uint_as_float(v[16 + 2 * e + 1]));
                      code_ballot(fmaxf(top, bot), 16 * hh + 8 * u + e, k0, k1);
                    }
                  }
                }
              }
              own[gi] = packed(k0, k1);
            }
          }
        }
        if (ok && a.y_codes) {
#pragma unroll
          for (int gi = 0; gi < kWinGpw; ++gi) {
            const int pi = 32 * (kWinEpiPerQ * gi + sub) + lane;
            const int pr = pi / halfw, px = pi - pr * halfw;
            const int py = (y0 >> 1) + pr;
            if (pi < npool && px < pw && py < ph)
              *(uint64_t*)(a.y_codes + (((size_t)b * ph + py) * pw + px) * rowb + chb) = own[gi];
          }
        }
        }
      }
      if (ok) {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty(ab));
      }
    }
  }

  // ---- teardown: every MMA has completed (done_bar) before tensor memory is released
  tc_fence_before();
  __syncthreads();
  if (warp == kWinMmaWarp) {
    tc_fence_after();
    mbar_wait(done_bar, 0);
    mbar_wait(a_full, 0);   // the A copies have landed (already true unless a wait ran out)
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace ifq
