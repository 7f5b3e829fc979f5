// Tensor-core path of the quantized convolution (Eq. (1) integer core with the
// thresholds of Eq. (7) fused as the epilogue), for sm_103a.
//
// GEMM view: D[m][n] = sum_k A[m][k] * B[n][k] with m = output pixel
// (b, oy, ox), n = output channel, k = (dy, dx, c) -- an implicit GEMM whose
// A rows are gathered on the fly from the packed k-bit NHWC input (k = 2 in
// 2-bit fields; k = 3, 4 in 4-bit fields, template parameter SB).
//
// Exact integer arithmetic on the fp8 tensor cores (sm_103a has no tcgen05
// integer MMA):
//   * A: code c in 0..15 is the e4m3 byte c, i.e. the value c * 2^-9
//     (subnormal below 8); the k-bit -> 8-bit expansion is a mask per byte lane.
//   * B: +1 / -1 are the e4m3 bytes 0x38 / 0xB8 (+-1.0), or 0x28 / 0xA8 (+-0.25)
//     at the K positions where the 2-bit expansion leaves a code as 4c.
//   * Every product is c * 2^-9 exactly; every partial sum is an integer
//     multiple of 2^-9 of magnitude <= (2^k - 1) K * 2^-9, far inside the
//     24-bit fp32 significand for the magnitudes the host admits, so the fp32
//     accumulator in tensor memory holds it exactly: D = A / 512.
//   * Thresholds: for 2-bit codes [sign*A > T] = sat(D * 512 sign - T), an exact integer
//     saturated to {0, 1} by one fma.sat on the FMA pipe; for 3- and 4-bit codes
//     sign*A > T  <=>  sign*D > T/512 (T/512 is exact in fp32, |T| < 2^24).
//
// K ordering inside each chunk of one 32-bit word of packed codes (16 two-bit
// or 8 four-bit codes): the expansion produces byte p = 4q + t from code
// (cpw/4) t + q, cpw = codes per word (a transpose).  The prepared filter rows
// use the same order, so the dot product over K is unchanged.  For 2-bit
// codes the odd registers q of a word hold 4c (a mask without a shift), and
// the filter bytes at those K positions are +-0.25: the product is c * 2^-9.
//
// Data path.  The expanded A operand never touches shared memory: gather
// threads load packed codes from global memory into registers several K
// stages ahead, expand them in registers and write them to tensor memory
// (tcgen05.st), and tcgen05.mma reads A from tensor memory.  Lane m of tensor
// memory holds output pixel m; 32-bit column c of an A stage holds K bytes
// 4c..4c+3.  Shared memory only carries the filter tiles (B), loaded by TMA in
// the 128B-swizzled K-major layout.
//
// Persistent, warp-specialized CTA (one per SM), tiles of 128 output pixels x
// BN output channels (BN <= 128) handed out round-robin; 27 warps:
//   warps 0-15   gather, in 4 groups of 4 warps; group g fills the K stages
//                g, g+4, g+8, ... so four stages are filled concurrently; warp
//                w writes rows 32*(w%4)..+31 (the tensor-memory lanes it may
//                access), all 128 K positions of the stage;
//   warp 16      TMA producer of the prepared filter tile;
//   warps 17, 26 TMEM allocation (17) and the tcgen05.mma issue, alternate pairs of K
//                stages each (one elected lane per warp);
//   warps 18-25  epilogue: tcgen05.ld of the finished accumulator (two
//                buffers, so it overlaps the next tile's mainloop), thresholds,
//                k-bit packing, stores.
// Tensor memory (512 columns): accumulators in [0, 2*BN), A stages in
// [256, 256 + 32*STAGES).  The K-stage pipeline runs continuously across tiles.
#pragma once
#include "conv_common.cuh"

namespace ifq {

// A second MMA-issuing warp after the epilogue warps (27 warps in all).
constexpr int kWarpMma2 = kWarpEpi0 + kEpiWarps;
constexpr int kConvThreads = kTcThreads + 32;

// The code of one accumulator against 15 ascending thresholds t[0..14] (+inf past 2^k - 1):
// #{ i : sign*D > t[i] } as a 4-ary search over five float4 per column,
//   t5[0] = {t3, t7, t11, sign},  t5[1+q] = {t(4q), t(4q+1), t(4q+2), -}  (q = 0..3):
// q = #{ t3, t7, t11 below sign*D } picks the group of four codes, and the group's three
// thresholds give the code 4q + #{ t(4q+j) below }.  Two dependent loads, the first one the same
// for every row of the column.
__device__ __forceinline__ uint32_t code15(float d, const float4* t5) {
  const float4 h = t5[0];
  const float sv = d * h.w;
  const uint32_t q = (uint32_t)(sv > h.x) + (uint32_t)(sv > h.y) + (uint32_t)(sv > h.z);
  const float4 g = t5[1 + q];
  return 4u * q + (uint32_t)(sv > g.x) + (uint32_t)(sv > g.y) + (uint32_t)(sv > g.z);
}

// The 2-bit code of one accumulator D = A / 512 against its column's thresholds
// t = (-T1, -T2, -T3, 512 s), as a float 0..3, on the FMA pipe: s A - T_i = fma(D, 512 s, -T_i) is
// an exact integer (|s A - T_i| < 2^24), and saturating it to [0, 1] gives exactly [s A > T_i]
// (sat_fma, conv_common.cuh).
__device__ __forceinline__ float code3f(float d, const float4& t) {
  return sat_fma(d, t.w, t.x) + sat_fma(d, t.w, t.y) + sat_fma(d, t.w, t.z);
}
// 32 lanes x 32 consecutive columns of tensor memory -> 32 registers, the wait in the same asm
// statement.
__device__ __forceinline__ void tc_ld32_sync(uint32_t t0, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
      "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
        "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(t0)
      : "memory");
}

// Codes are packed by accumulating code * 4^j into a float that starts at 2^23: its low mantissa
// bits are then the packed field (exact while the sum stays below 2^23, i.e. up to 8 codes).
constexpr float kPackBase = 8388608.0f;

// GB: bytes per gathered granule: 16, 8, 4 or 1 (the largest that divides the packed bytes of a
// pixel); SB: bits per stored input code (2 for k = 2, 4 for k = 3 and 4 and for the two nibbles of
// an 8-bit input value); SBO: bits per stored output code (2 or 4).
//
// KS > 1: split K.  The grid is made of clusters of KS CTAs; cluster c takes tiles c, c + C, ...
// (C clusters) and CTA r of it the K stages [r nk / KS, (r+1) nk / KS) of each, into its own
// accumulator.  Column block r of the tile (BN / KS columns) belongs to CTA r: in the epilogue every
// CTA sends the other blocks of its partial sum to their owners' receive slots (distributed shared
// memory), waits for the partners' partials of its own block, adds them and thresholds that block.
// The partial sums are exact integers (multiples of 2^-9 far inside the fp32 significand), so their
// order does not matter.  A receive slot is reused for the next tile once its owner has read it
// (send_ok); clusters synchronise once after setup and once before exit, so no CTA's shared memory
// goes away while a partner may still write it.
//
// BX = 1: the filter tile (B) is not loaded by TMA as e4m3 bytes but expanded in shared memory from
// the filters' sign bits (1 bit per weight instead of 8) by the gather group that fills the same K
// stage, into the 128B-swizzled layout TMA would have written.  For layers whose filters are read
// from DRAM about once (few row tiles, e.g. fully connected layers) that cuts the filter stream
// eightfold.  K positions past the filter read -1 from the bits, which is harmless: the gathered
// codes are zero there.
template <int BN, int GB, int SB, int SBO, int KS = 1, int BX = 0>
__global__ void __launch_bounds__(kConvThreads, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap tmap_w, const ConvArgs args) {
  static_assert(2 * BN <= kTmemA && kTmemA + 32 * kStages <= 512, "tensor memory budget");
  static_assert((SB == 2 || SB == 4) && (SBO == 2 || SBO == 4), "stored code width");
  static_assert(KS == 1 || KS == 2 || KS == 4, "K split");
  static_assert(BN / KS / 2 >= 16, "an epilogue thread takes at least 16 columns of a block");
  using L = TcSmem<BN, SBO, KS, BX>;
  constexpr int kU = kBK * SB / 8 / 16;       // 16-byte units of packed codes per K stage
  constexpr int kCpb = 8 / SB;                // codes per byte
  constexpr int kS = kStages;
  extern __shared__ uint8_t smem_raw_[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw_ + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sB = sbase + L::offB;
  float4* sThr = (float4*)(smem + L::offThr);      // SBO = 2: one float4 per column, SBO = 4: five
  int2* sTab = (int2*)(smem + L::offTab);
  const uint32_t barBase = sbase + L::offBar;
  // full[s]: the arrivals of the 4 warps of the gather group that owns stage s, plus
  // the TMA producer's (with the B bytes)
  auto full = [&](int s) { return barBase + 8u * s; };
  auto empty = [&](int s) { return barBase + 8u * (kS + s); };
  auto acc_full = [&](int b) { return barBase + 8u * (2 * kS + b); };
  auto acc_empty = [&](int b) { return barBase + 8u * (2 * kS + 2 + b); };
  const uint32_t done_bar = barBase + 8u * (2 * kS + 4);
  // KS > 1: recv_full completes when every partner has stored its partial of this CTA's column
  // block; send_ok when every partner has read the partial this CTA stored in its slot
  const uint32_t recv_full = barBase + 8u * (2 * kS + 5);
  const uint32_t send_ok = barBase + 8u * (2 * kS + 6);
  // BX: bits_full[i] completes when slot i of the sign-bit ring has landed; bits_empty[i] when the
  // gather group that read it is done with it
  constexpr int kBitBar0 = 2 * kS + 5 + (KS > 1 ? 2 : 0);
  auto bits_full = [&](int i) { return barBase + 8u * (kBitBar0 + i); };
  auto bits_empty = [&](int i) { return barBase + 8u * (kBitBar0 + L::kBitStages + i); };
  const uint32_t sBits = sbase + L::offBits;
  uint32_t* tmem_slot = (uint32_t*)(smem + L::offTmem);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr uint32_t kCols = 512;
  // tile schedule: cluster cid of G takes tiles cid, cid + G, ... (a cluster is one CTA for KS = 1)
  const uint32_t crank = KS > 1 ? cluster_ctarank() : 0u;
  const int cid = KS > 1 ? (int)cluster_id_x() : (int)blockIdx.x;
  const int G = KS > 1 ? (int)nclusters_x() : (int)gridDim.x;
  const int n_local = (args.ntiles - cid + G - 1) / G;
  // this CTA's K stages of every tile: [kb, kb + nk)
  const int kb = (int)((crank * (uint32_t)args.nk) / KS);
  const int nk = (int)(((crank + 1u) * (uint32_t)args.nk) / KS) - kb;

  // ---- setup (reads no global memory, so it may overlap the previous grid)
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(tmem_slot), kCols);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int s = 0; s < kS; ++s) {
      mbar_init(full(s), BX ? 4 : 4 + 1);   // one gather group (4 warps) [+ the TMA producer]
      mbar_init(empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 2);           // one commit from each MMA warp
      mbar_init(acc_empty(b), kEpiWarps);  // drained and zeroed by every epilogue warp
    }
    mbar_init(done_bar, 2);
    for (int i = 0; i < L::kBitStages; ++i) {
      mbar_init(bits_full(i), 1);
      mbar_init(bits_empty(i), 4);   // the 4 warps of the gather group that expands the stage
    }
    if constexpr (KS > 1) {
      mbar_init(recv_full, (KS - 1) * kEpiWarps * 32);   // every epilogue thread of every partner
      mbar_init(send_ok, (KS - 1) * kEpiWarps * 32);
    }
    fence_mbar_init();
  }
  if (warp == kWarpTma && lane == 0) prefetch_tmap(&tmap_w);
  // K-granule table: byte offset of each granule from the row's tap-(0,0)
  // pointer, and its tap as tap_mask(dy, dx); kTapNone past K.
  {
    const int cinb = args.cinb;
    for (int gk = tid; gk < args.ntab; gk += kConvThreads) {
      const int k0 = gk * kCpb * GB;
      const int tap = k0 / args.cin, cc = k0 - tap * args.cin;
      int2 e = make_int2(0, kTapNone);
      if (tap < args.kh * args.kw) {
        const int dy = tap / args.kw, dx = tap - dy * args.kw;
        e = make_int2((dy * args.w + dx) * cinb + cc / kCpb, tap_mask(dy, dx));
      }
      sTab[gk] = e;
    }
  }
  tc_fence_before();
  __syncthreads();
  // the partners' barriers are initialised before any CTA of the cluster reaches them
  if constexpr (KS > 1) cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_launch();
  // Each role waits for the kernels before this one (griddepcontrol.wait) where it first needs
  // them.  The gather warps read the previous layer's codes and always wait.  With args.early the
  // TMA warp (filters) and the epilogue warps (thresholds) start at once: the epilogue's stores
  // come after accumulators that the gathered codes fed, so after the gather's wait too.  The MMA
  // warps touch no global memory and never wait.

  if (warp < kGatherWarps) {
    grid_dep_wait();
    // =================== gather: packed codes -> registers -> tensor memory ===================
    const int group = warp >> 2, quarter = warp & 3;
    const int r = quarter * 32 + lane;                       // A row = tensor-memory lane
    const uint32_t tA = tmem + (uint32_t)kTmemA + ((uint32_t)(quarter * 32) << 16);
    const int total = n_local * nk;
    const int own = total > group ? (total - group + kGatherGroups - 1) / kGatherGroups : 0;   // stages of this group
    // load cursor over this group's stages it = group + 4*j: tile l_tile, K stage l_k
    int l_tile = 0, l_k = group;
    while (l_k >= nk) { l_k -= nk; ++l_tile; }
    RowGeom g = row_geom(args, l_tile < n_local ? (int)fdiv((uint32_t)(cid + l_tile * G), args.div_nt) * kBM + r
                                                : args.M);
    // packed codes of kAh of this group's stages in registers (16 registers either way)
    // (1-byte granules, 16 loads a unit: one stage ahead, within the register cap)
    constexpr int kAh = SB == 2 && GB > 1 ? kAhead : 1;
    // BX: this thread's share of a stage's filter tile: row bx_r of the channel tile, 16-bit chunks
    // bx_c0 .. bx_c0 + BN / 16 - 1 of the stage's 128 sign bits
    constexpr int kCpt = BN / 16;
    const int bx_gi = quarter * 32 + lane;
    const int bx_r = bx_gi / (8 / kCpt), bx_c0 = (bx_gi % (8 / kCpt)) * kCpt;
    auto next_load = [&](uint4 (&u)[kU]) {
#pragma unroll
      for (int q = 0; q < kU; ++q) u[q] = load_unit<GB>(sTab, g, (kb + l_k) * kU + q);
      l_k += kGatherGroups;
      if (l_k >= nk) {
        do { l_k -= nk; ++l_tile; } while (l_k >= nk);
        if (l_tile < n_local) g = row_geom(args, (int)fdiv((uint32_t)(cid + l_tile * G), args.div_nt) * kBM + r);
      }
    };
    uint4 ring[kAh][kU];
#pragma unroll
    for (int d = 0; d < kAh; ++d) {
#pragma unroll
      for (int q = 0; q < kU; ++q) ring[d][q] = make_uint4(0u, 0u, 0u, 0u);
      if (d < own) next_load(ring[d]);
    }
    bool ok = true;
#pragma unroll 1
    for (int base = 0; base < own && ok; base += kAh) {
#pragma unroll
      for (int d = 0; d < kAh; ++d) {
        const int j = base + d;
        if (j < own) {
          uint4 cur[kU];
#pragma unroll
          for (int q = 0; q < kU; ++q) cur[q] = ring[d][q];
          if (j + kAh < own) next_load(ring[d]);
          const int it = group + kGatherGroups * j;
          const int s = it % kS;
          const uint32_t ph = (uint32_t)(it / kS) & 1u;
          if (!__all_sync(0xffffffffu, mbar_wait_backoff(empty(s), ph ^ 1u, 64))) { ok = false; break; }
          tc_fence_after();
          if constexpr (SB == 2) {
            // 8 columns (two packed words) at a time: fewer live registers than 16
#pragma unroll
            for (int hq = 0; hq < 4; ++hq) {
              const uint4 u = cur[hq >> 1];
              uint32_t o8[8];
              expand2w((hq & 1) ? u.z : u.x, o8);
              expand2w((hq & 1) ? u.w : u.y, o8 + 4);
              tmem_st8_sync(tA + (uint32_t)(s * 32 + 8 * hq), o8);
            }
          } else {
            uint32_t o[16];
            expand4(cur[0], cur[1], o);
            tmem_st16_sync(tA + (uint32_t)(s * 32), o);
            expand4(cur[kU - 2], cur[kU - 1], o);
            tmem_st16_sync(tA + (uint32_t)(s * 32 + 16), o);
          }
          if constexpr (BX != 0) {
            // this K stage's filter tile from sign bits (loaded with the codes, kAh stages ahead):
            // 16-bit chunks -> 16 e4m3 bytes (+1 = 0x38, -1 = 0xB8) at row bx_r, chunk c of the
            // 128B-swizzled slot (chunk c of row r at c ^ (r % 8))
            const int rr = bx_r, c0 = bx_c0;
            const int bs = it % L::kBitStages;
            if (!__all_sync(0xffffffffu, mbar_wait(bits_full(bs), (uint32_t)(it / L::kBitStages) & 1u))) {
              ok = false;
              break;
            }
            uint32_t bw[(kCpt + 1) / 2];
#pragma unroll
            for (int q2 = 0; q2 < (kCpt + 1) / 2; ++q2) {
              uint32_t v;
              asm volatile("ld.shared.b32 %0, [%1];"
                           : "=r"(v)
                           : "r"(sBits + (uint32_t)(bs * L::kBitSlot + rr * 16 + c0 * 2 + 4 * q2)));
              bw[q2] = v;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bits_empty(bs));
            const uint32_t rowb = sB + (uint32_t)(s * L::kB) + (uint32_t)rr * 128u;
#pragma unroll
            for (int cc = 0; cc < kCpt; ++cc) {
              const uint32_t bits16 = (bw[cc >> 1] >> (16 * (cc & 1))) & 0xFFFFu;
              uint32_t w4[4];
#pragma unroll
              for (int nb = 0; nb < 4; ++nb) {
                // word nb of the chunk: +-1 (0x38 / 0xB8), or +-0.25 (0x28 / 0xA8) for the odd
                // words, whose gathered codes are 4c (expand2)
                const uint32_t x = (((bits16 >> (4 * nb)) & 0xFu) * 0x00204081u) & 0x01010101u;
                w4[nb] = ((nb & 1) ? 0xA8A8A8A8u : 0xB8B8B8B8u) - (x << 7);
              }
              const uint32_t dst = rowb + (uint32_t)((((c0 + cc) ^ (rr & 7)) & 7) << 4);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(w4[0]), "r"(w4[1]), "r"(w4[2]),
                           "r"(w4[3])
                           : "memory");
            }
            fence_proxy_async_smem();
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(full(s));
        }
      }
    }
  } else if (warp == kWarpTma) {
    if constexpr (BX != 0) {
      // =================== TMA producer (filter sign bits, kBitStages stages ahead) ===================
      // tmap_w maps the sign bits: [cout][Kpad / 8] bytes, boxes of BN rows x 16 bytes
      if (!args.early) grid_dep_wait();
      int it = 0;
      bool ok = true;
#pragma unroll 1
      for (int jt = 0; jt < n_local && ok; ++jt) {
        const int t = cid + jt * G;
        const int n0 = (t - (int)fdiv((uint32_t)t, args.div_nt) * args.nt) * BN;
#pragma unroll 1
        for (int k = 0; k < nk; ++k, ++it) {
          const int bs = it % L::kBitStages;
          const uint32_t ph = (uint32_t)(it / L::kBitStages) & 1u;
          if (!__all_sync(0xffffffffu, mbar_wait_backoff(bits_empty(bs), ph ^ 1u, 64))) { ok = false; break; }
          if (elect_one()) {
            mbar_arrive_expect_tx(bits_full(bs), (uint32_t)L::kBitSlot);
            tma_load_2d(sBits + (uint32_t)(bs * L::kBitSlot), &tmap_w, bits_full(bs), (kb + k) * (kBK / 8), n0);
          }
          __syncwarp();
        }
      }
      // drain: every bits load issued has landed before the CTA may exit
      if (!ok) {
        for (int i = it - L::kBitStages < 0 ? 0 : it - L::kBitStages; i < it; ++i)
          mbar_wait(bits_full(i % L::kBitStages), (uint32_t)(i / L::kBitStages) & 1u);
      }
      __syncwarp();
    }
    if constexpr (BX == 0) {
    if (!args.early) grid_dep_wait();
    // =================== TMA producer (filters) ===================
    // the whole warp runs the loop; one elected lane issues
    int it = 0;
    bool ok = true;
#pragma unroll 1
    for (int jt = 0; jt < n_local && ok; ++jt) {
      const int t = cid + jt * G;
      const int n0 = (t - (int)fdiv((uint32_t)t, args.div_nt) * args.nt) * BN;
#pragma unroll 1
      for (int k = 0; k < nk; ++k, ++it) {
        const int s = it % kS;
        const uint32_t ph = (uint32_t)(it / kS) & 1u;
        if (!__all_sync(0xffffffffu, mbar_wait_backoff(empty(s), ph ^ 1u, 64))) { ok = false; break; }
        if (elect_one()) {
          mbar_arrive_expect_tx(full(s), (uint32_t)L::kB);
          tma_load_2d(sB + (uint32_t)(s * L::kB), &tmap_w, full(s), (kb + k) * kBK, n0);
        }
        __syncwarp();
      }
    }
    // drain: every load issued into a slot has landed before the CTA may exit
    // (full(s) completes only when the gather warps and the bytes have arrived)
    if (!ok) {
      for (int i = it - kS < 0 ? 0 : it - kS; i < it; ++i)
        mbar_wait(full(i % kS), (uint32_t)(i / kS) & 1u);
    }
    __syncwarp();
    }
  } else if (warp == kWarpMma || warp == kWarpMma2) {
    // =================== MMA issue ===================
    // Two MMA warps take alternate pairs of K stages of every tile into the same accumulator:
    // one thread issuing tcgen05.mma costs more per instruction than an N <= 128 MMA takes on
    // the tensor pipe.  Every MMA accumulates into a buffer that
    // the epilogue left zeroed, so the order of the two warps' MMAs does not matter (the fp32
    // sums are exact integers in any order).  Each warp runs its loop uniformly; one elected
    // lane issues and commits.
    const int mi = warp == kWarpMma2 ? 1 : 0;
    constexpr uint32_t idesc = idesc_e4m3_f32(kBM, BN);
    int gp = 0;   // pairs of K stages seen so far (pairs alternate between the two warps)
    bool ok = true;
#pragma unroll 1
    for (int jt = 0; jt < n_local && ok; ++jt) {
      const int ab = jt & 1;
      // buffer ab is zero once the epilogue has drained it (phase 0: the zeroing at start)
      if (!__all_sync(0xffffffffu, mbar_wait(acc_empty(ab), (uint32_t)(jt >> 1) & 1u))) break;
      tc_fence_after();
      const uint32_t dacc = tmem + (uint32_t)(ab * BN);
      // stages k, k+1 of this tile (one vote, fence and elect for up to 8 MMAs)
#pragma unroll 1
      for (int k = 0; k < nk; k += 2, ++gp) {
        if ((gp & 1) != mi) continue;
        const bool two = k + 1 < nk;
        const int it = jt * nk + k;   // position in the CTA's stage sequence
        const int s0 = it % kS, s1 = (it + 1) % kS;
        const uint32_t ph0 = (uint32_t)(it / kS) & 1u, ph1 = (uint32_t)((it + 1) / kS) & 1u;
        bool got = mbar_wait(full(s0), ph0);
        if (two) got = got && mbar_wait(full(s1), ph1);
        if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
        tc_fence_after();
        if (elect_one()) {
          const uint32_t a0 = tmem + (uint32_t)(kTmemA + s0 * 32), b0 = sB + (uint32_t)(s0 * L::kB);
#pragma unroll
          for (int kk = 0; kk < kBK / 32; ++kk)
            mma_e4m3_tmem_a(dacc, a0 + (uint32_t)(8 * kk), sdesc_sw128(b0 + 32 * kk), idesc, 1u);
          mma_commit(empty(s0));
          if (two) {
            const uint32_t a1 = tmem + (uint32_t)(kTmemA + s1 * 32), b1 = sB + (uint32_t)(s1 * L::kB);
#pragma unroll
            for (int kk = 0; kk < kBK / 32; ++kk)
              mma_e4m3_tmem_a(dacc, a1 + (uint32_t)(8 * kk), sdesc_sw128(b1 + 32 * kk), idesc, 1u);
            mma_commit(empty(s1));
          }
        }
        __syncwarp();
      }
      if (ok && elect_one()) mma_commit(acc_full(ab));
      __syncwarp();
    }
    if (elect_one()) mma_commit(done_bar);   // fires once every MMA this warp issued has completed
    __syncwarp();
  } else {
    // =================== epilogue ===================
    if (!args.early) grid_dep_wait();
    // warp pair e, e+4 covers lane quarter (warp % 4), halves 0 and 1 of every column block (the
    // whole tile for KS = 1; with KS > 1 the block of CTA r is columns [r BN/KS, (r+1) BN/KS))
    constexpr int CB = BN / KS;                 // columns of a block
    constexpr int CW = CB / 2;                  // columns per thread in a block
    const int e = warp - kWarpEpi0;             // 0..7
    const int et = tid - kWarpEpi0 * 32;        // 0..255
    const int quarter = warp & 3;
    const int c_in = (e >> 2) * CW;             // this thread's first column within a block
    const int c_lo = (int)crank * CB + c_in;    // ... within this CTA's own block
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    bool ok = true;   // after a timed-out wait, keep only the named barriers (uniform over the 8 warps)
    // both accumulator buffers start at zero: every MMA accumulates
    {
#pragma unroll
      for (int b2 = 0; b2 < 2; ++b2)
#pragma unroll
        for (int p = 0; p < KS; ++p)
#pragma unroll
          for (int c0 = 0; c0 < CW; c0 += 16) tmem_zero16_sync(tmem + lane_off + (uint32_t)(b2 * BN + p * CB + c_in + c0));
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(acc_empty(0));
        mbar_arrive(acc_empty(1));
      }
    }
#pragma unroll 1
    for (int jt = 0; jt < n_local; ++jt) {
      const int t = cid + jt * G;
      const int mt = (int)fdiv((uint32_t)t, args.div_nt);
      const int n0 = (t - mt * args.nt) * BN;
      const int m = mt * kBM + row;
      const int tb = args.nt > 1 ? (jt & 1) : 0;
      if (jt == 0 || args.nt > 1) {
        for (int c = et; c < BN; c += 256) {
          const int nn = n0 + c;
          const bool has = nn < args.cout && args.thr;
          if constexpr (SBO == 2) {
            // (-T1, -T2, -T3, 512 s): code3f evaluates [s A > T_i] as sat(D * 512 s - T_i)
            float4 v = make_float4(0.f, 0.f, 0.f, 512.f);
            if (has)
              v = make_float4(-(float)args.thr[3 * nn], -(float)args.thr[3 * nn + 1], -(float)args.thr[3 * nn + 2],
                              512.f * (float)args.sign[nn]);
            sThr[tb * BN + c] = v;
          } else {
            // sign*A > T  <=>  sign*D > T/512 with D = A/512 (exact in fp32)
            float4* t5 = sThr + (size_t)(tb * BN + c) * 5;
            auto T = [&](int i) {
              return has && i < args.lvl ? (float)args.thr[(size_t)args.lvl * nn + i] * (1.0f / 512.0f) : INFINITY;
            };
            t5[0] = make_float4(T(3), T(7), T(11), has ? (float)args.sign[nn] : 1.0f);
#pragma unroll
            for (int q = 0; q < 4; ++q) t5[1 + q] = make_float4(T(4 * q), T(4 * q + 1), T(4 * q + 2), 0.0f);
          }
        }
        named_bar(1, kEpiWarps * 32);
      }
      const int ab = jt & 1;
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait_backoff(acc_full(ab), (uint32_t)(jt >> 1) & 1u, 64));
      if (!ok) continue;
      tc_fence_after();
      const uint32_t tbuf = tmem + (uint32_t)(ab * BN) + lane_off;   // this row of accumulator buffer ab
      const uint32_t tacc = tbuf + (uint32_t)c_lo;
      if constexpr (KS > 1) {
        // send the partners' blocks of this partial sum to their receive slots (slot s of CTA p
        // holds the partial of the s-th other CTA in rank order), once p has read the last tile's
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait_cluster(send_ok, ((uint32_t)jt & 1u) ^ 1u));
        if (ok) {
#pragma unroll 1
          for (int pp = 1; pp < KS; ++pp) {
            const uint32_t p = (crank + (uint32_t)pp) % KS;
            const uint32_t slot = crank < p ? crank : crank - 1u;
            const uint32_t dst = mapa_shared(
                sbase + (uint32_t)L::offRecv + slot * (uint32_t)L::kRecvSlot + (uint32_t)(row * L::kRecvRow + c_in) * 4u, p);
#pragma unroll
            for (int c0 = 0; c0 < CW; c0 += 16) {
              uint32_t v[16];
              tmem_ld16_sync(tbuf + (uint32_t)(p * CB + c_in + c0), v);
#pragma unroll
              for (int q = 0; q < 4; ++q)
                st_cluster_v4(dst + (uint32_t)(c0 + 4 * q) * 4u, v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            }
          }
#pragma unroll 1
          for (int pp = 1; pp < KS; ++pp) mbar_arrive_remote(mapa_shared(recv_full, (crank + (uint32_t)pp) % KS));
          ok = __all_sync(0xffffffffu, mbar_wait_cluster(recv_full, (uint32_t)jt & 1u));
        }
        if (!ok) continue;
      }
      const float4* th = sThr + (size_t)(tb * BN + c_lo) * (SBO == 2 ? 1 : 5);
      constexpr int kPW = CW * SBO / 32;          // 32-bit words of packed codes per thread
      uint32_t packed[kPW];
      // Plain 2-bit codes (no pool, no accumulators out, no K split): 32 columns per tensor-memory
      // load and wait, twice the independent work between waits (the 1x1 512 -> 512 layer 107.3 ->
      // 97.6 us).  Instances with 8- and 1-byte granules keep 16 columns: their gather leaves no
      // registers for it.
      constexpr bool kWide32 = (GB == 16 || GB == 4) && SB == 2 && SBO == 2 && KS == 1 && CW % 32 == 0;
      const bool wide32 = kWide32 && args.lpool == 0 && !args.y_acc;
      if constexpr (kWide32) {
        if (wide32) {
#pragma unroll
          for (int c0 = 0; c0 < CW; c0 += 32) {
            uint32_t v[32];
            tc_ld32_sync(tacc + c0, v);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              float lo = kPackBase, hi = kPackBase;
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                lo = fmaf(code3f(__uint_as_float(v[16 * h + j]), th[c0 + 16 * h + j]), (float)(1 << (2 * j)), lo);
                hi = fmaf(code3f(__uint_as_float(v[16 * h + j + 8]), th[c0 + 16 * h + j + 8]), (float)(1 << (2 * j)), hi);
              }
              packed[c0 / 16 + h] = __byte_perm(__float_as_uint(lo), __float_as_uint(hi), 0x5410);
              // the second half's thresholds are not loaded before the first half is done (registers)
              asm volatile("" ::: "memory");
            }
          }
        }
      }
#pragma unroll
      for (int c0 = 0; c0 < CW && !wide32; c0 += 16) {
        uint32_t v[16];
        tmem_ld16_sync(tacc + c0, v);
        if constexpr (KS > 1) {   // + the partners' partial sums of these 16 columns
#pragma unroll
          for (int sl = 0; sl < KS - 1; ++sl) {
            const float4* src =
                (const float4*)(smem + L::offRecv + (size_t)sl * L::kRecvSlot) + (row * L::kRecvRow + c_in + c0) / 4;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float4 f = src[q];
              v[4 * q] = __float_as_uint(__uint_as_float(v[4 * q]) + f.x);
              v[4 * q + 1] = __float_as_uint(__uint_as_float(v[4 * q + 1]) + f.y);
              v[4 * q + 2] = __float_as_uint(__uint_as_float(v[4 * q + 2]) + f.z);
              v[4 * q + 3] = __float_as_uint(__uint_as_float(v[4 * q + 3]) + f.w);
            }
          }
        }
        // Fused pool (Sec. 2.1: the pool acts on Y^conv, before BN and the quantizer): the window
        // maximum of A over the window's consecutive lanes, then the thresholds.
        if (args.lpool == 1) {
          // 2x2: a reduce-scatter over the window's 4 lanes (columns 8 apart with lane ^ 2, then
          // 4 apart with lane ^ 1) leaves this lane the maxima of 4 of the 16 columns,
          // [sub, sub + 4); it thresholds those alone and stores their byte of codes
          const bool h2 = (lane & 2) != 0, h1 = (lane & 1) != 0;
          float a8[8], a4[4];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float lo8 = __uint_as_float(v[j]), hi8 = __uint_as_float(v[j + 8]);
            a8[j] = fmaxf(h2 ? hi8 : lo8, __shfl_xor_sync(0xffffffffu, h2 ? lo8 : hi8, 2));
          }
#pragma unroll
          for (int j = 0; j < 4; ++j)
            a4[j] = fmaxf(h1 ? a8[j + 4] : a8[j], __shfl_xor_sync(0xffffffffu, h1 ? a8[j] : a8[j + 4], 1));
          const int sub = (h2 ? 8 : 0) + (h1 ? 4 : 0);
          uint32_t bits = 0;
          if constexpr (SBO == 2) {
            float pk = kPackBase;
#pragma unroll
            for (int j = 0; j < 4; ++j) pk = fmaf(code3f(a4[j], th[c0 + sub + j]), (float)(1 << (2 * j)), pk);
            bits = __float_as_uint(pk) & 0xFFu;
          } else {
#pragma unroll
            for (int j = 0; j < 4; ++j) bits |= code15(a4[j], th + (c0 + sub + j) * 5) << (4 * j);
          }
          const int cabs = n0 + c_lo + c0 + sub;
          if (args.y_codes && m < args.M && cabs < args.cout) {
            uint8_t* dst = args.y_codes + (size_t)(m >> 2) * ((args.cout * SBO) >> 3) + ((cabs * SBO) >> 3);
            if constexpr (SBO == 2) *dst = (uint8_t)bits;
            else *(uint16_t*)dst = (uint16_t)bits;   // cabs % 4 == 0: an even byte offset
          }
          continue;
        }
        if (args.lpool) {   // 4x4: every lane of the window gets the maxima of all 16 columns
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            float x = __uint_as_float(v[j]);
            for (int off = 1; off < (1 << (2 * args.lpool)); off <<= 1)
              x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, off));
            v[j] = __float_as_uint(x);
          }
        }
        if constexpr (SBO == 2) {
          float lo = kPackBase, hi = kPackBase;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            lo = fmaf(code3f(__uint_as_float(v[j]), th[c0 + j]), (float)(1 << (2 * j)), lo);
            hi = fmaf(code3f(__uint_as_float(v[j + 8]), th[c0 + j + 8]), (float)(1 << (2 * j)), hi);
          }
          packed[c0 / 16] = __byte_perm(__float_as_uint(lo), __float_as_uint(hi), 0x5410);
        } else {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t wd = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) wd |= code15(__uint_as_float(v[8 * h + j]), th + (c0 + 8 * h + j) * 5) << (4 * j);
            packed[c0 / 8 + h] = wd;
          }
        }
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
      // the partners may store the next tile's partials into this CTA's slots
      if constexpr (KS > 1) {
#pragma unroll 1
        for (int pp = 1; pp < KS; ++pp) mbar_arrive_remote(mapa_shared(send_ok, (crank + (uint32_t)pp) % KS));
      }
      // the accumulator buffer may be refilled once every epilogue warp has read and zeroed it
#pragma unroll
      for (int p = 0; p < KS; ++p)
#pragma unroll
        for (int c0 = 0; c0 < CW; c0 += 16) tmem_zero16_sync(tbuf + (uint32_t)(p * CB + c_in + c0));
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty(ab));
      // (2x2 pools stored their codes above; with a 4x4 pool the first lane of each window stores
      // the pooled pixel m >> 4)
      const bool store = args.y_codes && m < args.M && args.lpool != 1 && (m & ((1 << (2 * args.lpool)) - 1)) == 0;
      if (store) {
        const int rowb = (args.cout * SBO) >> 3;   // bytes per output pixel
        const int cb = n0 + c_lo;                 // first channel of this thread
        const int cbb = (cb * SBO) >> 3;           // its byte within the pixel
        uint8_t* dst = args.y_codes + (size_t)(m >> (2 * args.lpool)) * rowb + cbb;
        if (cb + CW <= args.cout && kPW >= 4 && (rowb & 15) == 0 && (cbb & 15) == 0) {
#pragma unroll
          for (int q = 0; q < kPW / 4; ++q)
            *(uint4*)(dst + 16 * q) =
                make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
        } else if (cb + CW <= args.cout && (rowb & 3) == 0 && (cbb & 3) == 0) {
#pragma unroll
          for (int q = 0; q < kPW; ++q) *(uint32_t*)(dst + 4 * q) = packed[q];
        } else {
          const int nbytes = (max(0, min(CW, args.cout - cb)) * SBO) >> 3;
#pragma unroll
          for (int q = 0; q < 4 * kPW; ++q)   // unrolled: packed[] stays in registers
            if (q < nbytes) dst[q] = (uint8_t)(packed[q >> 2] >> (8 * (q & 3)));
        }
      }
    }
  }

  // ---- teardown: every MMA has completed (done_bar) before TMEM is released
  tc_fence_before();
  __syncthreads();
  // no CTA leaves while a partner may still store into its receive slots or arrive on its barriers
  if constexpr (KS > 1) cluster_sync_all();
  if (warp == kWarpMma) {
    tc_fence_after();
    mbar_wait(done_bar, 0);
    tmem_dealloc(tmem, kCols);
  }
}

}  // namespace ifq
