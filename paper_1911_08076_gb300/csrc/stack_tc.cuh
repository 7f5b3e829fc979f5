// Persistent tensor-core kernel for a whole stack of quantized substructures
// (Sec. 3.1: the codes of one substructure are the input of the next).
//
// One cooperative launch, one CTA per SM, runs every conv layer of the stack
// in order; each CTA takes tiles blockIdx.x, blockIdx.x + G, ... of every
// layer.  The per-tile data path is the one of conv_tc.cuh (packed codes ->
// registers -> tensor memory, filters by TMA, elected-lane tcgen05.mma,
// double-buffered accumulators, threshold epilogue), and its pipeline (the K
// stage ring, the accumulator buffers) runs on across layer boundaries, so
// setup, tensor-memory allocation and pipeline fill are paid once per stack
// instead of once per layer.
//
// Layer dependencies, tile by tile.  Each layer has one completion counter per
// 128-row output block, complete when it equals the layer's number of
// output-channel tiles.  Every epilogue warp, once its part of a tile is
// stored, adds one to a CTA-local count in shared memory (release, CTA
// scope).  A publisher warp follows that count (acquire, CTA scope): when all
// epilogue warps have stored a tile, it issues one gpu-scope fence for every
// tile stored so far and then adds one to each such tile's block counter, so
// no epilogue warp ever stalls on a gpu-scope release.
// A dependency warp walks the CTA's tiles in order; for each it works out
// which 128-row blocks of the source layer the tile's receptive field can
// touch (every image row from the first to the last one any of its 128 output
// rows reads), waits (acquire, bounded in time) until each is complete, and
// then publishes the CTA-local tile index in shared memory (release, CTA
// scope).  The gather threads load a tile's codes only after observing that
// index (acquire).  The dependency warp is the only role that waits on other
// tiles, and it holds no pipeline resource while it waits: a gather warp may
// block on the next tile's index while still holding a loaded stage of the
// current tile, and the index must not depend on that stage being consumed
// (it only depends on tiles of earlier layers).  Codes are read with ordinary weak loads, never through the
// non-coherent read-only path.  A tile only waits on tiles of earlier layers,
// each CTA's pipeline consumes its tiles in order, and all CTAs are
// co-resident (cooperative launch), so the stack always completes; tiles of
// the next layer start as soon as their own inputs exist, so one layer's tail
// overlaps the next layer's head.
#pragma once
#include "conv_common.cuh"

namespace ifq {

constexpr int kMaxStackLayers = 24;
constexpr int kMaxStackTab = 2048;   // K-granule table entries of all layers together
constexpr int kStackBN = 128;        // largest output-channel tile (B slots are sized for it)
constexpr int kWarpDep = kWarpEpi0 + kEpiWarps;        // the dependency warp
constexpr int kWarpPub = kWarpDep + 1;                 // the publisher warp
constexpr int kStackThreads = kTcThreads + 64;

struct StackLayer {
  ConvArgs a;    // a.x: the stack input or the output codes of layer `dep`
  int bn;        // output-channel tile: 32, 64 or 128
  int gb;        // bytes per gathered granule: 16, 4 or 1
  int tab_off;   // first entry of this layer's K-granule table in shared memory
  int dep;       // layer of this launch whose codes are this layer's input, -1 for the stack input
  int cnt_off;   // first of this layer's per-128-row-block completion counters
};

struct StackParams {
  int nlayers;
  unsigned int* cnt;    // per-layer, per-128-row-block completion counters, zero at launch
  StackLayer L[kMaxStackLayers];
  CUtensorMap tm[kMaxStackLayers];
};

struct StackSmem {
  static constexpr int kB = kStackBN * kBK;            // one B slot
  static constexpr int offB = 0;
  static constexpr int offThr = offB + kStages * kB;   // 2 buffers of kStackBN float4
  static constexpr int offTab = offThr + 2 * kStackBN * 16;
  static constexpr int offLayers = offTab + kMaxStackTab * 8;   // the layer records, copied from the parameters
  static constexpr int offBar = offLayers + (int)((kMaxStackLayers * sizeof(StackLayer) + 15) / 16 * 16);
  static constexpr int nBar = 2 * kStages + 5;
  static constexpr int offTmem = offBar + nBar * 8;
  static constexpr int offReady = offTmem + 8;          // tiles whose inputs are complete (CTA-local count)
  static constexpr int offStored = offReady + 8;        // epilogue-warp tile stores done (CTA-local count)
  static constexpr int bytes = offStored + 8 + 1024;
};

static_assert(sizeof(StackLayer) % 8 == 0, "layer records are copied to shared memory in 4-byte words");
static_assert(StackSmem::bytes <= 227 * 1024, "shared memory budget");

__device__ __forceinline__ int stack_n_local(int ntiles, int c, int G) { return c < ntiles ? (ntiles - c + G - 1) / G : 0; }

// Wait until *p >= target, then order this thread's later loads after the
// writes that the counter publishes (acquire pattern: relaxed polls, one
// gpu-scope fence once the target is seen, so that polling does not keep
// invalidating the SM's L1); false after 2 s.
__device__ __forceinline__ bool wait_counter(const unsigned int* p, unsigned int target) {
  const unsigned long long t0 = global_ns();
  for (uint32_t it = 0; it < kWaitLimit; ++it) {
    unsigned int v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    if (v >= target) {
      asm volatile("fence.acq_rel.gpu;" ::: "memory");
      return true;
    }
    if ((it & 15u) == 15u && global_ns() - t0 > kWaitNs) break;
    __nanosleep(64);
  }
  set_status(IFQ_ETIMEOUT);
  return false;
}

__device__ __forceinline__ uint32_t ld_acquire_cta(uint32_t saddr) {
  uint32_t v;
  asm volatile("ld.acquire.cta.shared::cta.u32 %0, [%1];" : "=r"(v) : "r"(saddr) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_cta(uint32_t saddr, uint32_t v) {
  asm volatile("st.release.cta.shared::cta.u32 [%0], %1;" ::"r"(saddr), "r"(v) : "memory");
}
__device__ __forceinline__ void red_release_cta(uint32_t saddr, uint32_t v) {
  asm volatile("red.release.cta.shared::cta.add.u32 [%0], %1;" ::"r"(saddr), "r"(v) : "memory");
}

// Wait until a CTA-local count in shared memory reaches `target` (acquire, CTA scope);
// false after 2 s.
__device__ __forceinline__ bool wait_ready(uint32_t saddr, uint32_t target, uint32_t sleep_ns) {
  if (ld_acquire_cta(saddr) >= target) return true;
  const unsigned long long t0 = global_ns();
  for (uint32_t it = 0; it < kWaitLimit; ++it) {
    __nanosleep(sleep_ns);
    if (ld_acquire_cta(saddr) >= target) return true;
    if ((it & 15u) == 15u && global_ns() - t0 > kWaitNs) break;
  }
  set_status(IFQ_ETIMEOUT);
  return false;
}

// Warp-collective wait_ready: lane 0 alone polls (a whole warp polling would flood the
// shared-memory pipe that the working warps' loads use); __syncwarp then orders the other
// lanes' later loads after lane 0's acquire.
__device__ __forceinline__ bool warp_wait_ready(uint32_t saddr, uint32_t target, int lane) {
  bool ok = true;
  if (lane == 0) ok = wait_ready(saddr, target, 64);
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok;
}

// Warp-collective: wait until every 128-row block of layer S.dep that output
// block mt of S can read is complete.  Output rows m0..m1 cover images n0..n1;
// their receptive field lies within input image rows ih0 (of image n0) to ih1
// (of image n1), i.e. within flattened input pixels p0..p1, which are rows of
// the source layer's output.
__device__ __forceinline__ bool wait_deps(const StackLayer* sL, unsigned int* cnt, const StackLayer& S, int mt,
                                          int lane) {
  const ConvArgs& a = S.a;
  const StackLayer& D = sL[S.dep];
  const int m0 = mt * kBM, m1 = min(a.M, m0 + kBM) - 1;
  const int n0 = (int)fdiv((uint32_t)m0, a.div_hw), n1 = (int)fdiv((uint32_t)m1, a.div_hw);
  const int oh0 = (int)fdiv((uint32_t)(m0 - n0 * a.ho * a.wo), a.div_wo);
  const int oh1 = (int)fdiv((uint32_t)(m1 - n1 * a.ho * a.wo), a.div_wo);
  const int ih0 = min(max(oh0 * a.stride - a.pad, 0), a.h - 1);
  const int ih1 = min(max(oh1 * a.stride - a.pad + a.kh - 1, 0), a.h - 1);
  const long long p0 = ((long long)n0 * a.h + ih0) * a.w;
  const long long p1 = ((long long)n1 * a.h + ih1) * a.w + a.w - 1;
  const int b0 = (int)(p0 / kBM), b1 = (int)(p1 / kBM);
  const unsigned int target = (unsigned int)D.a.nt;
  bool ok = true;
  for (int b = b0 + lane; b <= b1 && ok; b += 32) ok = wait_counter(cnt + D.cnt_off + b, target);
  ok = __all_sync(0xffffffffu, ok);
  __syncwarp();   // orders every lane's acquire before lane 0's release of the ready count
  return ok;
}

// Own K stages of packed codes a gather thread of the stack kernel keeps in registers (one: the
// stack kernel's extra state leaves no room for a second at 72 registers).
constexpr int kStackAhead = 1;

// One gather group's share of one layer: its own K stages q = q0, q0+4, ... of
// the layer's local stage sequence (stage index it_base + q in the CTA ring).
template <int GB>
__device__ __forceinline__ bool stack_gather_layer(const ConvArgs& a, const int2* tab, int nl, int q0, int own,
                                                   int it_base, int gt_base, uint32_t sReady, uint32_t tA, int r,
                                                   int lane, uint32_t barBase) {
  const int nk = a.nk;
  const int G = gridDim.x;
  int l_tile = q0 / nk, l_k = q0 - (q0 / nk) * nk;
  int waited = -1;
  bool ok = true;
  RowGeom g = row_geom(a, (int)fdiv((uint32_t)((int)blockIdx.x + l_tile * G), a.div_nt) * kBM + r);
  auto next_load = [&](uint4& lo, uint4& hi) {
    if (l_tile != waited) {   // first codes of this tile: its inputs must be complete
      ok = warp_wait_ready(sReady, (uint32_t)(gt_base + l_tile + 1), lane) && ok;
      waited = l_tile;
    }
    lo = load_unit<GB, true>(tab, g, 2 * l_k);
    hi = load_unit<GB, true>(tab, g, 2 * l_k + 1);
    l_k += kGatherGroups;
    if (l_k >= nk) {
      do { l_k -= nk; ++l_tile; } while (l_k >= nk);
      if (l_tile < nl) g = row_geom(a, (int)fdiv((uint32_t)((int)blockIdx.x + l_tile * G), a.div_nt) * kBM + r);
    }
  };
  uint4 ring_lo[kStackAhead], ring_hi[kStackAhead];
#pragma unroll
  for (int d = 0; d < kStackAhead; ++d) {
    ring_lo[d] = ring_hi[d] = make_uint4(0u, 0u, 0u, 0u);
    if (d < own) next_load(ring_lo[d], ring_hi[d]);
  }
#pragma unroll 1
  for (int base = 0; base < own; base += kStackAhead) {
#pragma unroll
    for (int d = 0; d < kStackAhead; ++d) {
      const int j = base + d;
      if (j < own) {
        const uint4 lo = ring_lo[d], hi = ring_hi[d];
        if (j + kStackAhead < own) next_load(ring_lo[d], ring_hi[d]);
        const int it = it_base + q0 + kGatherGroups * j;
        const int s = it % kStages;
        const uint32_t ph = (uint32_t)(it / kStages) & 1u;
        if (!__all_sync(0xffffffffu, ok && mbar_wait_backoff(barBase + 8u * (kStages + s), ph ^ 1u, 64))) return false;   // empty(s)
        tc_fence_after();
        uint32_t o[16];
        expand2(lo, o);
        tmem_st16_sync(tA + (uint32_t)(s * 32), o);
        expand2(hi, o);
        tmem_st16_sync(tA + (uint32_t)(s * 32 + 16), o);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(barBase + 8u * s);   // full(s)
      }
    }
  }
  return true;
}

// One epilogue warp's part of a finished tile: CW accumulator columns of its 32
// rows from tensor memory (tacc), the three thresholds of Eq. (7) per column
// (th, already divided by 512 and with the sign-flip factor in .w), packed
// 2-bit codes and/or int32 accumulators to global memory.  Releases the
// accumulator buffer (acc_empty) as soon as the last column has been read.
template <int CW>
__device__ __forceinline__ void stack_epi_tile(const ConvArgs& a, uint32_t tacc, const float4* th, int m, int cb,
                                               uint32_t acc_empty, int lane) {
  uint32_t packed[CW / 16];
#pragma unroll
  for (int c0 = 0; c0 < CW; c0 += 16) {
    uint32_t v[16];
    tmem_ld16_sync(tacc + c0, v);
    // the code of D = A / 512 against th = (-T1, -T2, -T3, 512 s): [s A > T_i] = sat(D 512 s - T_i)
    // (exact integers, sat_fma), summed and packed by accumulating code * 4^j into a float based at
    // 2^23 (8 codes a float), on the FMA pipe
    float lo = 8388608.0f, hi = 8388608.0f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 ta = th[c0 + j], tb = th[c0 + j + 8];
      const float da = __uint_as_float(v[j]), db = __uint_as_float(v[j + 8]);
      lo = fmaf(sat_fma(da, ta.w, ta.x) + sat_fma(da, ta.w, ta.y) + sat_fma(da, ta.w, ta.z), (float)(1 << (2 * j)), lo);
      hi = fmaf(sat_fma(db, tb.w, tb.x) + sat_fma(db, tb.w, tb.y) + sat_fma(db, tb.w, tb.z), (float)(1 << (2 * j)), hi);
    }
    packed[c0 / 16] = __byte_perm(__float_as_uint(lo), __float_as_uint(hi), 0x5410);
    if (a.y_acc && m < a.M) {
      const int cbase = cb + c0;
      int32_t* dst = a.y_acc + (size_t)m * a.cout + cbase;
      if (cbase + 16 <= a.cout && (a.cout & 3) == 0) {
#pragma unroll
        for (int j = 0; j < 16; j += 4)
          *(int4*)(dst + j) = make_int4(__float2int_rn(__uint_as_float(v[j]) * 512.0f),
                                        __float2int_rn(__uint_as_float(v[j + 1]) * 512.0f),
                                        __float2int_rn(__uint_as_float(v[j + 2]) * 512.0f),
                                        __float2int_rn(__uint_as_float(v[j + 3]) * 512.0f));
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (cbase + j < a.cout) dst[j] = __float2int_rn(__uint_as_float(v[j]) * 512.0f);
      }
    }
  }
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(acc_empty);
  if (a.y_codes && m < a.M) {
    const int rowb = a.cout >> 2;
    uint8_t* dst = a.y_codes + (size_t)m * rowb + (cb >> 2);
    if (CW == 64 && cb + CW <= a.cout && (rowb & 15) == 0 && (cb & 63) == 0) {
      *(uint4*)dst = make_uint4(packed[0], packed[CW / 16 > 1 ? 1 : 0], packed[CW / 16 > 2 ? 2 : 0],
                                packed[CW / 16 > 3 ? 3 : 0]);
    } else if (cb + CW <= a.cout && (rowb & 3) == 0 && (cb & 15) == 0) {
#pragma unroll
      for (int q = 0; q < CW / 16; ++q) *(uint32_t*)(dst + 4 * q) = packed[q];
    } else {
      const int nbytes = max(0, min(CW, a.cout - cb)) >> 2;
      for (int q = 0; q < nbytes; ++q) dst[q] = (uint8_t)(packed[q >> 2] >> (8 * (q & 3)));
    }
  }
}

__global__ void __launch_bounds__(kStackThreads, 1) conv_stack_kernel(const __grid_constant__ StackParams P) {
  using L = StackSmem;
  extern __shared__ uint8_t smem_raw_[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw_ + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sB = sbase + L::offB;
  float4* sThr = (float4*)(smem + L::offThr);
  int2* sTab = (int2*)(smem + L::offTab);
  StackLayer* sL = (StackLayer*)(smem + L::offLayers);
  const uint32_t barBase = sbase + L::offBar;
  auto full = [&](int s) { return barBase + 8u * s; };
  auto empty = [&](int s) { return barBase + 8u * (kStages + s); };
  auto acc_full = [&](int b) { return barBase + 8u * (2 * kStages + b); };
  auto acc_empty = [&](int b) { return barBase + 8u * (2 * kStages + 2 + b); };
  const uint32_t done_bar = barBase + 8u * (2 * kStages + 4);
  uint32_t* tmem_slot = (uint32_t*)(smem + L::offTmem);
  const uint32_t sReady = sbase + L::offReady;
  const uint32_t sStored = sbase + L::offStored;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr uint32_t kCols = 512;
  const int G = gridDim.x;
  const int c = blockIdx.x;
  const int nlayers = P.nlayers;

  // ---- setup: tensor memory, barriers, every layer's K-granule table
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(tmem_slot), kCols);
    tmem_relinquish();
  }
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full(s), 4 + 1);   // one gather group (4 warps) + the TMA producer
      mbar_init(empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), kEpiWarps);
    }
    mbar_init(done_bar, 1);
    fence_mbar_init();
    *(volatile uint32_t*)(smem + L::offReady) = 0u;
    *(volatile uint32_t*)(smem + L::offStored) = 0u;
  }
  if (warp == kWarpTma)
    for (int l = lane; l < nlayers; l += 32) prefetch_tmap(&P.tm[l]);
  // every role reads its layer records from shared memory: indexing the parameter block with a
  // run-time layer index, from warps that are at different layers, thrashes the constant cache
  for (int i = tid; i < (int)(nlayers * sizeof(StackLayer) / 4); i += kStackThreads)
    ((uint32_t*)sL)[i] = ((const uint32_t*)P.L)[i];
  for (int l = 0; l < nlayers; ++l) {
    const ConvArgs& a = P.L[l].a;
    const int gran = 4 * P.L[l].gb;
    const int cinb = a.cin >> 2;
    for (int gk = tid; gk < a.ntab; gk += kStackThreads) {
      const int k0 = gk * gran;
      const int tap = k0 / a.cin, cc = k0 - tap * a.cin;
      int2 e = make_int2(0, kTapNone);
      if (tap < a.kh * a.kw) {
        const int dy = tap / a.kw, dx = tap - dy * a.kw;
        e = make_int2((dy * a.w + dx) * cinb + (cc >> 2), tap_mask(dy, dx));
      }
      sTab[P.L[l].tab_off + gk] = e;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_launch();
  grid_dep_wait();

  if (warp < kGatherWarps) {
    // =================== gather ===================
    const int group = warp >> 2, quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t tA = tmem + (uint32_t)kTmemA + ((uint32_t)(quarter * 32) << 16);
    int it_base = 0, gt_base = 0;
    bool ok = true;
#pragma unroll 1
    for (int l = 0; l < nlayers && ok; ++l) {
      const StackLayer& S = sL[l];
      const int nl = stack_n_local(S.a.ntiles, c, G);
      const int total = nl * S.a.nk;
      const int q0 = ((group - it_base) % kGatherGroups + kGatherGroups) % kGatherGroups;
      const int own = total > q0 ? (total - q0 + kGatherGroups - 1) / kGatherGroups : 0;
      if (own > 0) {
        const int2* tab = sTab + S.tab_off;
        if (S.gb == 16)
          ok = stack_gather_layer<16>(S.a, tab, nl, q0, own, it_base, gt_base, sReady, tA, r, lane, barBase);
        else if (S.gb == 4)
          ok = stack_gather_layer<4>(S.a, tab, nl, q0, own, it_base, gt_base, sReady, tA, r, lane, barBase);
        else
          ok = stack_gather_layer<1>(S.a, tab, nl, q0, own, it_base, gt_base, sReady, tA, r, lane, barBase);
      }
      it_base += total;
      gt_base += nl;
    }
  } else if (warp == kWarpTma) {
    // =================== TMA producer (filters) ===================
    int it = 0;
    bool ok = true;
#pragma unroll 1
    for (int l = 0; l < nlayers && ok; ++l) {
      const StackLayer& S = sL[l];
      const int nl = stack_n_local(S.a.ntiles, c, G);
      const uint32_t bytes = (uint32_t)(S.bn * kBK);
#pragma unroll 1
      for (int jt = 0; jt < nl && ok; ++jt) {
        const int t = c + jt * G;
        const int mt = (int)fdiv((uint32_t)t, S.a.div_nt);
        const int n0 = (t - mt * S.a.nt) * S.bn;
#pragma unroll 1
        for (int k = 0; k < S.a.nk; ++k, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (uint32_t)(it / kStages) & 1u;
          if (!__all_sync(0xffffffffu, mbar_wait_backoff(empty(s), ph ^ 1u, 64))) { ok = false; break; }
          if (elect_one()) {
            mbar_arrive_expect_tx(full(s), bytes);
            tma_load_2d(sB + (uint32_t)(s * L::kB), &P.tm[l], full(s), k * kBK, n0);
          }
          __syncwarp();
        }
      }
    }
    if (!ok) {
      for (int i = it - kStages < 0 ? 0 : it - kStages; i < it; ++i)
        mbar_wait(full(i % kStages), (uint32_t)(i / kStages) & 1u);
    }
    __syncwarp();
  } else if (warp == kWarpMma) {
    // =================== MMA issue ===================
    int it = 0, gt = 0;
    bool ok = true;
#pragma unroll 1
    for (int l = 0; l < nlayers && ok; ++l) {
      const StackLayer& S = sL[l];
      const int nl = stack_n_local(S.a.ntiles, c, G);
      const int nk = S.a.nk;
      const uint32_t idesc = idesc_e4m3_f32(kBM, S.bn);
#pragma unroll 1
      for (int jt = 0; jt < nl && ok; ++jt, ++gt) {
        const int ab = gt & 1;
        if (!__all_sync(0xffffffffu, mbar_wait(acc_empty(ab), ((uint32_t)(gt >> 1) & 1u) ^ 1u))) { ok = false; break; }
        tc_fence_after();
        const uint32_t dacc = tmem + (uint32_t)(ab * kStackBN);
#pragma unroll 1
        for (int k = 0; k < nk; k += 2, it += 2) {
          const bool two = k + 1 < nk;
          const int s0 = it % kStages, s1 = (it + 1) % kStages;
          const uint32_t ph0 = (uint32_t)(it / kStages) & 1u, ph1 = (uint32_t)((it + 1) / kStages) & 1u;
          bool got = mbar_wait(full(s0), ph0);
          if (two) got = got && mbar_wait(full(s1), ph1);
          if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
          tc_fence_after();
          if (elect_one()) {
            const uint32_t a0 = tmem + (uint32_t)(kTmemA + s0 * 32), b0 = sB + (uint32_t)(s0 * L::kB);
#pragma unroll
            for (int kk = 0; kk < kBK / 32; ++kk)
              mma_e4m3_tmem_a(dacc, a0 + (uint32_t)(8 * kk), sdesc_sw128(b0 + 32 * kk), idesc, (k | kk) != 0 ? 1u : 0u);
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
        if (!ok) break;
        if (nk & 1) it -= 1;   // the last round covered a single stage
        if (elect_one()) mma_commit(acc_full(ab));
        __syncwarp();
      }
    }
    if (elect_one()) mma_commit(done_bar);
    __syncwarp();
  } else if (warp == kWarpDep) {
    // =================== tile dependencies ===================
    int gt = 0;
#pragma unroll 1
    for (int l = 0; l < nlayers; ++l) {
      const StackLayer& S = sL[l];
      const int nl = stack_n_local(S.a.ntiles, c, G);
      bool ok = true;
#pragma unroll 1
      for (int jt = 0; jt < nl && ok; ++jt, ++gt) {
        if (S.dep >= 0) ok = wait_deps(sL, P.cnt, S, (int)fdiv((uint32_t)(c + jt * G), S.a.div_nt), lane);
        if (ok && lane == 0) st_release_cta(sReady, (uint32_t)(gt + 1));
      }
      if (!ok) break;
    }
    __syncwarp();
  } else if (warp == kWarpPub) {
    // =================== publisher ===================
    // Lane 0 alone: acquire the CTA-local store count, one gpu-scope fence per
    // batch of stored tiles, then one relaxed add per tile.
    if (lane == 0) {
      int gt = 0;
      uint32_t stored = 0;   // tiles whose stores were observed before the last fence
      bool ok = true;
#pragma unroll 1
      for (int l = 0; l < nlayers && ok; ++l) {
        const StackLayer& S = sL[l];
        const int nl = stack_n_local(S.a.ntiles, c, G);
#pragma unroll 1
        for (int jt = 0; jt < nl; ++jt, ++gt) {
          if ((uint32_t)gt >= stored) {
            ok = wait_ready(sStored, (uint32_t)(kEpiWarps * (gt + 1)), 32);
            if (!ok) break;
            stored = ld_acquire_cta(sStored) / kEpiWarps;
            asm volatile("fence.acq_rel.gpu;" ::: "memory");
          }
          unsigned int* ctr = P.cnt + S.cnt_off + (int)fdiv((uint32_t)(c + jt * G), S.a.div_nt);
          asm volatile("red.relaxed.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
        }
      }
    }
    __syncwarp();
  } else {
    // =================== epilogue ===================
    const int e = warp - kWarpEpi0;
    const int et = tid - kWarpEpi0 * 32;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    int gt = 0;
    bool ok = true;
    int thr_l = -1, thr_n0 = -1, tb = 1;   // channel tile whose thresholds are in sThr[tb]
#pragma unroll 1
    for (int l = 0; l < nlayers; ++l) {
      const StackLayer& S = sL[l];
      const ConvArgs& a = S.a;
      const int nl = stack_n_local(a.ntiles, c, G);
      const int bn = S.bn, CW = bn >> 1;
      const int c_lo = (e >> 2) * CW;
#pragma unroll 1
      for (int jt = 0; jt < nl; ++jt, ++gt) {
        const int t = c + jt * G;
        const int mt = (int)fdiv((uint32_t)t, a.div_nt);
        const int n0 = (t - mt * a.nt) * bn;
        const int m = mt * kBM + row;
        if (l != thr_l || n0 != thr_n0) {
          // a new channel tile: its thresholds go to the other buffer; the barrier also
          // guarantees that every warp is done with the tiles that used that buffer before
          tb ^= 1;
          thr_l = l;
          thr_n0 = n0;
          for (int cc = et; cc < bn; cc += 256) {
            const int nn = n0 + cc;
            float4 v = make_float4(0.f, 0.f, 0.f, 512.f);
            if (nn < a.cout && a.thr)
              v = make_float4(-(float)__ldg(a.thr + 3 * nn), -(float)__ldg(a.thr + 3 * nn + 1),
                              -(float)__ldg(a.thr + 3 * nn + 2), 512.f * (float)__ldg(a.sign + nn));
            sThr[tb * kStackBN + cc] = v;
          }
          named_bar(1, kEpiWarps * 32);
        }
        const int ab = gt & 1;
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait_backoff(acc_full(ab), (uint32_t)(gt >> 1) & 1u, 64));
        if (!ok) {
          if (lane == 0) red_release_cta(sStored, 1u);   // keep the publisher moving after an error
          continue;
        }
        tc_fence_after();
        const uint32_t tacc = tmem + (uint32_t)(ab * kStackBN + c_lo) + ((uint32_t)(quarter * 32) << 16);
        const float4* th = sThr + tb * kStackBN + c_lo;
        if (bn == 128) stack_epi_tile<64>(a, tacc, th, m, n0 + c_lo, acc_empty(ab), lane);
        else if (bn == 64) stack_epi_tile<32>(a, tacc, th, m, n0 + c_lo, acc_empty(ab), lane);
        else stack_epi_tile<16>(a, tacc, th, m, n0 + c_lo, acc_empty(ab), lane);
        __syncwarp();
        if (lane == 0) red_release_cta(sStored, 1u);   // this warp's part of the tile is stored
      }
    }
  }

  // ---- teardown
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    mbar_wait(done_bar, 0);
    tmem_dealloc(tmem, kCols);
  }
}

}  // namespace ifq
