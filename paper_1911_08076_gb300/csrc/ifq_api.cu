// C ABI entry points that launch device work: filter preparation, the
// quantized convolution (tensor-core and bit-serial paths), code pooling,
// the layer-stack driver and its CUDA-graph form, packing helpers and the
// device status word.  Host-only calls (the fold, shapes) live in ifq_host.cpp.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <algorithm>
#include <utility>
#include <vector>

#include "conv_bitserial.cuh"
#include "conv_direct.cuh"
#include "conv_tc.cuh"
#include "conv_warp.cuh"
#include "conv_win.cuh"
#include "ifq.h"
#include "pool_pack.cuh"
#include "selftest.cuh"
#include "stack_tc.cuh"

namespace {

using namespace ifq;

constexpr int kMaxK = 65536;
// Largest accumulator magnitude (2^k - 1) K of the tensor-core path.  Every partial sum is an
// integer multiple of 2^-9 below 2^24 * 2^-9, so an fp32 accumulation is exact; this bound is the
// largest magnitude at which exactness has been checked on GB300 with adversarial inputs
// (accumulators near the bound with odd addends all along K).
constexpr int kTcMaxAcc = 3 * 65536;
constexpr int kMaxDevices = 64;

inline bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }
inline int ceil_div(int a, int b) { return (a + b - 1) / b; }
inline size_t round_up(size_t a, size_t b) { return (a + b - 1) / b * b; }
inline cudaStream_t S(void* s) { return (cudaStream_t)s; }

// Guards the per-device state below (kernel attributes, SM count, occupancy lookups, the address
// of the no-allocation scratch array).
std::mutex g_dev_mu;

// ---------------------------------------------------------------- driver entry point for TMA descriptors

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encode() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  });
  return g_encode != nullptr;
}

// ---------------------------------------------------------------- kernel instances

// Programmatic dependent launch (on unless IFQ_PDL=0): a kernel may start its
// prologue while the previous kernel in the stream finishes; every kernel here
// waits (griddepcontrol.wait) before it touches global memory.
bool pdl_enabled() {
  static const bool on = [] {
    const char* v = getenv("IFQ_PDL");
    return !(v && v[0] == '0');
  }();
  return on;
}

template <typename... Exp, typename... Act>
cudaError_t launch_k(void (*kern)(Exp...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Act&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Act>(args)...);
}

// A launch in clusters of `cluster` CTAs along x (grid.x a multiple of it), with programmatic
// dependent launch as in launch_k.
template <typename... Exp, typename... Act>
cudaError_t launch_k_cluster(void (*kern)(Exp...), int cluster, dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                             Act&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = (unsigned)cluster;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Act>(args)...);
}

// One instance of the tensor-core kernel.  KS > 1 (split K over clusters of KS CTAs): the grid is
// as many clusters as can be resident at once (cudaOccupancyMaxActiveClusters), at most one per
// tile.
template <int BN, int GB, int SB, int SBO, int KS = 1, int BX = 0>
struct TcInst {
  using L = TcSmem<BN, SBO, KS, BX>;
  static_assert(L::bytes <= 232448, "shared memory budget");
  static constexpr auto kern = conv_tc_kernel<BN, GB, SB, SBO, KS, BX>;
  static cudaError_t set_attr() {
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::bytes);
  }
  // clusters of this instance that fit on the current device at once (0: none), looked up once per
  // device under the device-state lock
  static int max_clusters(int nsm) {
    static int cached[kMaxDevices];
    static bool known[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
    std::lock_guard<std::mutex> lk(g_dev_mu);
    if (!known[dev]) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3((unsigned)(nsm / KS * KS));
      cfg.blockDim = dim3(kConvThreads);
      cfg.dynamicSmemBytes = L::bytes;
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = KS;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      int n = 0;
      cached[dev] = cudaOccupancyMaxActiveClusters(&n, kern, &cfg) == cudaSuccess ? n : 0;
      cudaGetLastError();
      known[dev] = true;
    }
    return cached[dev];
  }
  static cudaError_t launch(const CUtensorMap& tm, const ConvArgs& a, int nsm, cudaStream_t st) {
    if constexpr (KS == 1) {
      const int grid = a.ntiles < nsm ? a.ntiles : nsm;
      return launch_k(kern, dim3(grid), dim3(kConvThreads), (size_t)L::bytes, st, tm, a);
    } else {
      const int mc = max_clusters(nsm);
      if (mc < 1) return cudaErrorInvalidConfiguration;
      const int nc = a.ntiles < mc ? a.ntiles : mc;
      return launch_k_cluster(kern, KS, dim3(nc * KS), dim3(kConvThreads), (size_t)L::bytes, st, tm, a);
    }
  }
};

// The (output-channel tile width, K split) instances of the tensor-core kernel; the split ones
// exist for 16-byte granules (every layer with 64 or more 2-bit, or 32 or more 4-bit, channels).
#define IFQ_TC_VARIANTS(X, GB, SB, SBO) X(128, GB, SB, SBO, 1) X(64, GB, SB, SBO, 1) X(32, GB, SB, SBO, 1)
#define IFQ_TC_SPLIT_VARIANTS(X, GB, SB, SBO) X(64, GB, SB, SBO, 2)
// the split instance that expands its filter tiles from sign bits (2-bit codes, 16-byte granules)
using TcSplitBits = TcInst<64, 16, 2, 2, 2, 1>;

template <int GB, int SB, int SBO>
cudaError_t set_attrs_gb() {
  cudaError_t e = cudaSuccess;
#define IFQ_SET(BN, G, S, SO, KS) \
  if (e == cudaSuccess) e = TcInst<BN, G, S, SO, KS>::set_attr();
  IFQ_TC_VARIANTS(IFQ_SET, GB, SB, SBO)
  if constexpr (GB == 16) {
    IFQ_TC_SPLIT_VARIANTS(IFQ_SET, GB, SB, SBO)
    if constexpr (SB == 2 && SBO == 2) {
      if (e == cudaSuccess) e = TcSplitBits::set_attr();
    }
  }
#undef IFQ_SET
  return e;
}

struct DevState {
  bool init = false;
  int nsm = 0;
  bool stack_ok = false;   // the stack kernel fits one CTA per SM (cooperative launch possible)
};
DevState g_dev[kMaxDevices];

// The warp-MMA kernel's instances (conv_warp.cuh) and their shared-memory limit.
constexpr int kWarpMaxSmem = 200 * 1024;
constexpr long long kWarpSmPerSm = 226 * 1024;   // shared memory of an SM available to CTAs
template <int E, int NT, int POOL, int IN8>
cudaError_t set_warp_attr() {
  return cudaFuncSetAttribute(conv_warp_kernel<E, NT, POOL, IN8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kWarpMaxSmem);
}
cudaError_t set_warp_attrs() {
  cudaError_t e = cudaSuccess;
  auto set = [&](cudaError_t r) { if (e == cudaSuccess) e = r; };
  set(set_warp_attr<8, 1, 1, 1>()); set(set_warp_attr<8, 1, 2, 1>());
  set(set_warp_attr<8, 2, 1, 1>()); set(set_warp_attr<8, 2, 2, 1>());
  set(set_warp_attr<8, 4, 1, 1>()); set(set_warp_attr<8, 4, 2, 1>());
  set(set_warp_attr<8, 1, 1, 0>()); set(set_warp_attr<8, 1, 2, 0>());
  set(set_warp_attr<8, 2, 1, 0>()); set(set_warp_attr<8, 2, 2, 0>());
  set(set_warp_attr<8, 4, 1, 0>()); set(set_warp_attr<8, 4, 2, 0>());
  set(set_warp_attr<16, 1, 1, 0>()); set(set_warp_attr<16, 1, 2, 0>());
  set(set_warp_attr<16, 2, 1, 0>()); set(set_warp_attr<16, 2, 2, 0>());
  set(set_warp_attr<16, 4, 1, 0>()); set(set_warp_attr<16, 4, 2, 0>());
  return e;
}

// Per-device one-time setup (shared-memory limits of the kernels, SM count).
int ensure_init(int* nsm_out, bool* stack_ok = nullptr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return IFQ_ECUDA;
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DevState& d = g_dev[dev];
  if (!d.init) {
    if (set_attrs_gb<16, 2, 2>() != cudaSuccess || set_attrs_gb<8, 2, 2>() != cudaSuccess ||
        set_attrs_gb<4, 2, 2>() != cudaSuccess || set_attrs_gb<1, 2, 2>() != cudaSuccess ||
        set_attrs_gb<16, 4, 4>() != cudaSuccess || set_attrs_gb<8, 4, 4>() != cudaSuccess ||
        set_attrs_gb<4, 4, 4>() != cudaSuccess || set_attrs_gb<16, 4, 2>() != cudaSuccess ||
        set_attrs_gb<8, 4, 2>() != cudaSuccess || set_attrs_gb<4, 4, 2>() != cudaSuccess)
      return IFQ_ECUDA;
    if (cudaFuncSetAttribute(conv_win_kernel<0, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, kWinMaxSmem) !=
            cudaSuccess ||
        cudaFuncSetAttribute(conv_win_kernel<0, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, kWinMaxSmem) !=
            cudaSuccess ||
        cudaFuncSetAttribute(conv_win_kernel<1, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, kWinMaxSmem) !=
            cudaSuccess)
      return IFQ_ECUDA;
    if (set_warp_attrs() != cudaSuccess) return IFQ_ECUDA;
    if (cudaDeviceGetAttribute(&d.nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return IFQ_ECUDA;
    if (cudaFuncSetAttribute(conv_stack_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, StackSmem::bytes) !=
        cudaSuccess)
      return IFQ_ECUDA;
    int per_sm = 0, coop = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, conv_stack_kernel, kStackThreads, StackSmem::bytes) !=
        cudaSuccess)
      return IFQ_ECUDA;
    if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess) return IFQ_ECUDA;
    d.stack_ok = per_sm >= 1 && coop != 0;
    d.init = true;
  }
  if (nsm_out) *nsm_out = d.nsm;
  if (stack_ok) *stack_ok = d.stack_ok;
  return IFQ_OK;
}

int launch_1d_blocks(size_t items, int threads, int nsm) {
  size_t b = (items + threads - 1) / threads;
  if (b > (size_t)nsm * 32) b = (size_t)nsm * 32;
  return b < 1 ? 1 : (int)b;
}

// Multiply-high divisor for n / d with 0 <= n < 2^31 (d >= 1): shift = ceil(log2 d),
// mul = floor(2^32 * (2^shift - d) / d) + 1, n / d = (umulhi(n, mul) + n) >> shift.
FastDiv make_fastdiv(uint32_t d) {
  FastDiv f;
  f.d = d;
  uint32_t l = 0;
  while ((1ull << l) < d) ++l;
  f.shift = l;
  f.mul = (uint32_t)(((1ull << 32) * ((1ull << l) - d)) / d + 1ull);
  return f;
}

int env_int(const char* name, int dflt) {
  const char* v = getenv(name);
  return (v && *v) ? atoi(v) : dflt;
}

// ---------------------------------------------------------------- descriptors and planning

// Code width of a descriptor's kbits field (0 means 2): k, the stored field width sb (2 for
// k = 2, 4 for k = 3 and 4) and the thresholds per channel 2^k - 1.  Returns an ifq_status.
int code_width(int kbits, int* k, int* sb, int* lvl) {
  if (kbits < 0) return IFQ_EINVAL;
  const int kk = kbits == 0 ? 2 : kbits;
  if (kk < 2 || kk > 4) return IFQ_EUNSUPPORTED;
  *k = kk;
  *sb = kk == 2 ? 2 : 4;
  *lvl = (1 << kk) - 1;
  return IFQ_OK;
}

struct ConvGeom {
  int ho, wo, M, K, Kpad, kwords;   // K: kh*kw*cin of the filters; Kpad: the kernel's K rounded up to 128
  int pool, pho, pwo;   // fused pool window (1: none) and the output shape after it
  int kb, sb, lvl;      // output code width k, its stored field bits, thresholds per channel
  bool in8;             // 8-bit input values (one byte each, read as two 4-bit fields)
  int sbi, cink, Kk;    // input field bits, the kernel's input channels (fields) and its K
};

int check_conv(const ifq_conv_desc* d, ConvGeom* g) {
  if (!d) return IFQ_EINVAL;
  int rc = ifq_conv_out_shape(d, &g->pho, &g->pwo);   // output shape, after the fused pool if any
  if (rc) return rc;
  if ((rc = code_width(d->kbits, &g->kb, &g->sb, &g->lvl))) return rc;
  if (d->in_bits < 0) return IFQ_EINVAL;
  if (d->in_bits != 0 && d->in_bits != 8 && d->in_bits != g->kb) return IFQ_EUNSUPPORTED;
  g->in8 = d->in_bits == 8;
  g->pool = d->pool > 1 ? d->pool : 1;
  g->ho = g->pho * g->pool;                            // the convolution's own output
  g->wo = g->pwo * g->pool;
  if (g->pool > 1 && d->out_mode != IFQ_OUT_CODES) return IFQ_EUNSUPPORTED;
  if (d->cin % 4 != 0) return IFQ_ESHAPE;
  if (d->out_mode < IFQ_OUT_CODES || d->out_mode > IFQ_OUT_BOTH) return IFQ_EINVAL;
  if ((d->out_mode & IFQ_OUT_CODES) && d->cout % 4 != 0) return IFQ_ESHAPE;
  if (d->path < IFQ_PATH_AUTO || d->path > IFQ_PATH_WARP) return IFQ_EINVAL;
  const long long K = (long long)d->kh * d->kw * d->cin;
  const long long M = (long long)d->n * g->ho * g->wo;
  if (K > kMaxK || d->cout > 65536 || M >= (1LL << 31)) return IFQ_ERANGE;
  if ((long long)d->n * d->h * d->w * d->cin >= (1LL << 40)) return IFQ_ERANGE;
  g->M = (int)M;
  g->K = (int)K;
  // an 8-bit value is two 4-bit fields (low nibble first): the kernel sees 2*cin fields of 4 bits
  g->sbi = g->in8 ? 4 : g->sb;
  g->cink = g->in8 ? 2 * d->cin : d->cin;
  g->Kk = g->in8 ? 2 * (int)K : (int)K;
  g->Kpad = (int)round_up((size_t)g->Kk, kBK);
  g->kwords = ceil_div((int)K, 32);
  return IFQ_OK;
}

size_t prep_bits_offset(const ifq_conv_desc* d, const ConvGeom& g) {
  return round_up((size_t)d->cout * g.Kpad, 256);
}

// Prepared filters: e4m3 rows, then the sign words, then (layers on 8-bit inputs) the per-tap
// masks of the direct path.
size_t prep_masks_offset(const ifq_conv_desc* d, const ConvGeom& g) {
  return prep_bits_offset(d, g) + round_up((size_t)d->cout * g.kwords * 4, 256);
}

// Layers on codes: then the sign bits in the e4m3 rows' K order, [cout][Kpad / 8] bytes, where the
// 8-bit-input layers keep their masks.
size_t prep_pbits_offset(const ifq_conv_desc* d, const ConvGeom& g) { return prep_masks_offset(d, g); }

size_t prep_bytes(const ifq_conv_desc* d, const ConvGeom& g) {
  return g.in8 ? prep_masks_offset(d, g) + (size_t)g.K * 4 : prep_pbits_offset(d, g) + (size_t)d->cout * g.Kpad / 8;
}

bool tc_supported(const ifq_conv_desc* d, const ConvGeom& g);

// The direct CUDA-core path: layers on 8-bit input values with at most 32 output channels and
// K <= 257 (the two 16-bit channel sums of a register stay apart).
bool direct_supported(const ifq_conv_desc* d, const ConvGeom& g) {
  return g.in8 && d->cout <= kDirectMaxCout && g.K <= kDirectMaxK;
}

// The narrow bit-serial kernel: 2-bit codes, cin 4, 8 or 16, 3x3, stride 1, cout <= 32 (and a
// multiple of 4), pool 1 or 2.
bool narrow_supported(const ifq_conv_desc* d, const ConvGeom& g) {
  return g.kb == 2 && !g.in8 && (d->cin == 4 || d->cin == 8 || d->cin == 16) && d->kh == 3 && d->kw == 3 &&
         d->stride == 1 && d->cout <= 32 && d->cout % 4 == 0 && (g.pool == 1 || g.pool == 2);
}

// Where the narrow kernel beats the tensor cores (measured on GB300): the narrowest layers, whose
// 128-pixel tiles of one K stage each are per-tile-overhead bound on the tensor cores.
bool narrow_wins(const ifq_conv_desc* d, const ConvGeom& g) {
  return narrow_supported(d, g) && d->cin * d->cout <= 128;
}

// The narrow bit-serial kernel instance for cin, pool and the channel bound.
template <int CIN, int P>
cudaError_t launch_narrow_cp(int cout, dim3 grid, dim3 block, const NarrowArgs& a, cudaStream_t st) {
  if (cout <= 8) return launch_k(conv_bitserial_narrow_kernel<CIN, P, 8>, grid, block, 0, st, a);
  if (cout <= 16) return launch_k(conv_bitserial_narrow_kernel<CIN, P, 16>, grid, block, 0, st, a);
  return launch_k(conv_bitserial_narrow_kernel<CIN, P, 32>, grid, block, 0, st, a);
}

cudaError_t launch_narrow(int cin, int pool, int cout, dim3 grid, dim3 block, const NarrowArgs& a, cudaStream_t st) {
  if (cin == 4) return pool == 2 ? launch_narrow_cp<4, 2>(cout, grid, block, a, st) : launch_narrow_cp<4, 1>(cout, grid, block, a, st);
  if (cin == 8) return pool == 2 ? launch_narrow_cp<8, 2>(cout, grid, block, a, st) : launch_narrow_cp<8, 1>(cout, grid, block, a, st);
  return pool == 2 ? launch_narrow_cp<16, 2>(cout, grid, block, a, st) : launch_narrow_cp<16, 1>(cout, grid, block, a, st);
}

// Geometry of the window kernel (conv_win.cuh) for a layer, or false where it does not apply:
// 2-bit codes in and out, stride 1, k x k with "same" padding (k odd, <= 7), cin 16 or a multiple of
// 32, cout 32, 64 or a multiple of 128 (at most one channel tile per SM), a fused pool of 2 on even
// sizes or none, input rows of whole 16-byte units (the copy engine stages them), an output row of
// at most 256 anchors, and the resident filters plus two staging and two band buffers within the
// shared memory of one CTA.  Fills every field but the pointers.
bool win_plan(const ifq_conv_desc* d, const ConvGeom& g, int nsm, WinArgs* wa, size_t* smem) {
  if (env_int("IFQ_WIN", 1) == 0) return false;
  if (g.in8 || g.kb != 2) return false;
  const int k = d->kh;
  if (d->stride != 1 || d->kw != k || (k & 1) == 0 || k > 7 || 2 * d->pad != k - 1) return false;
  if (!(d->cin == 16 || d->cin % 32 == 0)) return false;
  int ct;
  if (d->cout == 32 || d->cout == 64) ct = d->cout;
  else if (d->cout % 128 == 0) ct = 128;
  else return false;
  const int nct = d->cout / ct;
  if (nct > nsm) return false;
  if (g.pool != 1 && g.pool != 2) return false;
  const bool pool = g.pool == 2;
  const int H = g.ho, W = g.wo;
  if (pool && ((H & 1) || (W & 1))) return false;
  const int cinb = d->cin / 4;
  const long long row_bytes = (long long)W * cinb;   // one input row, copied whole
  if (row_bytes % 16 != 0) return false;
  const int ry = 128 / ct, planes = d->cin / 16;
  // anchor rows per tile: as many as fit N <= 256, fewer while the buffers exceed shared memory
  const int pitch = ry == 1 && pool ? (int)round_up((size_t)(W + k - 1), 16) : W + k - 1;
  if (pitch > 256) return false;
  const int r_max = ry > 1 ? std::max(1, std::min(256 / pitch, ceil_div(H, ry))) : std::min(H, 256 / pitch);
  const int kc_real = (ry + k - 1) * k * planes;
  const int kc = (int)round_up((size_t)kc_real, 2);
  if (kc / 2 > kWinMaxMma) return false;
  const uint32_t a_bytes = (uint32_t)ceil_div(kc, 8) * 16384u;   // 128-byte K stages of 128 rows
  const uint32_t xchg = ry > 1 && pool ? (uint32_t)kWinXchgBytes : 0u;   // row-pair exchange (stacked rows)
  int R = 0, seg_pitch = 0, rb = 0, N = 0, nseg = 0;
  uint32_t ps = 0, band_bytes = 0, stage_bytes = 0;
  size_t need = 0;
  for (int r = r_max; r >= 1; --r) {
    if (ry == 1 && pool && (r & 1)) continue;   // pooled row pairs
    // ry > 1: r row bands of ry output rows side by side along N;
    // ry = 1: r consecutive output rows sharing the band's input rows
    const int sp = ry > 1 ? r * pitch : pitch;
    const int rbr = ry > 1 ? ry + k - 1 : r + k - 1;
    const int n_ = (int)round_up((size_t)((r - 1) * pitch + W), 16);   // the last row's padding is not an anchor
    if (n_ > 256) continue;
    const int ns = ry > 1 ? r : 1;
    // slots a plane needs: the band rows, and what the MMAs read past them (N anchors from the
    // farthest tap, and the slot after the last core column), with slack
    const int iy_max = ry + k - 2;
    const int slots = std::max(rbr * sp, iy_max * sp + (k - 1) + n_ + 2) + 4;
    const uint32_t ps_ = (uint32_t)round_up((size_t)slots * 16, 128) + (planes > 1 ? 16u : 0u);
    const uint32_t bb = (uint32_t)round_up((size_t)planes * ps_, 1024);
    const uint32_t sb = (uint32_t)round_up((size_t)ns * rbr * row_bytes, 128);
    const size_t nd = 1024 + (size_t)a_bytes + 2 * (size_t)bb + 2 * (size_t)sb + xchg + kWinTabBytes + 128 +
                      kWinStashBytes;
    if (nd <= (size_t)kWinMaxSmem) {
      R = r; seg_pitch = sp; rb = rbr; N = n_; nseg = ns; ps = ps_; band_bytes = bb; stage_bytes = sb; need = nd;
      break;
    }
  }
  if (R == 0) return false;
  if (wa) {
    memset(wa, 0, sizeof(*wa));
    wa->n = d->n; wa->h = H; wa->w = W; wa->cin = d->cin; wa->cout = d->cout; wa->k = k; wa->pad = d->pad;
    wa->Kpad = g.Kpad;
    wa->planes = planes; wa->ct = ct; wa->ry = ry; wa->nct = nct; wa->R = R; wa->rows = ry * R;
    wa->pitch = pitch; wa->seg_pitch = seg_pitch; wa->nseg = nseg;
    wa->N = N; wa->rb = rb; wa->kc = kc; wa->kc_real = kc_real;
    wa->bands = ceil_div(H, wa->rows);
    wa->ntiles = d->n * wa->bands;
    wa->row_bytes = (int)row_bytes;
    wa->plane_stride = ps;
    wa->band_bytes = band_bytes;
    wa->stage_bytes = stage_bytes;
    wa->a_bytes = a_bytes;
    wa->xchg_bytes = xchg;
    wa->div_planes = make_fastdiv((uint32_t)planes);
    wa->div_pitch = make_fastdiv((uint32_t)pitch);
    wa->div_seg = make_fastdiv((uint32_t)seg_pitch);
    wa->div_bands = make_fastdiv((uint32_t)wa->bands);
    wa->div_chunks = make_fastdiv((uint32_t)(row_bytes / 16));
    wa->div_rb = make_fastdiv((uint32_t)rb);
  }
  if (smem) *smem = need;
  return true;
}

bool win_supported(const ifq_conv_desc* d, const ConvGeom& g) {
  int nsm = 0;
  if (ensure_init(&nsm)) nsm = 148;   // no device: plan as for a full GB300
  return win_plan(d, g, nsm, nullptr, nullptr);
}

// Where the window kernel is the default (measured on GB300 against the tensor-core kernel, layer
// by layer in the benchmark stacks): layers with a fused 2 x 2 pool and at most 64 input
// channels.  Tiny-YOLO conv2 (16 -> 32 at 208 x 208, b64) 54 vs 128 us, conv3 34 vs 51, conv4 21 vs
// 28; IFQ-Tinier-YOLO conv3..conv5 24 / 17 / 14 vs 38 / 21 / 16 us.  Without a pool its epilogue
// thresholds twice the columns, and with 128 or more input channels its resident filter block and
// per-tile setup cost more than the other kernel's gather: there the tensor-core kernel stays ahead
// (ResNet-18 stage 1: 21 vs 18 us; Tinier conv6: 16 vs 14 us).
bool win_wins(const ifq_conv_desc* d, const ConvGeom& g) {
  return g.pool == 2 && d->cin <= 64 && win_supported(d, g);
}

// Geometry of the warp-MMA kernel (conv_warp.cuh) for a layer, or false where it does not apply:
// 3 x 3, stride 1, padding 1; 2-bit codes in with cin 8 or 16, or 8-bit values with cin 4; 2-bit
// codes and / or int32 accumulators out, cout 8, 16 or 32; no pool or a 2 x 2 pool on even sizes;
// a band of at least two output rows within the shared memory of one CTA.  Fills every field but
// the pointers; *E and *NT select the instance.
bool warp_plan(const ifq_conv_desc* d, const ConvGeom& g, WarpConvArgs* wa, size_t* smem, int* E, int* NT) {
  if (env_int("IFQ_WARP", 1) == 0) return false;
  if (d->kh != 3 || d->kw != 3 || d->stride != 1 || d->pad != 1) return false;
  if (g.in8 ? d->cin != 4 : !(g.sbi == 2 && (d->cin == 8 || d->cin == 16))) return false;
  if (g.kb != 2 || !(d->cout == 8 || d->cout == 16 || d->cout == 32)) return false;
  if (g.pool != 1 && g.pool != 2) return false;
  if (g.pool == 2 && ((g.ho & 1) || (g.wo & 1))) return false;
  const int e = g.in8 ? 8 : d->cin, nt = d->cout / 8;
  const int pp = e / 8, ksd = (3 * pp + 3) / 4, nb = nt * 3 * ksd;
  const int strips = ceil_div(g.wo, 16);
  const long long row_bytes = (long long)(16 * strips + 2) * e;
  const int cinb = g.in8 ? d->cin : d->cin / 4;
  const long long raw_pitch = (long long)g.wo * cinb;
  const int bulk = raw_pitch % 16 == 0 ? 1 : 0;   // whole 16-byte units: the copy engine stages the rows
  if (row_bytes > kWarpMaxSmem) return false;
  // output rows per band: up to 16, fewer while two CTAs' shared memory would not fit an SM
  // (then while one would not), so that a CTA's copy and expansion overlap the other's MMAs
  auto bytes_of = [&](int rb) {
    return (long long)warp_smem(nb, d->cout, rb, (int)row_bytes, (int)raw_pitch, bulk).bytes;
  };
  int rb = std::min(16, (int)round_up((size_t)g.ho, 2));
  while (rb > 2 && 2 * bytes_of(rb) > kWarpSmPerSm) rb -= 2;
  while (rb > 2 && bytes_of(rb) > kWarpMaxSmem) rb -= 2;
  if (bytes_of(rb) > kWarpMaxSmem) return false;
  if (wa) {
    memset(wa, 0, sizeof(*wa));
    wa->n = d->n; wa->h = g.ho; wa->w = g.wo; wa->cin = d->cin; wa->cout = d->cout; wa->kwords = g.kwords;
    wa->pho = g.pho; wa->pwo = g.pwo;
    wa->strips = strips;
    wa->rb = rb;
    wa->bands = ceil_div(g.ho, rb);
    wa->row_bytes = (int)row_bytes;
    wa->units = strips * (rb / 2);
    wa->bulk = bulk;
    wa->raw_pitch = (int)raw_pitch;
    wa->total = d->n * wa->bands;
    wa->div_bands = make_fastdiv((uint32_t)wa->bands);
    wa->div_strips = make_fastdiv((uint32_t)strips);
    wa->div_slots = make_fastdiv((uint32_t)(16 * strips + 2));
  }
  if (smem) *smem = (size_t)bytes_of(rb);
  if (E) *E = e;
  if (NT) *NT = nt;
  return true;
}

bool warp_supported(const ifq_conv_desc* d, const ConvGeom& g) {
  return warp_plan(d, g, nullptr, nullptr, nullptr, nullptr);
}

// Where the warp-MMA kernel is the default (measured on GB300, full-size layers at batch 64, L2
// flushed, against the kernel each layer took before): 2-bit layers with 8 input channels
// (IFQ-Tinier-YOLO conv2, 8 -> 16 at 208 x 208: 46 vs 103 us on the narrow bit-serial kernel with the
// fused pool, 62 vs 107 us without) and 8-bit-input layers without a fused pool (3 x 3 4 -> 8 at
// 416 x 416: 144 vs 207 us on the direct kernel).  Elsewhere it loses: one e4m3 mma.sync issues about
// four instructions on this GPU, and the tcgen05 window kernel (16-channel layers: Tiny-YOLO conv2
// 54 vs 124 us) or the direct kernel (the pooled first layer: 91 vs 107 us) stays ahead.
bool warp_wins(const ifq_conv_desc* d, const ConvGeom& g) {
  return warp_supported(d, g) && (g.in8 ? g.pool == 1 : d->cin == 8);
}

// A persistent launch: as many CTAs as fit the SMs at once (at most one per band).
template <int E, int NT, int POOL, int IN8>
cudaError_t launch_warp_inst(int nsm, size_t smem, cudaStream_t st, const WarpConvArgs& a) {
  const int threads = warp_conv_threads(E, NT);
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, conv_warp_kernel<E, NT, POOL, IN8>, threads,
                                                                smem);
  if (e != cudaSuccess) return e;
  const int grid = std::max(1, std::min(a.total, nsm * std::max(1, per_sm)));
  return launch_k(conv_warp_kernel<E, NT, POOL, IN8>, dim3((unsigned)grid), dim3((unsigned)threads), smem, st, a);
}

template <int E, int NT>
cudaError_t launch_warp_en(int pool, bool in8, int nsm, size_t smem, cudaStream_t st, const WarpConvArgs& a) {
  if constexpr (E == 8) {
    if (in8)
      return pool == 2 ? launch_warp_inst<E, NT, 2, 1>(nsm, smem, st, a) : launch_warp_inst<E, NT, 1, 1>(nsm, smem, st, a);
  }
  return pool == 2 ? launch_warp_inst<E, NT, 2, 0>(nsm, smem, st, a) : launch_warp_inst<E, NT, 1, 0>(nsm, smem, st, a);
}

cudaError_t launch_warp(int E, int NT, int pool, bool in8, int nsm, size_t smem, cudaStream_t st,
                        const WarpConvArgs& a) {
  if (E == 8)
    return NT == 1 ? launch_warp_en<8, 1>(pool, in8, nsm, smem, st, a)
                   : (NT == 2 ? launch_warp_en<8, 2>(pool, in8, nsm, smem, st, a)
                              : launch_warp_en<8, 4>(pool, in8, nsm, smem, st, a));
  return NT == 1 ? launch_warp_en<16, 1>(pool, false, nsm, smem, st, a)
                 : (NT == 2 ? launch_warp_en<16, 2>(pool, false, nsm, smem, st, a)
                            : launch_warp_en<16, 4>(pool, false, nsm, smem, st, a));
}

int choose_path(const ifq_conv_desc* d, const ConvGeom& g) {
  int path = d->path;
  if (path == IFQ_PATH_AUTO) {
    const int forced = env_int("IFQ_FORCE_PATH", 0);
    path = forced ? forced
                  : (warp_wins(d, g) ? IFQ_PATH_WARP
                                     : (direct_supported(d, g) ? IFQ_PATH_DIRECT
                                                               : (win_wins(d, g) ? IFQ_PATH_WIN
                                                                                 : (narrow_wins(d, g) ? IFQ_PATH_BITSERIAL
                                                                                                      : IFQ_PATH_TC))));
  }
  if (path == IFQ_PATH_WARP && !warp_supported(d, g)) path = IFQ_PATH_TC;
  if (path == IFQ_PATH_WIN && !win_supported(d, g)) path = IFQ_PATH_TC;
  if (path == IFQ_PATH_DIRECT && !direct_supported(d, g)) path = IFQ_PATH_TC;
  if (path == IFQ_PATH_TC && !tc_supported(d, g)) path = IFQ_PATH_BITSERIAL;
  // the fused pool has a bit-serial form only in the narrow kernel; 8-bit inputs have none
  if (path == IFQ_PATH_BITSERIAL && (g.in8 || (g.pool > 1 && !narrow_supported(d, g)))) return -1;
  return path;
}

// Output-channel tile BN of the persistent tensor-core kernel (128 pixels x BN).
// Cost model: one 128 x BN x 32 e4m3 MMA takes t(BN) cycles on GB300 (measured
// 52 / 54 / 72 at BN = 32 / 64 / 128, independent of whether consecutive MMAs
// share an accumulator), a K stage issues 4 of them, and the makespan is
// ceil(tiles / SMs) * nk * 4 * t(BN).  Ties go to the wider tile.
int choose_bn(const ConvGeom& g, int cout, int nsm) {
  const int forced = env_int("IFQ_TC_BN", 0);
  if (forced == 32 || forced == 64 || forced == 128) return forced;
  int best = 32;
  double best_cost = 1e300;
  for (int bn = 32; bn <= 128; bn *= 2) {
    if (bn > 32 && bn / 2 >= cout) break;   // no wider than needed to cover cout
    const long long tiles = (long long)ceil_div(g.M, kBM) * ceil_div(cout, bn);
    const double t = bn == 32 ? 52.0 : (bn == 64 ? 54.0 : 72.0);
    const double cost = (double)((tiles + nsm - 1) / nsm) * t;
    if (cost <= best_cost * (1.0 + 1e-9)) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

template <int GB, int SB, int SBO>
int tc_max_clusters(int bn, int ks, int nsm) {
  if constexpr (GB == 16) {
#define IFQ_MC(BN, G, S, SO, KS) \
  if (bn == BN && ks == KS) return TcInst<BN, G, S, SO, KS>::max_clusters(nsm);
    IFQ_TC_SPLIT_VARIANTS(IFQ_MC, GB, SB, SBO)
#undef IFQ_MC
  }
  return 0;
}

// K split of the tensor-core kernel (1: none).  Splitting K over a cluster of two CTAs halves each
// CTA's K stages but adds the exchange of partial sums, and with as many tiles as SMs it leaves the
// per-CTA work unchanged.  Measured on GB300: AlexNet FC6 (one 128-row tile, K = 9216) 20.6 -> 16.5
// us at BN = 64; every ResNet-18 layer at batch 32 slower (the 7x7 512-channel layers have 104
// tiles at BN = 64, so a split would need 208 CTAs).  So the split is taken only where the unsplit
// layer would leave more than half of the SMs idle, the split grid fits in one wave of clusters and
// every CTA keeps at least eight K stages.  IFQ_TC_KS = 1 / 2 forbids / forces it where eligible.
template <int GB, int SB, int SBO>
void choose_split(const ConvGeom& g, int cout, int nsm, int* bn, int* ks) {
  *ks = 1;
  if constexpr (GB == 16) {
    const int forced = env_int("IFQ_TC_KS", 0);
    if (forced == 1) return;
    const int nk = g.Kpad / kBK;
    if (cout <= 32 || nk < 4) return;   // the split instance is BN = 64, KS = 2
    const long long tiles = (long long)ceil_div(g.M, kBM) * ceil_div(cout, 64);
    const int mc = tc_max_clusters<GB, SB, SBO>(64, 2, nsm);
    if (mc < 1) return;
    if (forced == 2 || (nk >= 16 && 2 * tiles <= nsm && tiles <= mc)) {
      *bn = 64;
      *ks = 2;
    }
  }
}

template <int GB, int SB, int SBO>
cudaError_t launch_tc_gb(int bn, int ks, const CUtensorMap& tm, const ConvArgs& a, int nsm, cudaStream_t st,
                         bool bx = false) {
  if constexpr (GB == 16 && SB == 2 && SBO == 2) {
    if (bx && bn == 64 && ks == 2) return TcSplitBits::launch(tm, a, nsm, st);
  }
#define IFQ_LAUNCH(BN, G, S, SO, KS) \
  if (bn == BN && ks == KS) return TcInst<BN, G, S, SO, KS>::launch(tm, a, nsm, st);
  IFQ_TC_VARIANTS(IFQ_LAUNCH, GB, SB, SBO)
  if constexpr (GB == 16) {
    IFQ_TC_SPLIT_VARIANTS(IFQ_LAUNCH, GB, SB, SBO)
  }
#undef IFQ_LAUNCH
  return cudaErrorInvalidValue;
}

// Bytes of packed codes per input pixel.
int pixel_bytes(const ifq_conv_desc*, const ConvGeom& g) { return g.cink * g.sbi / 8; }

// Bytes of packed codes per gathered granule: the largest of 16, 8, 4, 1 that divides a pixel's
// bytes (the persistent stack kernel has no 8-byte instance: 16, 4, 1 there).
int granule_bytes(const ifq_conv_desc* d, const ConvGeom& g, bool stack = false) {
  const int pb = pixel_bytes(d, g);
  return pb % 16 == 0 ? 16 : (pb % 8 == 0 && !stack ? 8 : (pb % 4 == 0 ? 4 : 1));
}

// Whether the tensor-core kernel supports this shape: an accumulator magnitude inside the
// checked exact range, filter rows and columns addressable by 15-bit masks (kh, kw <= 15), a K-granule table that fits, and an
// instantiated granule (4-bit fields need 4-byte granules, cin % 8 == 0).
bool tc_supported(const ifq_conv_desc* d, const ConvGeom& g) {
  const long long amax = (long long)(g.in8 ? 255 : g.lvl) * g.K;   // largest |A|
  if (amax > kTcMaxAcc || d->kh > 15 || d->kw > 15) return false;
  const int gb = granule_bytes(d, g, true);   // the smaller granule of the two kernels: the larger table
  if (g.sbi == 4 && gb == 1) return false;
  if ((long long)g.Kpad * g.sbi / 8 / gb > kMaxTab) return false;
  const long long pb = pixel_bytes(d, g);
  const long long span = ((long long)(d->kh - 1) * d->w + d->kw) * pb + pb;
  return span < (1LL << 31);
}

// TMA descriptor of the prepared e4m3 filter rows: [cout][Kpad] bytes, box 128 x bn, 128B swizzle.
bool encode_wmap(const ifq_conv_desc* d, const ConvGeom& g, const void* w_prep, int bn, CUtensorMap* tm) {
  if (!get_encode()) return false;
  cuuint64_t gdim[2] = {(cuuint64_t)g.Kpad, (cuuint64_t)d->cout};
  cuuint64_t gstride[1] = {(cuuint64_t)g.Kpad};
  cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)bn};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(w_prep), gdim, gstride, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// TMA descriptor of the filter sign bits in the e4m3 rows' K order ([cout][Kpad / 8] bytes after the
// sign words): boxes of bn rows x 16 bytes (one K stage), no swizzle.
bool encode_bitmap(const ifq_conv_desc* d, const ConvGeom& g, const void* w_prep, int bn, CUtensorMap* tm) {
  if (!get_encode()) return false;
  cuuint64_t gdim[2] = {(cuuint64_t)(g.Kpad / 8), (cuuint64_t)d->cout};
  cuuint64_t gstride[1] = {(cuuint64_t)(g.Kpad / 8)};
  cuuint32_t box[2] = {16u, (cuuint32_t)bn};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, (uint8_t*)const_cast<void*>(w_prep) + prep_pbits_offset(d, g),
                  gdim, gstride, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

void fill_conv_args(const ifq_conv_desc* d, const ConvGeom& g, int bn, const void* x, const int32_t* thr,
                    const int8_t* sign, uint8_t* yc, int32_t* ya, ConvArgs* a, bool stack = false) {
  a->x = (const uint8_t*)x;
  a->wbits = nullptr;
  a->thr = thr;
  a->sign = sign;
  a->y_codes = yc;
  a->y_acc = ya;
  a->n = d->n; a->h = d->h; a->w = d->w; a->cin = g.cink; a->cout = d->cout;
  a->kh = d->kh; a->kw = d->kw; a->stride = d->stride; a->pad = d->pad; a->ho = g.ho; a->wo = g.wo;
  a->cinb = pixel_bytes(d, g);
  a->lvl = g.lvl;
  a->M = g.M;
  a->K = g.Kk;
  a->nk = g.Kpad / kBK;
  a->nt = ceil_div(d->cout, bn);
  a->ntiles = ceil_div(g.M, kBM) * a->nt;
  a->ntab = g.Kpad * g.sbi / 8 / granule_bytes(d, g, stack);
  a->div_hw = make_fastdiv((uint32_t)(g.ho * g.wo));
  a->div_wo = make_fastdiv((uint32_t)g.wo);
  a->div_nt = make_fastdiv((uint32_t)a->nt);
  a->lpool = g.pool == 4 ? 2 : (g.pool == 2 ? 1 : 0);
  a->early = 0;
  a->div_phw = make_fastdiv((uint32_t)(g.pho * g.pwo));
  a->div_pwo = make_fastdiv((uint32_t)g.pwo);
}

// early: the kernels before this one in the stream write neither w_prep nor thr / sign (a layer of a
// stack after the first), so the tensor-core kernel may load them before its dependency wait.
int run_conv(const ifq_conv_desc* d, const void* x, const void* w_prep, const int32_t* thr, const int8_t* sign,
             void* y_codes, int32_t* y_acc, cudaStream_t st, bool early = false) {
  ConvGeom g;
  int rc = check_conv(d, &g);
  if (rc) return rc;
  if (!x || !w_prep) return IFQ_EINVAL;
  if ((d->out_mode & IFQ_OUT_CODES) && (!y_codes || !thr || !sign)) return IFQ_EINVAL;
  if ((d->out_mode & IFQ_OUT_ACC) && !y_acc) return IFQ_EINVAL;
  if (!aligned16(x) || !aligned16(w_prep) || (y_codes && !aligned16(y_codes)) || (y_acc && !aligned16(y_acc)))
    return IFQ_EALIGN;
  if (g.M == 0) return IFQ_OK;   // an empty batch: nothing to compute
  int nsm = 0;
  if ((rc = ensure_init(&nsm))) return rc;
  uint8_t* yc = (d->out_mode & IFQ_OUT_CODES) ? (uint8_t*)y_codes : nullptr;
  int32_t* ya = (d->out_mode & IFQ_OUT_ACC) ? y_acc : nullptr;
  const int path = choose_path(d, g);
  if (path < 0) return IFQ_EUNSUPPORTED;
  cudaError_t e;
  if (path == IFQ_PATH_DIRECT) {
    DirectArgs a;
    a.x = (const uint8_t*)x;
    a.wmask = (const uint32_t*)((const uint8_t*)w_prep + prep_masks_offset(d, g));
    a.thr = thr;
    a.sign = sign;
    a.y_codes = yc;
    a.y_acc = ya;
    a.n = d->n; a.h = d->h; a.w = d->w; a.cin = d->cin; a.cout = d->cout;
    a.kh = d->kh; a.kw = d->kw; a.stride = d->stride; a.pad = d->pad; a.ho = g.ho; a.wo = g.wo;
    a.K = g.K;
    a.lvl = g.lvl;
    a.sbo = g.sb;
    a.pool = g.pool;
    a.pho = g.pho;
    a.pwo = g.pwo;
    a.total = d->n * g.pho * g.pwo;
    a.div_pwo = make_fastdiv((uint32_t)g.pwo);
    a.div_pho = make_fastdiv((uint32_t)g.pho);
    const dim3 grid(launch_1d_blocks((size_t)a.total, kDirectThreads, nsm)), block(kDirectThreads);
    // the RGB first layer (cin 4, 3x3, stride 1, pool 1 or 2) has its own instances
    const bool rgb3 = d->cin == 4 && d->kh == 3 && d->kw == 3 && d->stride == 1 && (g.pool == 1 || g.pool == 2);
    if (rgb3 && d->cout <= 8)
      e = g.pool == 2 ? launch_k(conv_direct_rgb3_kernel<8, 2>, grid, block, 0, st, a)
                      : launch_k(conv_direct_rgb3_kernel<8, 1>, grid, block, 0, st, a);
    else if (rgb3 && d->cout <= 16)
      e = g.pool == 2 ? launch_k(conv_direct_rgb3_kernel<16, 2>, grid, block, 0, st, a)
                      : launch_k(conv_direct_rgb3_kernel<16, 1>, grid, block, 0, st, a);
    else if (d->cout <= 8) e = launch_k(conv_direct_kernel<4>, grid, block, 0, st, a);
    else if (d->cout <= 16) e = launch_k(conv_direct_kernel<8>, grid, block, 0, st, a);
    else e = launch_k(conv_direct_kernel<16>, grid, block, 0, st, a);
  } else if (path == IFQ_PATH_WARP) {
    WarpConvArgs wa;
    size_t smem = 0;
    int E = 0, NT = 0;
    if (!warp_plan(d, g, &wa, &smem, &E, &NT)) return IFQ_EUNSUPPORTED;
    wa.x = (const uint8_t*)x;
    wa.wbits = (const uint32_t*)((const uint8_t*)w_prep + prep_bits_offset(d, g));
    wa.thr = thr;
    wa.sign = sign;
    wa.y_codes = yc;
    wa.y_acc = ya;
    e = launch_warp(E, NT, g.pool, g.in8, nsm, smem, st, wa);
  } else if (path == IFQ_PATH_WIN) {
    WinArgs wa;
    size_t smem = 0;
    if (!win_plan(d, g, nsm, &wa, &smem)) return IFQ_EUNSUPPORTED;
    wa.x = (const uint8_t*)x;
    wa.w_prep = (const uint8_t*)w_prep;
    wa.thr = thr;
    wa.sign = sign;
    wa.y_codes = yc;
    wa.y_acc = ya;
    // CTAs come in groups of nct, one per channel tile, each group sharing the band tiles
    const int per = std::max(1, std::min(wa.ntiles, nsm / wa.nct));
    const dim3 grid((unsigned)(per * wa.nct)), block(kWinThreads);
    wa.early = early ? 1 : 0;
    CUtensorMap tma;
    if (!encode_wmap(d, g, w_prep, wa.ct, &tma)) return IFQ_ECUDA;
    if (g.pool == 2) e = launch_k(conv_win_kernel<1, 0>, grid, block, smem, st, tma, wa);
    else if (ya) e = launch_k(conv_win_kernel<0, 1>, grid, block, smem, st, tma, wa);
    else e = launch_k(conv_win_kernel<0, 0>, grid, block, smem, st, tma, wa);
  } else if (path == IFQ_PATH_TC) {
    int bn = choose_bn(g, d->cout, nsm), ks = 1;
    const int gb = granule_bytes(d, g);
    if (gb == 16) {
      if (g.sbi == 2) choose_split<16, 2, 2>(g, d->cout, nsm, &bn, &ks);
      else if (g.sb == 4) choose_split<16, 4, 4>(g, d->cout, nsm, &bn, &ks);
      else choose_split<16, 4, 2>(g, d->cout, nsm, &bn, &ks);
    }
    ConvArgs a;
    fill_conv_args(d, g, bn, x, thr, sign, yc, ya, &a);
    a.early = early ? 1 : 0;
    a.wbits = g.in8 ? nullptr : (const uint8_t*)w_prep + prep_pbits_offset(d, g);
    // Filter tiles expanded from sign bits in shared memory (the split instance only, its TMA warp
    // streaming the bits): opt-in.  It reads 1 bit per weight from DRAM instead of an e4m3 byte, but
    // on AlexNet's FC layers (b128) it measured 22.4 / 16.3 us against 20.6 / 16.4 us for FC6 / FC7:
    // those single-tile launches are bound by the K-stage pipeline's latency, not by the filter
    // stream.  IFQ_TC_BX = 1 takes it where the filters are read about once (at most two 128-row
    // tiles), 2 wherever the split instance runs.
    const int bx_env = env_int("IFQ_TC_BX", 0);
    const bool bx = bx_env != 0 && (bx_env == 2 || ceil_div(g.M, kBM) <= 2) && bn == 64 && ks == 2 && gb == 16 &&
                    g.sbi == 2 && g.sb == 2;
    CUtensorMap tm;
    if (!(bx ? encode_bitmap(d, g, w_prep, bn, &tm) : encode_wmap(d, g, w_prep, bn, &tm))) return IFQ_ECUDA;
    if (g.sbi == 2 && g.sb == 2) {
      if (gb == 16) e = launch_tc_gb<16, 2, 2>(bn, ks, tm, a, nsm, st, bx);
      else if (gb == 8) e = launch_tc_gb<8, 2, 2>(bn, ks, tm, a, nsm, st);
      else if (gb == 4) e = launch_tc_gb<4, 2, 2>(bn, ks, tm, a, nsm, st);
      else e = launch_tc_gb<1, 2, 2>(bn, ks, tm, a, nsm, st);
    } else if (g.sb == 4) {
      if (gb == 16) e = launch_tc_gb<16, 4, 4>(bn, ks, tm, a, nsm, st);
      else if (gb == 8) e = launch_tc_gb<8, 4, 4>(bn, ks, tm, a, nsm, st);
      else e = launch_tc_gb<4, 4, 4>(bn, ks, tm, a, nsm, st);
    } else {   // 8-bit input values, 2-bit output codes
      if (gb == 16) e = launch_tc_gb<16, 4, 2>(bn, ks, tm, a, nsm, st);
      else if (gb == 8) e = launch_tc_gb<8, 4, 2>(bn, ks, tm, a, nsm, st);
      else e = launch_tc_gb<4, 4, 2>(bn, ks, tm, a, nsm, st);
    }
  } else if (narrow_supported(d, g)) {
    NarrowArgs a;
    a.x = (const uint8_t*)x;
    a.wbits = (const uint32_t*)((const uint8_t*)w_prep + prep_bits_offset(d, g));
    a.thr = thr;
    a.sign = sign;
    a.y_codes = yc;
    a.y_acc = ya;
    a.n = d->n; a.h = d->h; a.w = d->w; a.cout = d->cout; a.pad = d->pad;
    a.ho = g.ho; a.wo = g.wo; a.pho = g.pho; a.pwo = g.pwo; a.kwords = g.kwords;
    a.total = d->n * g.pho * g.pwo;
    a.div_pwo = make_fastdiv((uint32_t)g.pwo);
    a.div_pho = make_fastdiv((uint32_t)g.pho);
    const dim3 grid(launch_1d_blocks((size_t)a.total, kNarrowThreads, nsm)), block(kNarrowThreads);
    e = launch_narrow(d->cin, g.pool, d->cout, grid, block, a, st);
  } else {
    BsArgs a;
    a.x = (const uint8_t*)x;
    a.wbits = (const uint32_t*)((const uint8_t*)w_prep + prep_bits_offset(d, g));
    a.thr = thr;
    a.sign = sign;
    a.y_codes = yc;
    a.y_acc = ya;
    a.n = d->n; a.h = d->h; a.w = d->w; a.cin = d->cin; a.cout = d->cout;
    a.kh = d->kh; a.kw = d->kw; a.stride = d->stride; a.pad = d->pad; a.ho = g.ho; a.wo = g.wo;
    a.M = g.M;
    a.K = g.K;
    a.kwords = g.kwords;
    a.lvl = g.lvl;
    dim3 grid(ceil_div(g.M, kBsTM), ceil_div(d->cout, kBsTN));
    if (g.sb == 2) e = launch_k(conv_bitserial_kernel<2>, grid, dim3(kBsThreads), 0, st, a);
    else e = launch_k(conv_bitserial_kernel<4>, grid, dim3(kBsThreads), 0, st, a);
  }
  return e == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int check_pool(const ifq_pool_desc* d, int* ho, int* wo, int* sb = nullptr) {
  int rc = ifq_pool_out_shape(d, ho, wo);
  if (rc) return rc;
  int k, f, lvl;
  if ((rc = code_width(d->kbits, &k, &f, &lvl))) return rc;
  if (sb) *sb = f;
  if (d->c % 4 != 0 || d->pad >= d->k) return IFQ_ESHAPE;
  if ((long long)d->n * d->h * d->w * d->c >= (1LL << 40)) return IFQ_ERANGE;
  // the pool kernels index output bytes of codes with 32-bit integers
  if ((long long)d->n * *ho * *wo * (d->c * f / 8) >= (1LL << 31)) return IFQ_ERANGE;
  return IFQ_OK;
}

// The word-vector pool kernel for U words per item, field width sb and window k (k = 2, 3 have
// their own instances that load the whole window first).
template <int U, int SB>
cudaError_t launch_pool_u(int k, dim3 grid, const PoolArgs& a, cudaStream_t st) {
  if (k == 2) return launch_k(maxpool_codes_kernel<U, SB, 2>, grid, dim3(256), 0, st, a);
  if (k == 3) return launch_k(maxpool_codes_kernel<U, SB, 3>, grid, dim3(256), 0, st, a);
  return launch_k(maxpool_codes_kernel<U, SB, 0>, grid, dim3(256), 0, st, a);
}

cudaError_t launch_pool_words(int U, int sb, int k, dim3 grid, const PoolArgs& a, cudaStream_t st) {
  if (sb == 2) {
    if (U == 4) return launch_pool_u<4, 2>(k, grid, a, st);
    if (U == 2) return launch_pool_u<2, 2>(k, grid, a, st);
    return launch_pool_u<1, 2>(k, grid, a, st);
  }
  if (U == 4) return launch_pool_u<4, 4>(k, grid, a, st);
  if (U == 2) return launch_pool_u<2, 4>(k, grid, a, st);
  return launch_pool_u<1, 4>(k, grid, a, st);
}

int run_pool(const ifq_pool_desc* d, const void* x, const int8_t* sign, void* y, cudaStream_t st) {
  int ho, wo, sb;
  int rc = check_pool(d, &ho, &wo, &sb);
  if (rc) return rc;
  if (!x || !y) return IFQ_EINVAL;
  if (!aligned16(x) || !aligned16(y)) return IFQ_EALIGN;
  if (d->n == 0) return IFQ_OK;   // an empty batch
  int nsm = 0;
  if ((rc = ensure_init(&nsm))) return rc;
  PoolArgs a;
  a.x = (const uint8_t*)x;
  a.sign = sign;
  a.y = (uint8_t*)y;
  a.n = d->n; a.h = d->h; a.w = d->w; a.c = d->c; a.k = d->k; a.stride = d->stride; a.pad = d->pad;
  a.ho = ho; a.wo = wo;
  const size_t pix = (size_t)d->n * ho * wo;
  const int pb = d->c * sb / 8;   // packed bytes per pixel
  // one vector of 16, 8 or 4 bytes (else one byte) of a pixel per item
  const int vb = pb % 16 == 0 ? 16 : (pb % 8 == 0 ? 8 : (pb % 4 == 0 ? 4 : 1));
  a.groups = pb / vb;
  a.total = (int)(pix * a.groups);
  a.div_groups = make_fastdiv((uint32_t)a.groups);
  a.div_wo = make_fastdiv((uint32_t)wo);
  a.div_ho = make_fastdiv((uint32_t)ho);
  // 2x2 / stride 2 without padding on 4- or 8-byte pixels: whole 16-byte row segments per item
  const int kp = pb == 4 ? 2 : 1;
  if (d->k == 2 && d->stride == 2 && d->pad == 0 && (pb == 4 || pb == 8) && ((size_t)d->w * pb) % 16 == 0 &&
      wo % kp == 0) {
    a.wq = wo / kp;
    a.div_wq = make_fastdiv((uint32_t)a.wq);
    a.total = (int)((size_t)d->n * ho * a.wq);
    const dim3 grid(launch_1d_blocks((size_t)a.total, 256, nsm));
    cudaError_t e;
    if (sb == 2) e = pb == 4 ? launch_k(maxpool2x2_rowpair_kernel<2, 4>, grid, dim3(256), 0, st, a)
                             : launch_k(maxpool2x2_rowpair_kernel<2, 8>, grid, dim3(256), 0, st, a);
    else e = pb == 4 ? launch_k(maxpool2x2_rowpair_kernel<4, 4>, grid, dim3(256), 0, st, a)
                     : launch_k(maxpool2x2_rowpair_kernel<4, 8>, grid, dim3(256), 0, st, a);
    return e == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
  }
  const dim3 b256(256), grid(launch_1d_blocks((size_t)a.total, 256, nsm));
  cudaError_t e;
  if (vb >= 4)
    e = launch_pool_words(vb / 4, sb, d->k, grid, a, st);
  else
    e = sb == 2 ? launch_k(maxpool_codes_bytes_kernel<2>, grid, b256, 0, st, a)
                : launch_k(maxpool_codes_bytes_kernel<4>, grid, b256, 0, st, a);
  return e == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int check_fixed(int rows, int cout, int m) {
  if (rows < 0 || cout < 1 || m < 1 || m > 24) return IFQ_EINVAL;
  if ((long long)rows * cout >= (1LL << 31)) return IFQ_ERANGE;
  return IFQ_OK;
}

int run_fixed(const int32_t* acc, int rows, int cout, const int64_t* mul, const int64_t* add, int m, int32_t* y,
              cudaStream_t st) {
  int rc = check_fixed(rows, cout, m);
  if (rc) return rc;
  if (!acc || !mul || !add || !y) return IFQ_EINVAL;
  if (((uintptr_t)acc & 3u) || ((uintptr_t)y & 3u) || ((uintptr_t)mul & 7u) || ((uintptr_t)add & 7u)) return IFQ_EALIGN;
  if (rows == 0) return IFQ_OK;
  int nsm = 0;
  if ((rc = ensure_init(&nsm))) return rc;
  const int total = rows * cout;
  const cudaError_t e = launch_k(fixed_output_kernel, dim3(launch_1d_blocks((size_t)total, 256, nsm)), dim3(256), 0,
                                 st, acc, total, make_fastdiv((uint32_t)cout), mul, add, m, y);
  return e == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

// Output shape (n, h, w, c) of a layer, whether it produces codes, and their width k (a layer's
// input codes and its output codes have the same width).  A fixed-point output layer has its
// source conv's shape and no codes.
int layer_out(const ifq_layer* layers, int i, int* n, int* h, int* w, int* c, bool* codes, int* kb) {
  const ifq_layer& l = layers[i];
  if (l.kind == IFQ_LAYER_FIXED) {
    if (l.src < 0 || l.src >= i || layers[l.src].kind != IFQ_LAYER_CONV) return IFQ_EINVAL;
    int rc = layer_out(layers, l.src, n, h, w, c, codes, kb);
    if (rc) return rc;
    if (!(layers[l.src].conv.out_mode & IFQ_OUT_ACC)) return IFQ_ESHAPE;
    if ((rc = check_fixed(*n * *h * *w, *c, l.fixed.m))) return rc;
    *codes = false;
    return IFQ_OK;
  }
  if (l.kind == IFQ_LAYER_CONV) {
    ConvGeom g;
    int rc = check_conv(&l.conv, &g);
    if (rc) return rc;
    *n = l.conv.n; *h = g.pho; *w = g.pwo; *c = l.conv.cout;
    *codes = (l.conv.out_mode & IFQ_OUT_CODES) != 0;
    *kb = g.kb;
    return IFQ_OK;
  }
  if (l.kind == IFQ_LAYER_POOL) {
    int ho, wo;
    int rc = check_pool(&l.pool, &ho, &wo);
    if (rc) return rc;
    *n = l.pool.n; *h = ho; *w = wo; *c = l.pool.c;
    *codes = true;
    *kb = l.pool.kbits == 0 ? 2 : l.pool.kbits;
    return IFQ_OK;
  }
  return IFQ_EINVAL;
}

int check_stack(const ifq_layer* layers, int nlayers, const void* x) {
  if (!layers || nlayers < 1 || !x) return IFQ_EINVAL;
  for (int i = 0; i < nlayers; ++i) {
    const ifq_layer& l = layers[i];
    int n, h, w, c, kb;
    bool codes;
    if (l.src < -1 || l.src >= i) return IFQ_EINVAL;
    int rc = layer_out(layers, i, &n, &h, &w, &c, &codes, &kb);
    if (rc) return rc;
    if (l.kind == IFQ_LAYER_FIXED) continue;   // reads its source conv's accumulators (checked above)
    if (l.src >= 0) {
      int sn, sh, sw, sc, skb;
      bool sc_codes;
      layer_out(layers, l.src, &sn, &sh, &sw, &sc, &sc_codes, &skb);
      // the width a layer reads: its code width, or 8 for a layer on 8-bit input values
      const int in_kb = l.kind == IFQ_LAYER_CONV && l.conv.in_bits == 8 ? 8 : kb;
      if (!sc_codes || skb != in_kb) return IFQ_ESHAPE;
      const int in_n = l.kind == IFQ_LAYER_CONV ? l.conv.n : l.pool.n;
      const int in_h = l.kind == IFQ_LAYER_CONV ? l.conv.h : l.pool.h;
      const int in_w = l.kind == IFQ_LAYER_CONV ? l.conv.w : l.pool.w;
      const int in_c = l.kind == IFQ_LAYER_CONV ? l.conv.cin : l.pool.c;
      if (in_n != sn || in_h != sh || in_w != sw || in_c != sc) return IFQ_ESHAPE;
    }
  }
  return IFQ_OK;
}

// Completion counters of the persistent stack kernel: one per 128-row block of every layer.
size_t stack_counters(const ifq_layer* layers, int nlayers) {
  size_t n = 0;
  for (int i = 0; i < nlayers; ++i) {
    ConvGeom g;
    check_conv(&layers[i].conv, &g);
    n += (size_t)ceil_div(g.M, kBM);
  }
  return n;
}

// Whether a (validated) stack can run as one persistent launch: conv layers only, each on the
// tensor-core path, at most kMaxStackLayers, K tables that fit in shared memory.  `bytes` gets
// the workspace it needs (the completion counters).
bool stack_eligible(const ifq_layer* layers, int nlayers, size_t* bytes) {
  if (nlayers < 1 || nlayers > kMaxStackLayers) return false;
  int tab = 0;
  for (int i = 0; i < nlayers; ++i) {
    if (layers[i].kind != IFQ_LAYER_CONV) return false;
    ConvGeom g;
    if (check_conv(&layers[i].conv, &g)) return false;
    if (g.pool > 1 || g.kb != 2 || g.in8) return false;   // the persistent kernel: 2-bit codes, no fused pool
    if (g.M == 0) return false;                           // an empty batch runs (as nothing) layer by layer
    // the persistent kernel computes every layer with the tensor-core data path: layers whose own
    // launch would take that path or the window path qualify
    const int p = choose_path(&layers[i].conv, g);
    if (!(p == IFQ_PATH_TC || ((p == IFQ_PATH_WIN || p == IFQ_PATH_WARP) && tc_supported(&layers[i].conv, g))))
      return false;
    tab += g.Kpad / (4 * granule_bytes(&layers[i].conv, g, true));
  }
  if (tab > kMaxStackTab) return false;
  if (bytes) *bytes = round_up(stack_counters(layers, nlayers) * sizeof(unsigned int), 256);
  return true;
}

// The persistent stack kernel is opt-in (IFQ_STACK=1, read on every call): on the stacks
// measured so far one launch per layer, chained with programmatic dependent launch, is faster.
bool stack_enabled() {
  const char* v = getenv("IFQ_STACK");
  return v && v[0] == '1';
}

// The persistent stack kernel orders a layer only after the layer it reads, so it needs every
// buffer a layer writes to be disjoint from every other buffer of the stack (input, weights,
// thresholds, signs, other outputs, counters).  Stacks that reuse buffers run layer by layer,
// where stream order makes reuse safe.
struct Span { uintptr_t lo, hi; bool written; };

bool stack_buffers_disjoint(const ifq_layer* layers, int nlayers, const void* x, const void* ws, size_t ws_bytes) {
  std::vector<Span> v;
  auto add = [&](const void* p, size_t n, bool wr) {
    if (p && n) v.push_back({(uintptr_t)p, (uintptr_t)p + n, wr});
  };
  size_t x_bytes = 0;
  for (int i = 0; i < nlayers; ++i)
    if (layers[i].src < 0) {
      const ifq_conv_desc& d = layers[i].conv;
      x_bytes = std::max(x_bytes, (size_t)d.n * d.h * d.w * d.cin / 4);
    }
  add(x, x_bytes, false);
  add(ws, ws_bytes, true);
  for (int i = 0; i < nlayers; ++i) {
    const ifq_conv_desc& d = layers[i].conv;
    ConvGeom g;
    check_conv(&d, &g);
    const size_t rows = (size_t)d.n * g.pho * g.pwo;
    add(layers[i].w_prep, prep_bits_offset(&d, g) + (size_t)d.cout * g.kwords * 4, false);
    if (d.out_mode & IFQ_OUT_CODES) {
      add(layers[i].thr, (size_t)d.cout * 3 * 4, false);
      add(layers[i].sign, (size_t)d.cout, false);
      add(layers[i].y_codes, rows * d.cout / 4, true);
    }
    if (d.out_mode & IFQ_OUT_ACC) add(layers[i].y_acc, rows * d.cout * 4, true);
  }
  for (size_t i = 0; i < v.size(); ++i)
    for (size_t j = i + 1; j < v.size(); ++j)
      if ((v[i].written || v[j].written) && v[i].lo < v[j].hi && v[j].lo < v[i].hi) return false;
  return true;
}

int launch_stack_kernel(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t need,
                        cudaStream_t st);

int run_stack_kernel(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes,
                     cudaStream_t st) {
  size_t need = 0;
  if (!stack_enabled() || !stack_eligible(layers, nlayers, &need) || !ws || ws_bytes < need) return IFQ_EUNSUPPORTED;
  return launch_stack_kernel(layers, nlayers, x, ws, need, st);
}

// The launch itself, for an eligible stack with `need` bytes of counters at ws.
int launch_stack_kernel(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t need,
                        cudaStream_t st) {
  int nsm = 0;
  bool ok = false;
  int rc = ensure_init(&nsm, &ok);
  if (rc) return rc;
  if (!ok) return IFQ_EUNSUPPORTED;
  if (!stack_buffers_disjoint(layers, nlayers, x, ws, need)) return IFQ_EUNSUPPORTED;
  for (int i = 0; i < nlayers; ++i) {
    const ifq_layer& l = layers[i];
    const void* in = l.src < 0 ? x : layers[l.src].y_codes;
    if (!in || !l.w_prep || !aligned16(in) || !aligned16(l.w_prep)) return IFQ_EUNSUPPORTED;
    if ((l.conv.out_mode & IFQ_OUT_CODES) && (!l.y_codes || !l.thr || !l.sign || !aligned16(l.y_codes)))
      return IFQ_EUNSUPPORTED;
    if ((l.conv.out_mode & IFQ_OUT_ACC) && (!l.y_acc || !aligned16(l.y_acc))) return IFQ_EUNSUPPORTED;
  }
  StackParams P;
  memset(&P, 0, sizeof(P));
  P.nlayers = nlayers;
  P.cnt = (unsigned int*)ws;
  int tab = 0, cnt = 0;
  for (int i = 0; i < nlayers; ++i) {
    const ifq_layer& l = layers[i];
    ConvGeom g;
    check_conv(&l.conv, &g);
    const int bn = choose_bn(g, l.conv.cout, nsm);
    if (!encode_wmap(&l.conv, g, l.w_prep, bn, &P.tm[i])) return IFQ_ECUDA;
    uint8_t* yc = (l.conv.out_mode & IFQ_OUT_CODES) ? (uint8_t*)l.y_codes : nullptr;
    int32_t* ya = (l.conv.out_mode & IFQ_OUT_ACC) ? l.y_acc : nullptr;
    StackLayer& S = P.L[i];
    fill_conv_args(&l.conv, g, bn, l.src < 0 ? x : layers[l.src].y_codes, l.thr, l.sign, yc, ya, &S.a, true);
    S.bn = bn;
    S.gb = granule_bytes(&l.conv, g, true);
    S.tab_off = tab;
    S.dep = l.src;
    S.cnt_off = cnt;
    tab += S.a.ntab;
    cnt += ceil_div(g.M, kBM);
  }
  if (cudaMemsetAsync(ws, 0, need, st) != cudaSuccess) return IFQ_ECUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(nsm);
  cfg.blockDim = dim3(kStackThreads);
  cfg.dynamicSmemBytes = StackSmem::bytes;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, conv_stack_kernel, P) == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

// Counter scratch of ifq_forward_noalloc.  That entry point serves callers that cannot hand
// the library device scratch (a plain C host without a device allocator, or a serving loop that
// must not call cudaMalloc, which can synchronize the whole device), so its counters live in a
// file-scope device array instead of a caller's workspace: 65536 counters, one per 128-row
// output block, enough for the ResNet-18 body at batch 256.
constexpr size_t kNoallocCounterBytes = 256 * 1024;
static __device__ __align__(256) unsigned int g_noalloc_counters[kNoallocCounterBytes / sizeof(unsigned int)];
void* g_noalloc_addr[kMaxDevices];   // device address of g_noalloc_counters per device (g_dev_mu)

// Device address of the counter array on the current device: looked up once per device, with
// that device current (cudaGetSymbolAddress allocates nothing).
int noalloc_counters(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return IFQ_ECUDA;
  std::lock_guard<std::mutex> lk(g_dev_mu);
  if (!g_noalloc_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_counters) != cudaSuccess || !p) return IFQ_ECUDA;
    g_noalloc_addr[dev] = p;
  }
  *out = g_noalloc_addr[dev];
  return IFQ_OK;
}

// Launch mode of this host thread's last successful ifq_forward / ifq_forward_noalloc (0: none yet).
thread_local int t_last_forward = 0;

int note_forward(int rc, int mode) {
  if (rc == IFQ_OK) t_last_forward = mode;
  return rc;
}

int run_layer(const ifq_layer* layers, int i, const void* x, cudaStream_t st) {
  const ifq_layer& l = layers[i];
  const void* in = l.src < 0 ? x : layers[l.src].y_codes;
  // every kernel of a stack before layer i is a layer of the stack or a copy of its input or results
  if (l.kind == IFQ_LAYER_CONV) return run_conv(&l.conv, in, l.w_prep, l.thr, l.sign, l.y_codes, l.y_acc, st, i > 0);
  if (l.kind == IFQ_LAYER_POOL) return run_pool(&l.pool, in, l.sign, l.y_codes, st);
  const ifq_layer& sl = layers[l.src];
  ConvGeom g;
  int rc = check_conv(&sl.conv, &g);
  if (rc) return rc;
  return run_fixed(sl.y_acc, sl.conv.n * g.pho * g.pwo, sl.conv.cout, l.fx_mul, l.fx_add, l.fixed.m, l.y_acc, st);
}

int run_stack(const ifq_layer* layers, int nlayers, const void* x, cudaStream_t st) {
  for (int i = 0; i < nlayers; ++i) {
    const int rc = run_layer(layers, i, x, st);
    if (rc) return rc;
  }
  return IFQ_OK;
}

// Whether the device addresses p directly at the same address: device or managed memory, or
// pinned host memory under unified addressing.
bool device_addressable(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();   // an unregistered pointer is not an error to keep
    return false;
  }
  if (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) return true;
  return at.type == cudaMemoryTypeHost && at.devicePointer == p;
}

// One copy of a graph's input or of a layer's result; `sm`: on the SMs (copy16_kernel), else
// cudaMemcpyAsync.
struct IoCopy {
  void* dst;
  const void* src;
  size_t bytes;
  bool sm;
};

IoCopy make_copy(void* dst, const void* src, size_t n) {
  const bool sm = aligned16(dst) && aligned16(src) && n % 16 == 0 && device_addressable(dst) && device_addressable(src);
  return IoCopy{dst, src, n, sm};
}

int enqueue_copy(const IoCopy& c, int nsm, cudaStream_t st) {
  if (c.bytes == 0) return IFQ_OK;
  if (!c.sm) return cudaMemcpyAsync(c.dst, c.src, c.bytes, cudaMemcpyDefault, st) == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
  const size_t n16 = c.bytes / 16;
  size_t blocks = (n16 + 255) / 256;
  if (blocks > (size_t)nsm * 8) blocks = (size_t)nsm * 8;
  return launch_k(copy16_kernel, dim3((unsigned)blocks), dim3(256), 0, st, (const uint4*)c.src, (uint4*)c.dst, n16) ==
                 cudaSuccess
             ? IFQ_OK
             : IFQ_ECUDA;
}

// The copies a graph makes around the stack: the input before the first layer, and after layer
// i the results of layer i.
struct IoPlan {
  IoCopy in{nullptr, nullptr, 0, false};
  std::vector<std::vector<IoCopy>> after;
  int nsm = 0;
  int copies_after(int i, cudaStream_t st) const {
    if (after.empty()) return IFQ_OK;
    for (const IoCopy& c : after[i]) {
      const int rc = enqueue_copy(c, nsm, st);
      if (rc) return rc;
    }
    return IFQ_OK;
  }
};

// Bytes of layer i's code and accumulator buffers (0 where it has none).
int layer_buffer_bytes(const ifq_layer* layers, int i, size_t* codes, size_t* acc) {
  int n, h, w, c, kb;
  bool has_codes;
  const int rc = layer_out(layers, i, &n, &h, &w, &c, &has_codes, &kb);
  if (rc) return rc;
  int k, f, lvl;
  if (code_width(kb, &k, &f, &lvl)) f = 2;
  const size_t px = (size_t)n * h * w;
  const ifq_layer& l = layers[i];
  *codes = has_codes ? px * c * f / 8 : 0;
  *acc = (l.kind == IFQ_LAYER_FIXED || (l.kind == IFQ_LAYER_CONV && (l.conv.out_mode & IFQ_OUT_ACC))) ? px * c * 4 : 0;
  return IFQ_OK;
}

// Bytes of packed input read by the layers with src = -1 (they must agree).
int stack_input_bytes(const ifq_layer* layers, int nlayers, size_t* bytes) {
  *bytes = 0;
  for (int i = 0; i < nlayers; ++i) {
    const ifq_layer& l = layers[i];
    if (l.src >= 0 || l.kind == IFQ_LAYER_FIXED) continue;
    size_t b;
    if (l.kind == IFQ_LAYER_CONV) {
      ConvGeom g;
      const int rc = check_conv(&l.conv, &g);
      if (rc) return rc;
      b = (size_t)l.conv.n * l.conv.h * l.conv.w * pixel_bytes(&l.conv, g);
    } else {
      int k, f, lvl;
      const int rc = code_width(l.pool.kbits, &k, &f, &lvl);
      if (rc) return rc;
      b = (size_t)l.pool.n * l.pool.h * l.pool.w * l.pool.c * f / 8;
    }
    if (*bytes && *bytes != b) return IFQ_ESHAPE;
    *bytes = b;
  }
  return IFQ_OK;
}

// Stream capture of a stack with its side branches: a layer whose output no later layer reads (a
// ResNet shortcut conv), other than the last, does not hold up the layers after it, so it runs on a
// second stream that forks from the main stream when its source layer has run and joins it at the
// end.  The graph then lets it overlap the main chain, on SMs that under-filled layers leave idle.
// Outputs are the same; only the graph's edges differ.  The streams and events live until the
// capture has ended (release()).
struct BranchedCapture {
  cudaStream_t side = nullptr;
  std::vector<cudaEvent_t> events;

  int run(const ifq_layer* layers, int nlayers, const void* x, cudaStream_t main, const IoPlan& io) {
    int rc;
    if ((rc = enqueue_copy(io.in, io.nsm, main))) return rc;
    std::vector<char> read(nlayers, 0);
    for (int i = 0; i < nlayers; ++i)
      if (layers[i].src >= 0) read[layers[i].src] = 1;
    std::vector<char> is_side(nlayers, 0);
    int nside = 0;
    for (int i = 0; i + 1 < nlayers; ++i)
      if (!read[i]) is_side[i] = 1, ++nside;
    const char* v = getenv("IFQ_GRAPH_BRANCH");
    if (nside == 0 || (v && v[0] == '0')) {
      for (int i = 0; i < nlayers; ++i)
        if ((rc = run_layer(layers, i, x, main)) || (rc = io.copies_after(i, main))) return rc;
      return IFQ_OK;
    }
    if (cudaStreamCreateWithFlags(&side, cudaStreamNonBlocking) != cudaSuccess) return IFQ_ECUDA;
    auto fork = [&](int s) -> int {   // side layer s after everything issued so far on main
      cudaEvent_t e;
      if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return IFQ_ECUDA;
      events.push_back(e);
      if (cudaEventRecord(e, main) != cudaSuccess || cudaStreamWaitEvent(side, e, 0) != cudaSuccess) return IFQ_ECUDA;
      const int r = run_layer(layers, s, x, side);
      return r ? r : io.copies_after(s, side);
    };
    for (int s = 0; s < nlayers; ++s)   // side layers on the stack input fork before anything runs
      if (is_side[s] && layers[s].src < 0 && (rc = fork(s))) return rc;
    for (int i = 0; i < nlayers; ++i) {
      if (is_side[i]) continue;
      if ((rc = run_layer(layers, i, x, main)) || (rc = io.copies_after(i, main))) return rc;
      for (int s = i + 1; s < nlayers; ++s)
        if (is_side[s] && layers[s].src == i && (rc = fork(s))) return rc;
    }
    cudaEvent_t join;
    if (cudaEventCreateWithFlags(&join, cudaEventDisableTiming) != cudaSuccess) return IFQ_ECUDA;
    events.push_back(join);
    if (cudaEventRecord(join, side) != cudaSuccess || cudaStreamWaitEvent(main, join, 0) != cudaSuccess)
      return IFQ_ECUDA;
    return IFQ_OK;
  }

  void release() {
    for (cudaEvent_t e : events) cudaEventDestroy(e);
    events.clear();
    if (side) cudaStreamDestroy(side);
    side = nullptr;
  }
};

}  // namespace

struct ifq_graph {
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
};

extern "C" {

int ifq_weights_prep_bytes(const ifq_conv_desc* d, size_t* bytes) {
  ConvGeom g;
  if (!bytes) return IFQ_EINVAL;
  int rc = check_conv(d, &g);
  if (rc) return rc;
  *bytes = prep_bytes(d, g);
  return IFQ_OK;
}

int ifq_pack_weights(const ifq_conv_desc* d, const uint32_t* w_bits, void* w_prep, void* stream) {
  ConvGeom g;
  int rc = check_conv(d, &g);
  if (rc) return rc;
  if (!w_bits || !w_prep) return IFQ_EINVAL;
  if (!aligned16(w_prep) || ((uintptr_t)w_bits & 3u)) return IFQ_EALIGN;
  int nsm = 0;
  if ((rc = ensure_init(&nsm))) return rc;
  uint8_t* base = (uint8_t*)w_prep;
  const int blocks = launch_1d_blocks((size_t)d->cout * (g.Kpad / 4), 256, nsm);
  prep_weights_kernel<<<blocks, 256, 0, S(stream)>>>(
      w_bits, base, (uint32_t*)(base + prep_bits_offset(d, g)),
      g.in8 ? nullptr : (uint32_t*)(base + prep_pbits_offset(d, g)), d->cout, g.Kk, g.Kpad, g.kwords, 32 / g.sbi,
      g.in8 ? 1 : 0);
  if (g.in8)
    prep_direct_masks_kernel<<<launch_1d_blocks((size_t)g.K, 256, nsm), 256, 0, S(stream)>>>(
        (const uint32_t*)(base + prep_bits_offset(d, g)), (uint32_t*)(base + prep_masks_offset(d, g)), d->cout, g.K,
        g.kwords);
  return cudaGetLastError() == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int ifq_conv_plan(const ifq_conv_desc* d, int* path) {
  ConvGeom g;
  if (!path) return IFQ_EINVAL;
  int rc = check_conv(d, &g);
  if (rc) return rc;
  const int p = choose_path(d, g);
  if (p < 0) return IFQ_EUNSUPPORTED;
  *path = p;
  return IFQ_OK;
}

int ifq_conv_workspace_bytes(const ifq_conv_desc* d, size_t* bytes) {
  ConvGeom g;
  if (!bytes) return IFQ_EINVAL;
  int rc = check_conv(d, &g);
  if (rc) return rc;
  *bytes = 0;
  return IFQ_OK;
}

int ifq_conv2bit(const ifq_conv_desc* d, const void* x, const void* w_prep, const int32_t* thr, const int8_t* sign,
                 void* y_codes, int32_t* y_acc, void* ws, size_t ws_bytes, void* stream) {
  (void)ws;
  (void)ws_bytes;
  return run_conv(d, x, w_prep, thr, sign, y_codes, y_acc, S(stream));
}

int ifq_maxpool2bit(const ifq_pool_desc* d, const void* x, const int8_t* sign, void* y, void* stream) {
  return run_pool(d, x, sign, y, S(stream));
}

int ifq_forward_workspace_bytes(const ifq_layer* layers, int nlayers, size_t* bytes) {
  if (!layers || nlayers < 1 || !bytes) return IFQ_EINVAL;
  size_t need = 0;
  *bytes = stack_enabled() && stack_eligible(layers, nlayers, &need) ? need : 0;
  return IFQ_OK;
}

int ifq_forward(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes, void* stream) {
  int rc = check_stack(layers, nlayers, x);
  if (rc) return rc;
  rc = run_stack_kernel(layers, nlayers, x, ws, ws_bytes, S(stream));
  if (rc != IFQ_EUNSUPPORTED) return note_forward(rc, IFQ_FORWARD_PERSISTENT);
  return note_forward(run_stack(layers, nlayers, x, S(stream)), IFQ_FORWARD_LAYERS);
}

int ifq_forward_noalloc(const ifq_layer* layers, int nlayers, const void* x, void* stream) {
  int rc = check_stack(layers, nlayers, x);
  if (rc) return rc;
  size_t need = 0;
  if (!stack_eligible(layers, nlayers, &need))
    return note_forward(run_stack(layers, nlayers, x, S(stream)), IFQ_FORWARD_LAYERS);
  if (need > kNoallocCounterBytes) return IFQ_EWORKSPACE;
  void* ws = nullptr;
  if ((rc = noalloc_counters(&ws))) return rc;
  rc = launch_stack_kernel(layers, nlayers, x, ws, need, S(stream));
  if (rc != IFQ_EUNSUPPORTED) return note_forward(rc, IFQ_FORWARD_PERSISTENT);
  return note_forward(run_stack(layers, nlayers, x, S(stream)), IFQ_FORWARD_LAYERS);
}

int ifq_last_forward_mode(int* mode) {
  if (!mode || t_last_forward == 0) return IFQ_EINVAL;
  *mode = t_last_forward;
  return IFQ_OK;
}

}  // extern "C"

namespace {

int graph_create(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes, const IoPlan& io,
                 void* stream, ifq_graph** out) {
  cudaStream_t cap = S(stream);
  bool own = false;
  if (cap == nullptr) {
    if (cudaStreamCreateWithFlags(&cap, cudaStreamNonBlocking) != cudaSuccess) return IFQ_ECUDA;
    own = true;
  }
  ifq_graph* g = new ifq_graph();
  int rc = IFQ_OK;
  if (cudaStreamBeginCapture(cap, cudaStreamCaptureModeThreadLocal) != cudaSuccess) rc = IFQ_ECUDA;
  if (!rc) {
    BranchedCapture bc;
    int frc = enqueue_copy(io.in, io.nsm, cap);
    if (!frc) {
      frc = run_stack_kernel(layers, nlayers, x, ws, ws_bytes, cap);
      if (!frc) {   // the whole stack in one launch: every result copy after it
        for (int i = 0; i < nlayers && !frc; ++i) frc = io.copies_after(i, cap);
      } else if (frc == IFQ_EUNSUPPORTED) {
        IoPlan rest = io;
        rest.in = IoCopy{nullptr, nullptr, 0, false};   // enqueued above
        frc = bc.run(layers, nlayers, x, cap, rest);
      }
    }
    const cudaError_t e = cudaStreamEndCapture(cap, &g->graph);
    bc.release();
    if (frc) rc = frc;
    else if (e != cudaSuccess) rc = IFQ_ECUDA;
  }
  if (!rc && cudaGraphInstantiate(&g->exec, g->graph, 0) != cudaSuccess) rc = IFQ_ECUDA;
  if (own) cudaStreamDestroy(cap);
  if (rc) {
    ifq_graph_destroy(g);
    return rc;
  }
  *out = g;
  return IFQ_OK;
}

}  // namespace

extern "C" {

int ifq_graph_create(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes, void* stream,
                     ifq_graph** out) {
  return ifq_graph_create_io(layers, nlayers, x, ws, ws_bytes, nullptr, 0, nullptr, nullptr, stream, out);
}

int ifq_graph_create_io(const ifq_layer* layers, int nlayers, const void* x, void* ws, size_t ws_bytes,
                        const void* x_src, size_t x_bytes, void* const* y_codes_dst, void* const* y_acc_dst,
                        void* stream, ifq_graph** out) {
  if (!out) return IFQ_EINVAL;
  *out = nullptr;
  int rc = check_stack(layers, nlayers, x);
  if (rc) return rc;
  int nsm = 0;
  if ((rc = ensure_init(&nsm))) return rc;
  if (!get_encode()) return IFQ_ECUDA;
  // the copies are planned (sizes checked, device addressability looked up) before the capture
  IoPlan io;
  io.nsm = nsm;
  if (x_src) {
    size_t need = 0;
    if ((rc = stack_input_bytes(layers, nlayers, &need))) return rc;
    if (x_bytes != need) return IFQ_ESHAPE;
    io.in = make_copy(const_cast<void*>(x), x_src, x_bytes);
  }
  if (y_codes_dst || y_acc_dst) {
    io.after.resize(nlayers);
    for (int i = 0; i < nlayers; ++i) {
      size_t cb = 0, ab = 0;
      if ((rc = layer_buffer_bytes(layers, i, &cb, &ab))) return rc;
      void* dc = y_codes_dst ? y_codes_dst[i] : nullptr;
      void* da = y_acc_dst ? y_acc_dst[i] : nullptr;
      if ((dc && (!cb || !layers[i].y_codes)) || (da && (!ab || !layers[i].y_acc))) return IFQ_EINVAL;
      if (dc) io.after[i].push_back(make_copy(dc, layers[i].y_codes, cb));
      if (da) io.after[i].push_back(make_copy(da, layers[i].y_acc, ab));
    }
  }
  return graph_create(layers, nlayers, x, ws, ws_bytes, io, stream, out);
}

int ifq_graph_launch(ifq_graph* g, void* stream) {
  if (!g || !g->exec) return IFQ_EINVAL;
  return cudaGraphLaunch(g->exec, S(stream)) == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int ifq_graph_destroy(ifq_graph* g) {
  if (!g) return IFQ_EINVAL;
  if (g->exec) cudaGraphExecDestroy(g->exec);
  if (g->graph) cudaGraphDestroy(g->graph);
  delete g;
  return IFQ_OK;
}

int ifq_pack_codes_kbits(const uint8_t* codes, void* packed, size_t n, int kbits, void* stream) {
  int k, sb, lvl, rc;
  if ((rc = code_width(kbits, &k, &sb, &lvl))) return rc;
  if (!codes || !packed || n % 4 != 0) return IFQ_EINVAL;
  if (n == 0) return IFQ_OK;
  int nsm = 0;
  if ((rc = ensure_init(&nsm))) return rc;
  const size_t nb = n * sb / 8;
  if (sb == 2) pack_codes_kernel<2><<<launch_1d_blocks(nb, 256, nsm), 256, 0, S(stream)>>>(codes, (uint8_t*)packed, nb);
  else pack_codes_kernel<4><<<launch_1d_blocks(nb, 256, nsm), 256, 0, S(stream)>>>(codes, (uint8_t*)packed, nb);
  return cudaGetLastError() == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int ifq_unpack_codes_kbits(const void* packed, uint8_t* codes, size_t n, int kbits, void* stream) {
  int k, sb, lvl, rc;
  if ((rc = code_width(kbits, &k, &sb, &lvl))) return rc;
  if (!codes || !packed || n % 4 != 0) return IFQ_EINVAL;
  if (n == 0) return IFQ_OK;
  int nsm = 0;
  if ((rc = ensure_init(&nsm))) return rc;
  const size_t nb = n * sb / 8;
  const uint8_t* p = (const uint8_t*)packed;
  if (sb == 2) unpack_codes_kernel<2><<<launch_1d_blocks(nb, 256, nsm), 256, 0, S(stream)>>>(p, codes, nb);
  else unpack_codes_kernel<4><<<launch_1d_blocks(nb, 256, nsm), 256, 0, S(stream)>>>(p, codes, nb);
  return cudaGetLastError() == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int ifq_pack_codes(const uint8_t* codes, void* packed, size_t n, void* stream) {
  return ifq_pack_codes_kbits(codes, packed, n, 2, stream);
}

int ifq_unpack_codes(const void* packed, uint8_t* codes, size_t n, void* stream) {
  return ifq_unpack_codes_kbits(packed, codes, n, 2, stream);
}

int ifq_pack_signs(const int8_t* w, uint32_t* bits, int rows, int K, void* stream) {
  if (!w || !bits || rows < 1 || K < 1) return IFQ_EINVAL;
  if ((uintptr_t)bits & 3u) return IFQ_EALIGN;
  int nsm = 0, rc;
  if ((rc = ensure_init(&nsm))) return rc;
  const int kwords = ceil_div(K, 32);
  pack_signs_kernel<<<launch_1d_blocks((size_t)rows * kwords, 256, nsm), 256, 0, S(stream)>>>(w, bits, rows, K,
                                                                                               kwords);
  return cudaGetLastError() == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int ifq_fixed_output(const int32_t* acc, int rows, int cout, const int64_t* mul, const int64_t* add, int m,
                     int32_t* y, void* stream) {
  return run_fixed(acc, rows, cout, mul, add, m, y, S(stream));
}

// Whether the device can dereference p as is: device or managed memory, or host memory that
// cudaHostAlloc / cudaHostRegister mapped at the same address (unified addressing).

int ifq_copy_bytes(void* dst, const void* src, size_t n, void* stream) {
  if ((!dst || !src) && n) return IFQ_EINVAL;
  if (n == 0) return IFQ_OK;
  if (!aligned16(dst) || !aligned16(src) || n % 16 != 0 || !device_addressable(dst) || !device_addressable(src))
    return cudaMemcpyAsync(dst, src, n, cudaMemcpyDefault, S(stream)) == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
  int nsm = 0, rc;
  if ((rc = ensure_init(&nsm))) return rc;
  const size_t n16 = n / 16;
  size_t blocks = (n16 + 255) / 256;
  if (blocks > (size_t)nsm * 8) blocks = (size_t)nsm * 8;
  const cudaError_t e = launch_k(copy16_kernel, dim3((unsigned)blocks), dim3(256), 0, S(stream), (const uint4*)src,
                                 (uint4*)dst, n16);
  return e == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int ifq_wait_selftest(int limit_us, void* stream) {
  if (limit_us < 1 || limit_us > 1000000) return IFQ_EINVAL;
  int rc;
  if ((rc = ensure_init(nullptr))) return rc;
  wait_selftest_kernel<<<1, 32, 0, S(stream)>>>((unsigned long long)limit_us * 1000ull);
  return cudaGetLastError() == cudaSuccess ? IFQ_OK : IFQ_ECUDA;
}

int ifq_device_status(void* stream, int* status) {
  if (!status) return IFQ_EINVAL;
  if (cudaStreamSynchronize(S(stream)) != cudaSuccess) return IFQ_ECUDA;
  int v = 0, zero = 0;
  if (cudaMemcpyFromSymbol(&v, ifq::g_status, sizeof(int)) != cudaSuccess) return IFQ_ECUDA;
  if (v != 0 && cudaMemcpyToSymbol(ifq::g_status, &zero, sizeof(int)) != cudaSuccess) return IFQ_ECUDA;
  *status = v;
  return IFQ_OK;
}

}  // extern "C"
