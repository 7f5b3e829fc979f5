// Instruction-rate probes that bench.py runs in the same process as its timed region, so
// that the fractions it reports use rates measured on the same GPU at the same time:
//   * tcgen05.mma.cta_group::1.kind::f8f6f4 (e4m3 x e4m3 -> f32), the instruction the
//     tensor-core conv issues, at M = 128, K = 32 and a given N;
//   * warp mma.sync.m16n8k32 s8 x s8 -> s32, the dense INT8 tensor path of sm_103a (it
//     has no tcgen05 integer MMA), the denominator of the metric's "% of dense INT8 peak".
// Not part of the library: a benchmark helper with a plain C ABI, built by
// __graft_entry__.build() into _build/libbench_rates.so.  Every wait is bounded.
#include <cuda_runtime.h>

#include <cstdint>

namespace {

__device__ int g_rate_err;

__device__ __forceinline__ uint32_t saddr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ unsigned long long now_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// Wait for an mbarrier phase, giving up (error flag set) after 2 s of wall time.
__device__ __forceinline__ void bounded_wait(uint32_t bar, uint32_t parity) {
  const unsigned long long t0 = now_ns();
  for (uint32_t i = 0; i < (1u << 26); ++i) {
    uint32_t done;
    asm volatile("{.reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p;}"
                 : "=r"(done)
                 : "r"(bar), "r"(parity)
                 : "memory");
    if (done) return;
    if ((i & 255u) == 255u && now_ns() - t0 > 2000000000ull) break;
  }
  atomicExch(&g_rate_err, 1);
}

// K-major shared-memory operand, 128-byte swizzle (8-row atoms 1024 bytes apart).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t a) {
  return (uint64_t)((a & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

constexpr int kOperandBytes = 32768;   // A: 128 rows x 128 B; B: up to 256 rows x 128 B

// One CTA per SM: one thread issues `iters` M128 x N x K32 e4m3 MMAs on operands of +1.0,
// alternating between two accumulators; the rest of the CTA waits.  a_tmem = 0: both operands in
// shared memory; a_tmem = 1 (N <= 128): A in tensor memory (columns 256..287, written by every
// warp for its lane quarter), B in shared memory, the form the tensor-core conv issues.
__global__ void __launch_bounds__(128, 1) tc_e4m3_rate_kernel(int n, int iters, int a_tmem, float* sink) {
  extern __shared__ uint8_t raw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)raw + 1023) & ~(uintptr_t)1023);
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tslot;
  const int tid = threadIdx.x, warp = tid >> 5;
  for (int i = tid; i < (128 * 128 + kOperandBytes) / 4; i += blockDim.x) ((uint32_t*)sm)[i] = 0x38383838u;
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(saddr(&tslot)) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(saddr(&bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tslot;
  if (a_tmem) {
    // A: 128 lanes x 32 columns of e4m3 +1.0 (four K = 32 steps of 8 columns)
    const uint32_t ta = tmem + 256u + ((uint32_t)(warp * 32) << 16);
    const uint32_t one = 0x38383838u;
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2};\n\t"
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%1], {%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2,%2};\n\t"
        "tcgen05.wait::st.sync.aligned;" ::"r"(ta), "r"(ta + 16u), "r"(one)
        : "memory");
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  }
  if (tid == 0) {
    const uint32_t idesc = (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
    const uint64_t ad = sw128_desc(saddr(sm)), bd = sw128_desc(saddr(sm + 128 * 128));
    if (a_tmem) {
      for (int i = 0; i < iters; ++i)
        asm volatile(
            "{.reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;}" ::"r"(
                tmem + (uint32_t)((i & 1) * 128)),
            "r"(tmem + 256u + (uint32_t)(8 * (i & 3))), "l"(bd + 2 * (i & 3)), "r"(idesc), "r"(i > 1 ? 1 : 0)
            : "memory");
    } else {
      for (int i = 0; i < iters; ++i)
        asm volatile(
            "{.reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;}" ::"r"(
                tmem + (uint32_t)((i & 1) * 256)),
            "l"(ad + 2 * (i & 3)), "l"(bd + 2 * (i & 3)), "r"(idesc), "r"(i > 1 ? 1 : 0)
            : "memory");
    }
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(saddr(&bar))
                 : "memory");
  }
  bounded_wait(saddr(&bar), 0);
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 0) {
    uint32_t r;
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];\n\ttcgen05.wait::ld.sync.aligned;"
                 : "=r"(r)
                 : "r"(tmem)
                 : "memory");
    if (tid == 0) sink[blockIdx.x] = __uint_as_float(r);
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
}

// Every warp issues 8 independent m16n8k32 s8 MMAs per iteration (enough in flight to
// saturate the pipe).
__global__ void mma_s8_rate_kernel(int iters, int* sink) {
  const int a0 = (int)threadIdx.x, a1 = a0 * 3, a2 = a0 * 5, a3 = a0 * 7, b0 = a0 * 11, b1 = a0 * 13;
  int c[8][4] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      asm volatile(
          "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
          : "+r"(c[j][0]), "+r"(c[j][1]), "+r"(c[j][2]), "+r"(c[j][3])
          : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  }
  int s = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 0x7fffffff) sink[0] = s;   // never true in practice; keeps the MMAs live
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return n;
}

}  // namespace

extern "C" {

// Dense ops per second (2 per MAC), in TOPS, of the e4m3 tcgen05 MMA at M = 128, K = 32 and
// the given N (a multiple of 16, 16..256; at most 128 with a_tmem), A in shared memory (a_tmem = 0)
// or in tensor memory (a_tmem = 1), measured over `reps` launches of `iters` MMAs per SM on
// `stream` (after one warm-up launch).  Returns 0 on success, 1 on a bad argument, 2 on a CUDA
// error, 3 if a wait ran out.
int bench_tc_e4m3_tops_a(int n, int a_tmem, int iters, int reps, void* stream, double* tops) {
  if (!tops || n < 16 || n > (a_tmem ? 128 : 256) || n % 16 || iters < 1 || reps < 1) return 1;
  const int sms = sm_count();
  if (sms < 1) return 2;
  cudaStream_t st = (cudaStream_t)stream;
  // 120 KB of shared memory keeps one CTA per SM (the kernel itself uses the first 49 KB)
  const int smem = 120 * 1024;
  float* sink = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  int rc = 2;
  if (cudaFuncSetAttribute(tc_e4m3_rate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) == cudaSuccess &&
      cudaMalloc(&sink, sizeof(float) * sms) == cudaSuccess && cudaEventCreate(&e0) == cudaSuccess &&
      cudaEventCreate(&e1) == cudaSuccess) {
    tc_e4m3_rate_kernel<<<sms, 128, smem, st>>>(n, 64, a_tmem, sink);
    cudaEventRecord(e0, st);
    for (int r = 0; r < reps; ++r) tc_e4m3_rate_kernel<<<sms, 128, smem, st>>>(n, iters, a_tmem, sink);
    cudaEventRecord(e1, st);
    float ms = 0.f;
    if (cudaEventSynchronize(e1) == cudaSuccess && cudaEventElapsedTime(&ms, e0, e1) == cudaSuccess && ms > 0.f) {
      *tops = 2.0 * sms * (double)reps * iters * 128.0 * n * 32.0 / (ms * 1e-3) / 1e12;
      int err = 0;
      cudaMemcpyFromSymbol(&err, g_rate_err, sizeof(int));
      rc = err ? 3 : 0;
    }
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (sink) cudaFree(sink);
  return rc;
}

// bench_tc_e4m3_tops_a with A in shared memory.
int bench_tc_e4m3_tops(int n, int iters, int reps, void* stream, double* tops) {
  return bench_tc_e4m3_tops_a(n, 0, iters, reps, stream, tops);
}

// Dense ops per second (2 per MAC), in TOPS, of warp mma.sync.m16n8k32 s8 x s8 -> s32 with 4
// CTAs of 8 warps per SM, each warp issuing 8 independent MMAs per iteration.  Same return
// codes as bench_tc_e4m3_tops.
int bench_mma_s8_tops(int iters, int reps, void* stream, double* tops) {
  if (!tops || iters < 1 || reps < 1) return 1;
  const int sms = sm_count();
  if (sms < 1) return 2;
  cudaStream_t st = (cudaStream_t)stream;
  const int blocks = 4 * sms, threads = 256;
  int* sink = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  int rc = 2;
  if (cudaMalloc(&sink, sizeof(int)) == cudaSuccess && cudaEventCreate(&e0) == cudaSuccess &&
      cudaEventCreate(&e1) == cudaSuccess) {
    mma_s8_rate_kernel<<<blocks, threads, 0, st>>>(16, sink);
    cudaEventRecord(e0, st);
    for (int r = 0; r < reps; ++r) mma_s8_rate_kernel<<<blocks, threads, 0, st>>>(iters, sink);
    cudaEventRecord(e1, st);
    float ms = 0.f;
    if (cudaEventSynchronize(e1) == cudaSuccess && cudaEventElapsedTime(&ms, e0, e1) == cudaSuccess && ms > 0.f) {
      const double warp_mmas = (double)reps * blocks * (threads / 32) * iters * 8.0;
      *tops = 2.0 * warp_mmas * 16 * 8 * 32 / (ms * 1e-3) / 1e12;
      rc = 0;
    }
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (sink) cudaFree(sink);
  return rc;
}

}  // extern "C"
