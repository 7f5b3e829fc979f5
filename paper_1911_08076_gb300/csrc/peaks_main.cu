// Peak-rate microbenchmark for the instructions the quantized conv can use on
// sm_103a: tcgen05.mma kind::f8f6f4 (e4m3) at N = 64/128/256, legacy warp
// mma.sync (s8, e4m3, b1 and.popc) and CUDA-core popc.  Standalone program;
// prints one JSON object.  Built and run by paper_1911_08076_gb300.peaks.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>
#include <cstdlib>

#define CK(x)                                                                           \
  do {                                                                                  \
    cudaError_t e_ = (x);                                                               \
    if (e_ != cudaSuccess) {                                                            \
      fprintf(stderr, "CUDA error %s at %s:%d\n", cudaGetErrorString(e_), __FILE__, __LINE__); \
      exit(1);                                                                          \
    }                                                                                   \
  } while (0)

__device__ int g_err;

__device__ __forceinline__ uint32_t su32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ unsigned long long gns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// bounded (2 s) wait on an mbarrier phase
__device__ __forceinline__ void wait_bar(uint32_t bar, uint32_t ph) {
  const unsigned long long t0 = gns();
  for (uint32_t i = 0; i < (1u << 24); ++i) {
    uint32_t ok;
    asm volatile("{.reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0,1,0,p;}"
                 : "=r"(ok)
                 : "r"(bar), "r"(ph)
                 : "memory");
    if (ok) return;
    if ((i & 255u) == 255u && gns() - t0 > 2000000000ull) break;
  }
  atomicExch(&g_err, 1);
}

__device__ __forceinline__ uint64_t sdesc(uint32_t a) {
  return (uint64_t)((a & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)64 << 32) | ((uint64_t)1 << 46) |
         ((uint64_t)2 << 61);
}

// One CTA per SM issues `iters` M128 x N x K32 e4m3 MMAs on fixed shared-memory operands.
__global__ void __launch_bounds__(128) tc_rate(int N, int iters, float* sink) {
  extern __shared__ uint8_t smraw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tslot;
  const int tid = threadIdx.x, warp = tid >> 5;
  for (int i = tid; i < 48 * 1024 / 4; i += 128) ((uint32_t*)sm)[i] = 0x38383838u;
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&tslot)), "r"(512));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(su32(&bar)));
    asm volatile("fence.mbarrier_init.release.cluster;");
  }
  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;");
  const uint32_t tm = tslot;
  if (tid == 0) {
    const uint32_t idesc = (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
    const uint64_t ad = sdesc(su32(sm)), bd = sdesc(su32(sm + 16384));
    for (int i = 0; i < iters; ++i)
      asm volatile(
          "{.reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;}" ::"r"(
              tm + (uint32_t)((i & 1) * 256)),
          "l"(ad + 2 * (i & 3)), "l"(bd + 2 * (i & 3)), "r"(idesc), "r"(1));
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(&bar))
                 : "memory");
  }
  wait_bar(su32(&bar), 0);
  asm volatile("tcgen05.fence::after_thread_sync;");
  if (warp == 0) {
    uint32_t r;
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];\n\ttcgen05.wait::ld.sync.aligned;" : "=r"(r) : "r"(tm));
    if (tid == 0) sink[blockIdx.x] = __uint_as_float(r);
  }
  asm volatile("tcgen05.fence::before_thread_sync;");
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tm), "r"(512));
}

__global__ void mma_s8_rate(int iters, int* sink) {
  const int a0 = threadIdx.x, a1 = a0 * 3, a2 = a0 * 5, a3 = a0 * 7, b0 = a0 * 11, b1 = a0 * 13;
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
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 0x7fffffff) sink[0] = s;
}

__global__ void mma_e4m3_rate(int iters, float* sink) {
  const uint32_t a0 = 0x38383838u, b0 = 0x38383838u;
  float c[8][4] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      asm volatile(
          "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
          : "+f"(c[j][0]), "+f"(c[j][1]), "+f"(c[j][2]), "+f"(c[j][3])
          : "r"(a0), "r"(a0), "r"(a0), "r"(a0), "r"(b0), "r"(b0));
  }
  float s = 0;
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 1.2345f) sink[0] = s;
}

__global__ void mma_b1_rate(int iters, int* sink) {
  const uint32_t a0 = threadIdx.x * 0x9E3779B9u, b0 = a0 ^ 0x5555u;
  int c[8][4] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      asm volatile(
          "mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.and.popc {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
          "{%0,%1,%2,%3};"
          : "+r"(c[j][0]), "+r"(c[j][1]), "+r"(c[j][2]), "+r"(c[j][3])
          : "r"(a0), "r"(a0), "r"(a0), "r"(a0), "r"(b0), "r"(b0));
  }
  int s = 0;
  for (int j = 0; j < 8; ++j) s += c[j][0] + c[j][1] + c[j][2] + c[j][3];
  if (s == 0x7fffffff) sink[0] = s;
}

__global__ void popc_rate(int iters, int* sink) {
  uint32_t x = threadIdx.x * 0x9E3779B9u + blockIdx.x, y = x ^ 0xA5A5A5A5u;
  int acc[8] = {};
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      acc[j] += __popc(x & (y + j));
      x = x * 1664525u + 1013904223u;
    }
  }
  int s = 0;
  for (int j = 0; j < 8; ++j) s += acc[j];
  if (s == 0x7fffffff) sink[0] = s;
}

int main() {
  int sms = 0, clk = 0;
  CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0));
  CK(cudaDeviceGetAttribute(&clk, cudaDevAttrClockRate, 0));
  float* sink;
  CK(cudaMalloc(&sink, 4096 * sizeof(float)));
  cudaEvent_t e0, e1;
  CK(cudaEventCreate(&e0));
  CK(cudaEventCreate(&e1));
  const int smem = 120 * 1024;   // one CTA per SM (tensor memory is taken whole)
  CK(cudaFuncSetAttribute(tc_rate, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  printf("{\"sms\": %d, \"max_clock_mhz\": %d", sms, clk / 1000);
  for (int N : {64, 128, 256}) {
    const int iters = 8192;
    tc_rate<<<sms, 128, smem>>>(N, 64, sink);
    CK(cudaDeviceSynchronize());
    CK(cudaEventRecord(e0));
    tc_rate<<<sms, 128, smem>>>(N, iters, sink);
    CK(cudaEventRecord(e1));
    CK(cudaEventSynchronize(e1));
    float ms;
    CK(cudaEventElapsedTime(&ms, e0, e1));
    const double ops = 2.0 * sms * (double)iters * 128.0 * N * 32.0;
    printf(", \"tcgen05_e4m3_n%d_tops\": %.1f", N, ops / (ms * 1e-3) / 1e12);
  }
  const int blocks = sms * 4, threads = 256, iters = 4096;
  const double warp_mmas = (double)blocks * (threads / 32) * iters * 8;
  float ms;
  mma_s8_rate<<<blocks, threads>>>(16, (int*)sink);
  CK(cudaDeviceSynchronize());
  CK(cudaEventRecord(e0));
  mma_s8_rate<<<blocks, threads>>>(iters, (int*)sink);
  CK(cudaEventRecord(e1));
  CK(cudaEventSynchronize(e1));
  CK(cudaEventElapsedTime(&ms, e0, e1));
  printf(", \"mma_sync_s8_tops\": %.1f", 2.0 * warp_mmas * 16 * 8 * 32 / (ms * 1e-3) / 1e12);
  mma_e4m3_rate<<<blocks, threads>>>(16, sink);
  CK(cudaDeviceSynchronize());
  CK(cudaEventRecord(e0));
  mma_e4m3_rate<<<blocks, threads>>>(iters, sink);
  CK(cudaEventRecord(e1));
  CK(cudaEventSynchronize(e1));
  CK(cudaEventElapsedTime(&ms, e0, e1));
  printf(", \"mma_sync_e4m3_tflops\": %.1f", 2.0 * warp_mmas * 16 * 8 * 32 / (ms * 1e-3) / 1e12);
  mma_b1_rate<<<blocks, threads>>>(16, (int*)sink);
  CK(cudaDeviceSynchronize());
  CK(cudaEventRecord(e0));
  mma_b1_rate<<<blocks, threads>>>(iters, (int*)sink);
  CK(cudaEventRecord(e1));
  CK(cudaEventSynchronize(e1));
  CK(cudaEventElapsedTime(&ms, e0, e1));
  printf(", \"mma_sync_b1_popc_bit_tops\": %.1f", 2.0 * warp_mmas * 16 * 8 * 256 / (ms * 1e-3) / 1e12);
  popc_rate<<<blocks, threads>>>(16, (int*)sink);
  CK(cudaDeviceSynchronize());
  CK(cudaEventRecord(e0));
  popc_rate<<<blocks, threads>>>(iters, (int*)sink);
  CK(cudaEventRecord(e1));
  CK(cudaEventSynchronize(e1));
  CK(cudaEventElapsedTime(&ms, e0, e1));
  const double pops = (double)blocks * threads * iters * 8;
  printf(", \"popc_per_clk_per_sm\": %.1f", pops / (ms * 1e-3) / sms / (clk * 1e3));
  int err = 0;
  CK(cudaMemcpyFromSymbol(&err, g_err, sizeof(int)));
  printf(", \"wait_timeouts\": %d}\n", err);
  return err ? 2 : 0;
}
