// Measurement probe of the tensor pipe: how many MACs per SM clock tcgen05.mma kind::f16
// sustains when 1, 2 or 4 warps (one elected thread each) issue `reps` M = 128, K = 16
// instructions of width N into accumulators of their own (1-SM form, operands in shared
// memory). The attention and GEMM kernels are judged against this rate.
#include "kernels.h"

namespace {

__device__ __forceinline__ uint64_t probe_desc_sw128(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

constexpr int PROBE_THREADS = 128;
constexpr int PROBE_STAGE = 49152;  // per issuer: A 128 x 64 bf16 (16 KB) + B 256 x 64 (32 KB)
constexpr int PROBE_SMEM = 4 * PROBE_STAGE + 1024;

__global__ void __launch_bounds__(PROBE_THREADS, 1)
    mma_rate_kernel(int issuers, int N, int reps, unsigned long long* cycles, int* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t bar;
  __shared__ uint32_t holder;
  __shared__ unsigned long long t0;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (threadIdx.x == 0) {
    mbar_init(&bar, issuers);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) tmem_alloc(&holder, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = holder;
  griddep_wait();
  if (threadIdx.x == 0) t0 = clock64();
  __syncthreads();
  if (warp < issuers && lane == 0) {
    const uint32_t base = smem_u32(sm + warp * PROBE_STAGE);
    const uint64_t ad = probe_desc_sw128(base), bd = probe_desc_sw128(base + 16384);
    const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
                           ((uint32_t)(128 >> 4) << 24);
    const uint32_t acc = tm + (uint32_t)(warp * N);  // issuers * N <= 512 columns
    for (int i = 0; i < reps; ++i) {
      const uint32_t kk = i & 3;
      tc_mma_f16(acc, ad + 2 * kk, bd + 2 * kk, idesc, i > 0 ? 1u : 0u);
    }
    tc_commit(&bar);
  }
  if (threadIdx.x == 0) {
    const bool ok = mbar_wait(&bar, 0, err);
    if (ok) cycles[blockIdx.x] = clock64() - t0;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
}

}  // namespace

cudaError_t mma_rate_probe(int issuers, int N, int reps, int grid, unsigned long long* cycles,
                           int* err, cudaStream_t st) {
  if (issuers < 1 || issuers > 4 || (N != 64 && N != 128 && N != 256) || issuers * N > 512 ||
      reps < 1 || grid < 1)
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(mma_rate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       PROBE_SMEM);
  if (e != cudaSuccess) return e;
  e = launch_k(mma_rate_kernel, dim3(grid), dim3(PROBE_THREADS), PROBE_SMEM, st, issuers, N, reps,
               cycles, err);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
