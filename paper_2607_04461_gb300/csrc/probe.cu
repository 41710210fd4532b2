// Measurement probes of the SM's pipes, against which the attention and GEMM kernels are
// judged:
//  * mma_rate: how many MACs per SM clock tcgen05.mma kind::f16 sustains when 1, 2 or 4
//    warps (one elected thread each) issue `reps` M = 128, K = 16 instructions of width N
//    into accumulators of their own (1-SM form, operands in shared memory);
//  * mma_gap: the same rate when one thread issues batches of 8 such instructions (N =
//    128) with a spin of `gap` clocks after each batch (how much queued work hides a gap
//    in the issuing thread);
//  * mufu: ex2.approx, tanh.approx, rcp.approx or ex2.approx.f16x2 (two results per
//    instruction) results per SM clock (16 independent chains per thread, 256 threads
//    per SM);
//  * tmem_load: clocks from four 32x32b.x32 TMEM loads (128 columns) to their wait's end,
//    with the tensor pipe idle or running;
//  * mma_mix: the rate of batches shaped like one attention step of one query tile
//    (8 instructions into an O-like accumulator, then 8 into an S-like one) for three
//    operand forms of the first eight, with up to 7 other warps reading and writing
//    TMEM meanwhile, as softmax warps do.
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

// ---- issue gaps: batches of 8 MMAs (M = N = 128, K = 16) with `gap` clocks between them
__global__ void __launch_bounds__(PROBE_THREADS, 1)
    mma_gap_kernel(int gap, int batches, unsigned long long* cycles, int* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t bar;
  __shared__ uint32_t holder;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (threadIdx.x / 32 == 0) tmem_alloc(&holder, 128);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = holder;
  griddep_wait();
  if (threadIdx.x == 0) {
    const uint64_t ad = probe_desc_sw128(smem_u32(sm)), bd = probe_desc_sw128(smem_u32(sm) + 16384);
    const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(128 >> 3) << 17) |
                           ((uint32_t)(128 >> 4) << 24);
    const long long t0 = clock64();
    for (int b = 0; b < batches; ++b) {
#pragma unroll
      for (int k = 0; k < 8; ++k) tc_mma_f16(tm, ad + 2 * (k & 3), bd + 2 * (k & 3), idesc, (b | k) ? 1u : 0u);
      const long long c0 = clock64();
      while (clock64() - c0 < gap) {
      }
    }
    tc_commit(&bar);
    if (mbar_wait(&bar, 0, err)) cycles[blockIdx.x] = clock64() - t0;
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x / 32 == 0) {
    tc_fence_after();
    tmem_dealloc(tm, 128);
  }
}

// ---- MUFU rates: 16 independent chains per thread of one operation
constexpr int PROBE_THREADS2 = 256;  // the MUFU and TMEM-load probes: 8 warps
template <int OP>
__global__ void __launch_bounds__(PROBE_THREADS2, 1) mufu_kernel(int reps, unsigned long long* cycles,
                                                                float* sink) {
  griddep_wait();
  float a[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) a[i] = 0.001f * (float)(threadIdx.x + i) + 0.5f;
  uint32_t hv[16];  // op 3: pairs of f16
#pragma unroll
  for (int i = 0; i < 16; ++i) hv[i] = 0x3800b800u ^ (uint32_t)(threadIdx.x & 7);  // {-0.5, 0.5}
  const long long t0 = clock64();
  for (int r = 0; r < reps; ++r) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if (OP == 3) {
        uint32_t y;
        asm volatile("ex2.approx.f16x2 %0, %1;" : "=r"(y) : "r"(hv[i]));
        hv[i] = y ^ 0x40004000u;  // keeps the pairs in range (sign and exponent bits)
        continue;
      }
      float y;
      if (OP == 0) asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(a[i]));
      else if (OP == 1) asm volatile("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(a[i]));
      else asm volatile("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(a[i]));
      a[i] = OP == 0 ? y - 1.0f : y + 0.5f;  // bounded chains
    }
  }
  const long long t1 = clock64();
  float acc = 0.f;
#pragma unroll
  for (int i = 0; i < 16; ++i) acc += a[i] + (float)(hv[i] & 1u);
  if (acc == 12345.f) sink[0] = acc;  // keeps the chains
  if (threadIdx.x == 0) cycles[blockIdx.x] = t1 - t0;
}

// ---- TMEM load latency: warps 4-7 time `reps` loads of 128 columns (4 x 32x32b.x32, one
// wait) of their lane quarter; with busy != 0, thread 0 keeps the tensor pipe running
// (M = N = 128 MMAs into other columns) meanwhile
__global__ void __launch_bounds__(PROBE_THREADS2, 1)
    tmem_load_kernel(int reps, int busy, unsigned long long* cycles, int* err, float* sink) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t bar;
  __shared__ uint32_t holder;
  __shared__ volatile int done;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (threadIdx.x == 0) {
    done = 0;
    mbar_init(&bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) tmem_alloc(&holder, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = holder;
  griddep_wait();
  if (threadIdx.x == 0 && busy) {
    const uint64_t ad = probe_desc_sw128(smem_u32(sm)), bd = probe_desc_sw128(smem_u32(sm) + 16384);
    const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(128 >> 3) << 17) |
                           ((uint32_t)(128 >> 4) << 24);
    for (int i = 0; i < 200000 && done < 4; ++i)
      tc_mma_f16(tm, ad + 2 * (i & 3), bd + 2 * (i & 3), idesc, i ? 1u : 0u);
    tc_commit(&bar);
    mbar_wait(&bar, 0, err);
  }
  if (warp >= 4 && warp < 8) {
    const uint32_t ta = tm + ((uint32_t)((warp & 3) * 32) << 16) + 256;
    long long tot = 0;
    float x = 0.f;
    for (int it = 0; it < reps; ++it) {
      uint32_t r[128];
      const long long c0 = clock64();
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(ta + c * 32, r + c * 32);
      tmem_ld_wait();
#pragma unroll
      for (int c = 0; c < 4; ++c) reg_fence32(r + c * 32);
      // the second clock read takes a loaded value as an operand, so it cannot run before
      // the data has arrived (a wait may return before its registers are written)
      const float y = __uint_as_float(r[0]) + __uint_as_float(r[127]);
      long long c1;
      asm volatile("{\n\t.reg .f32 t;\n\tmov.b32 t, %1;\n\tmov.u64 %0, %%clock64;\n\t}"
                   : "=l"(c1) : "f"(y) : "memory");
      tot += c1 - c0;
      x += y;
    }
    if (x == 12345.f) sink[0] = x;
    if (lane == 0) cycles[blockIdx.x * 4 + (warp & 3)] = (unsigned long long)(tot / reps);
    __syncwarp();
    if (lane == 0) atomicAdd((int*)&done, 1);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
}

// ---- attention-shaped batches. Per batch: 8 instructions (M = N = 128, K = 16) into D0
// (columns 0-127) in form 0 (A and B K-major in shared memory), 1 (B MN-major, 64-element
// rows 16 KB apart, as the PV product reads V) or 2 (B MN-major, A from TMEM columns
// 256-319, as PV reads P), then 8 K-major instructions into D1 (columns 128-255, as S).
// Forms 3 and 4 issue the attention kernel's whole step instead (32 instructions per
// batch: PV_A, S_A, PV_B, S_B over its shared-memory rings and TMEM map, every operand
// slice distinct), form 4 with its tcgen05.commit after S_A, PV_B and S_B (two). Forms 3
// and 4 build each descriptor from its address per instruction; forms 5 and 6 are forms
// 3 and 4 with the descriptors' lower words hoisted (one add per operand).
// Warps 1..loaders meanwhile each load columns 128-255 of their lane quarter (4 x
// 32x32b.x32, one wait), store 64 columns (2 x 32x32b.x32 into columns 384-447) and spin
// `loader_gap` clocks, until thread 0 is done (at most 1 << 20 rounds). With SOFTMAX the
// loaders also do a softmax row's arithmetic between load and store: the row maximum,
// 128 scaled exponentials (ex2.approx), their sum and the bf16 packing.
__device__ __forceinline__ void probe_tmem_st32(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ uint64_t probe_desc_mn_sw128(uint32_t saddr, uint32_t lbo) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}
__device__ __forceinline__ void probe_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                             uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

template <int FORM, bool SOFTMAX>
__global__ void __launch_bounds__(PROBE_THREADS2, 1)
    mma_mix_kernel(int loaders, int loader_gap, int batches, unsigned long long* cycles, int* err,
                   float* sink) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t bar, bar2[3];  // bar2: commits nobody waits for (form 4)
  __shared__ uint32_t holder;
  __shared__ volatile int done;
  const int warp = threadIdx.x / 32;
  if (threadIdx.x == 0) {
    done = 0;
    mbar_init(&bar, 1);
    for (int i = 0; i < 3; ++i) mbar_init(&bar2[i], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) tmem_alloc(&holder, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = holder;
  griddep_wait();
  if (threadIdx.x == 0) {
    const uint32_t base = smem_u32(sm);
    const uint64_t ad = probe_desc_sw128(base), bd = probe_desc_sw128(base + 16384);
    const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(128 >> 3) << 17) |
                           ((uint32_t)(128 >> 4) << 24);
    const uint32_t idesc_mn = idesc | (1u << 16);
    const long long t0 = clock64();
    // forms 5 and 6: the same step from descriptor lower words hoisted out of the loop
    const uint32_t dhi = DESC_HI, q_lo = desc_lo_k(base), k_lo = desc_lo_k(base + 65536);
    const uint32_t v_lo = desc_lo_mn(base + 163840, 16384);
    for (int b = 0; b < batches && FORM >= 5; ++b) {
      const uint32_t ka = k_lo + (uint32_t)(b % 3) * 2048, va = v_lo + (uint32_t)(b & 1) * 2048;
#pragma unroll
      for (int g = 0; g < 2; ++g) {
#pragma unroll
        for (int k = 0; k < 8; ++k)
          tc_mma_ts_lo(tm + 256 + 128 * g, tm + 128 * g + 8 * k, va + k * 128, dhi, idesc_mn,
                       (b | k) ? 1u : 0u);
        if (FORM == 6 && g == 1) tc_commit(&bar2[1]);
        const uint32_t qa = q_lo + (uint32_t)g * 2048;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t off = ((k >> 2) * 16384 + (k & 3) * 32) >> 4;
          tc_mma_ss_lo(tm + 128 * g, qa + off, ka + off, dhi, idesc, k ? 1u : 0u);
        }
        if (FORM == 6) tc_commit(&bar2[0]);
        if (FORM == 6 && g == 1) tc_commit(&bar2[2]);
      }
    }
    for (int b = 0; b < batches && FORM >= 3 && FORM < 5; ++b) {
      // one attention step: Q tiles at 0 and 32 KB, K ring (3 x 32 KB) from 64 KB, V ring
      // (2 x 32 KB) from 160 KB; TMEM S_A|P_A, S_B|P_B, O_A, O_B at columns 0/128/256/384
      const uint32_t ka = base + 65536 + (uint32_t)(b % 3) * 32768;
      const uint32_t va = base + 163840 + (uint32_t)(b & 1) * 32768;
#pragma unroll
      for (int g = 0; g < 2; ++g) {
#pragma unroll
        for (int k = 0; k < 8; ++k)
          probe_mma_ts(tm + 256 + 128 * g, tm + 128 * g + 8 * k,
                       probe_desc_mn_sw128(va + k * 2048, 16384), idesc_mn, (b | k) ? 1u : 0u);
        if (FORM == 4 && g == 1) tc_commit(&bar2[1]);
        const uint32_t qa = base + (uint32_t)g * 32768;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const uint32_t off = (k >> 2) * 16384 + (k & 3) * 32;
          tc_mma_f16(tm + 128 * g, probe_desc_sw128(qa + off), probe_desc_sw128(ka + off), idesc,
                     k ? 1u : 0u);
        }
        if (FORM == 4) tc_commit(&bar2[0]);
        if (FORM == 4 && g == 1) tc_commit(&bar2[2]);
      }
    }
    for (int b = 0; b < batches && FORM < 3; ++b) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const uint32_t acc = (b | k) ? 1u : 0u;
        if (FORM == 0)
          tc_mma_f16(tm, ad + 2 * (k & 3), bd + 2 * (k & 3), idesc, acc);
        else if (FORM == 1)
          tc_mma_f16(tm, ad + 2 * (k & 3), probe_desc_mn_sw128(base + 16384 + k * 2048, 16384),
                     idesc_mn, acc);
        else
          probe_mma_ts(tm, tm + 256 + 8 * k, probe_desc_mn_sw128(base + 16384 + k * 2048, 16384),
                       idesc_mn, acc);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k)
        tc_mma_f16(tm + 128, ad + 2 * (k & 3), bd + 2 * (k & 3), idesc, k ? 1u : 0u);
    }
    tc_commit(&bar);
    if (mbar_wait(&bar, 0, err)) cycles[blockIdx.x] = clock64() - t0;
    done = 1;
  }
  if (warp >= 1 && warp <= loaders) {
    const uint32_t lq = tm + ((uint32_t)((warp & 3) * 32) << 16);
    float x = 0.f;
    for (int it = 0; it < (1 << 20) && !done; ++it) {
      uint32_t r[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(lq + 128 + c * 32, r + c * 32);
      tmem_ld_wait();
#pragma unroll
      for (int c = 0; c < 4; ++c) reg_fence32(r + c * 32);
      if (SOFTMAX) {
        float m = -INFINITY;
#pragma unroll
        for (int i = 0; i < 128; ++i) m = fmaxf(m, __uint_as_float(r[i] & 0x3fffffffu));
        float l = 0.f;
#pragma unroll
        for (int i = 0; i < 64; ++i) {
          float e0, e1;
          const float a0 = fmaf(__uint_as_float(r[2 * i] & 0x3fffffffu), 0.125f, -m);
          const float a1 = fmaf(__uint_as_float(r[2 * i + 1] & 0x3fffffffu), 0.125f, -m);
          asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(e0) : "f"(a0));
          asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(e1) : "f"(a1));
          l += e0 + e1;
          asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r[i]) : "f"(e1), "f"(e0));
        }
        x += l;
      } else {
#pragma unroll
        for (int i = 0; i < 64; ++i) r[i] ^= r[64 + i];
      }
      probe_tmem_st32(lq + 384, r);
      probe_tmem_st32(lq + 416, r + 32);
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      x += __uint_as_float(r[0] & 0x3fffffffu);
      const long long c0 = clock64();
      while (clock64() - c0 < loader_gap) {
      }
    }
    if (x == 12345.f) sink[0] = x;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
}

}  // namespace

cudaError_t mma_mix_probe(int form, int loaders, int loader_gap, int batches, int grid,
                          unsigned long long* cycles, int* err, float* sink, cudaStream_t st) {
  if (form < 0 || form > 13 || loaders < 0 || loaders > 7 || loader_gap < 0 || batches < 1 ||
      grid < 1)
    return cudaErrorInvalidValue;
  using K = void (*)(int, int, int, unsigned long long*, int*, float*);
  const K ks[14] = {mma_mix_kernel<0, false>, mma_mix_kernel<1, false>, mma_mix_kernel<2, false>,
                    mma_mix_kernel<3, false>, mma_mix_kernel<4, false>, mma_mix_kernel<5, false>,
                    mma_mix_kernel<6, false>,
                    mma_mix_kernel<0, true>,  mma_mix_kernel<1, true>,  mma_mix_kernel<2, true>,
                    mma_mix_kernel<3, true>,  mma_mix_kernel<4, true>,  mma_mix_kernel<5, true>,
                    mma_mix_kernel<6, true>};
  const K k = ks[form];
  const int smem = (form % 7 >= 3 ? 7 * 32768 : PROBE_STAGE) + 1024;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = launch_k(k, dim3(grid), dim3(PROBE_THREADS2), smem, st, loaders, loader_gap, batches,
               cycles, err, sink);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t mma_gap_probe(int gap, int batches, int grid, unsigned long long* cycles, int* err,
                          cudaStream_t st) {
  if (gap < 0 || batches < 1 || grid < 1) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(mma_gap_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       PROBE_STAGE + 1024);
  if (e != cudaSuccess) return e;
  e = launch_k(mma_gap_kernel, dim3(grid), dim3(PROBE_THREADS), PROBE_STAGE + 1024, st, gap,
               batches, cycles, err);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t mufu_probe(int op, int reps, int grid, unsigned long long* cycles, float* sink,
                       cudaStream_t st) {
  if (op < 0 || op > 3 || reps < 1 || grid < 1) return cudaErrorInvalidValue;
  auto k = op == 0 ? mufu_kernel<0> : op == 1 ? mufu_kernel<1> : op == 2 ? mufu_kernel<2>
                                                                         : mufu_kernel<3>;
  cudaError_t e = launch_k(k, dim3(grid), dim3(PROBE_THREADS2), 0, st, reps, cycles, sink);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t tmem_load_probe(int reps, int busy, int grid, unsigned long long* cycles, int* err,
                            float* sink, cudaStream_t st) {
  if (reps < 1 || grid < 1) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(tmem_load_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       PROBE_STAGE + 1024);
  if (e != cudaSuccess) return e;
  e = launch_k(tmem_load_kernel, dim3(grid), dim3(PROBE_THREADS2), PROBE_STAGE + 1024, st, reps,
               busy, cycles, err, sink);
  return e != cudaSuccess ? e : cudaGetLastError();
}

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
