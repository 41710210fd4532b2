// tcgen05 / TMEM GEMM for sm_103a: out[M][N] = epilogue(A[M][K] * W[N][K]^T).
//
// The dense projections of the DiT block (Eq. 7's B_l: QKV, attention output, cross
// query, cross output, FFN up and down) and the text projection run here.
//
// Design (one CTA per SM, persistent over output tiles of 128 x BN):
//  * warp 0, one thread: TMA producer. Loads 128x64 tiles of A and BNx64 tiles of W
//    (bf16, 128-byte swizzle) into a ring of STAGES shared-memory stages; each stage
//    has a "full" mbarrier (TMA transaction bytes) and an "empty" one (MMA done).
//  * warp 1: allocates 2*BN TMEM columns (two fp32 accumulators of 128 lanes x BN);
//    one thread issues tcgen05.mma (M=128, N=BN, K=16, bf16 -> fp32), commits each
//    stage back to its "empty" barrier and each finished tile to "tmem_full".
//  * warps 2-9: epilogue. Warp w reads TMEM lanes 32*(w%4).. (its lane quarter) and one
//    half of the tile's columns ((w-2)/4) with tcgen05.ld, applies bias / GELU / gated
//    residual / contribution write, stores to global, and releases the accumulator
//    ("tmem_empty") so that the MMA of the tile after next can start while this
//    epilogue runs. Two warps per lane quarter keep twice the epilogue's loads in
//    flight, which the fp32 residual epilogues need to keep up with the mainloop.
// Every mbarrier wait is bounded (mbar_wait): on timeout the kernel records the error,
// stops issuing work, waits (bounded) for its own TMA loads, frees TMEM and returns.
#include <cudaTypedefs.h>

#include "kernels.h"

namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // 64 bf16 = 128 bytes: one swizzle row
constexpr int NUM_THREADS = 320;       // producer, MMA, 8 epilogue warps
constexpr int EPI_THREADS = 256;

template <int BN>
struct TcCfg {
  static constexpr int STAGES = (BN == 256) ? 4 : 6;
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;  // 256 or 512 (power of two >= 32)
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/;
};

// Shared-memory matrix descriptor: K-major, 128-byte swizzle; 8-row core-matrix groups
// are 1024 bytes apart (stride byte offset); leading byte offset unused for this layout.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;                 // leading byte offset (16 B, ignored)
  d |= (uint64_t)(1024 >> 4) << 32;       // stride byte offset
  d |= (uint64_t)1 << 46;                 // descriptor version (tcgen05)
  d |= (uint64_t)2 << 61;                 // layout: 128-byte swizzle
  return d;
}

// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major, M=128, N=BN.
template <int BN>
__device__ __forceinline__ uint32_t idesc_bf16() {
  return (1u << 4)                     // D format: f32
         | (1u << 7)                   // A format: bf16
         | (1u << 10)                  // B format: bf16
         | ((uint32_t)(BN >> 3) << 17) // N >> 3
         | ((uint32_t)(BM >> 4) << 24);// M >> 4
}

template <int BN, int KIND>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmW,
                   int M, int N, int K, GemmEpi epi, int* err) {
  using C = TcCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tmem_full = empty + C::STAGES;
  uint64_t* tmem_empty = tmem_full + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(tmem_empty + 2);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int n_mt = (M + BM - 1) / BM, n_nt = N / BN, n_tiles = n_mt * n_nt;
  const int nk = K / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tmem_full[a], 1);
      mbar_init(&tmem_empty[a], EPI_THREADS);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmW);
  }
  if (warp == 1) tmem_alloc(tmem_holder, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // The weights do not depend on the previous kernel: the producer starts loading the W
  // tiles of its first tile's first stages before waiting for its predecessor.
  const int pre = (warp == 0 && lane == 0 && (int)blockIdx.x < n_tiles)
                      ? (nk < C::STAGES ? nk : C::STAGES) : 0;
  for (int kb = 0; kb < pre; ++kb) {
    uint8_t* sa = smem + kb * C::STAGE_BYTES;
    mbar_expect_tx(&full[kb], C::STAGE_BYTES);
    tma_load_2d(sa + C::A_BYTES, &tmW, &full[kb], kb * BK, ((int)blockIdx.x % n_nt) * BN);
  }
  griddep_wait();  // inputs written by the previous kernel are visible from here on
  griddep_launch();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued[C::STAGES];
#pragma unroll
      for (int s = 0; s < C::STAGES; ++s) issued[s] = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
        const int m0 = (tile / n_nt) * BM, n0 = (tile % n_nt) * BN;
        for (int kb = 0; kb < nk; ++kb) {
          uint8_t* sa = smem + stage * C::STAGE_BYTES;
          if (tile == (int)blockIdx.x && kb < pre) {
            tma_load_2d(sa, &tmA, &full[stage], kb * BK, m0);  // W already requested
          } else {
            if (!mbar_wait(&empty[stage], phase ^ 1u, err)) { ok = false; break; }
            mbar_expect_tx(&full[stage], C::STAGE_BYTES);
            tma_load_2d(sa, &tmA, &full[stage], kb * BK, m0);
            tma_load_2d(sa + C::A_BYTES, &tmW, &full[stage], kb * BK, n0);
          }
          ++issued[stage];
          if (++stage == C::STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        // Let this CTA's loads in flight land before the CTA exits.
        for (int s = 0; s < C::STAGES; ++s)
          if (issued[s]) {
            const uint32_t a = smem_u32(&full[s]);
            const uint64_t t0 = fb_globaltimer();
            while (!mbar_try(a, (issued[s] - 1) & 1u) &&
                   fb_globaltimer() - t0 < FB_WAIT_LIMIT_NS) {
            }
          }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = idesc_bf16<BN>();
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int it = 0;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++it) {
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&tmem_empty[acc], acc_phase ^ 1u, err)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&full[stage], phase, err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * C::STAGE_BYTES);
          const uint64_t adesc = sdesc_sw128(sa), bdesc = sdesc_sw128(sa + C::A_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // +32 bytes per K=16 step inside the swizzle row (encoded >> 4 -> +2)
            tc_mma_f16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb | k) ? 1u : 0u);
          }
          tc_commit(&empty[stage]);
          if (++stage == C::STAGES) { stage = 0; phase ^= 1u; }
        }
        if (ok) tc_commit(&tmem_full[acc]);
      }
    }
  } else {
    // ---------------- epilogue (warps 2..9) ----------------
    const int quarter = warp & 3, half = (warp - 2) >> 2;
    int it = 0;
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const int m0 = (tile / n_nt) * BM, n0 = (tile % n_nt) * BN;
      // short-K tiles only: over a long mainloop the streamed operands evict the rows
      if (nk <= 48 && m0 + quarter * 32 + lane < M)
        epi_prefetch<KIND>(epi, m0 + quarter * 32 + lane, n0 + half * (BN / 2), BN / 2);
      // every lane waits; the warp leaves together if any lane gave up, so the
      // .sync.aligned tcgen05.ld below is always executed by the whole warp
      const bool ok = mbar_wait(&tmem_full[acc], acc_phase, err);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const int row = m0 + quarter * 32 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * BN;
#pragma unroll 1
      for (int c = half * (BN / 64); c < (half + 1) * (BN / 64); ++c) {
        uint32_t r[32];
        tmem_ld32(taddr + c * 32, r);
        tmem_ld_wait();
        reg_fence32(r);
        if (row < M) {
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
          epi_apply32<KIND>(epi, row, n0 + c * 32, v);
        }
      }
      tc_fence_before();
      mbar_arrive(&tmem_empty[acc]);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// ---- 2-SM variant -------------------------------------------------------------------
// A cluster of two CTAs computes a 256 x 256 tile with tcgen05.mma.cta_group::2: CTA r
// of the pair holds rows 128 r .. 128 r + 127 of the A tile and rows 128 r .. of the W
// tile in its shared memory, and receives rows 128 r .. of the accumulator in its TMEM.
// Per SM this moves 32 KB per K block instead of 48 KB for the same MMA work, so six
// stages fit. The even CTA issues the MMAs; its "full" barriers count the TMA bytes of
// both CTAs (the odd CTA's loads complete on them across the pair), its commits arrive on
// the "empty" / "tmem_full" barriers of both CTAs, and both CTAs' epilogue warps release
// an accumulator on its "tmem_empty" barrier.
constexpr int C2_BN = 256;
constexpr int C2_HALF_BYTES = 128 * BK * 2;          // 16 KB: 128 rows x 64 bf16
constexpr int C2_STAGE_BYTES = 2 * C2_HALF_BYTES;    // this CTA's A rows + W rows
constexpr int C2_TMEM_COLS = 2 * C2_BN;
// fp32 residual epilogues stage each 32 x 32 accumulator chunk in shared memory (one
// [32][33] float tile per epilogue warp) so that their global loads and stores are
// whole 128-byte rows; that space comes out of the operand ring (5 stages instead of 6).
constexpr int EPI_STAGE_FLOATS = 32 * 33;
template <int KIND>
struct C2Cfg {
  static constexpr bool STAGED = KIND >= EPI_RESID;
  static constexpr int STAGES = STAGED ? 5 : 6;
  static constexpr int EPI_BYTES = STAGED ? 8 * EPI_STAGE_FLOATS * 4 : 0;
  static constexpr int SMEM_BYTES = STAGES * C2_STAGE_BYTES + EPI_BYTES + 1024 + 256;
};

// Staged residual epilogue of one warp for one 32 x 32 chunk: rows row0..row0+31 (the
// warp's TMEM lane quarter), columns col0..col0+31; acc holds the thread's row (lane).
template <int KIND>
__device__ __forceinline__ void epi_resid_staged(const GemmEpi& e, float* stg, int lane,
                                                 int row0, int col0, int M, const float* acc) {
#pragma unroll
  for (int j = 0; j < 32; ++j) stg[lane * 33 + j] = acc[j];
  __syncwarp();
  const int col = col0 + lane;
  const float g = e.gate ? e.gate[col] : 1.f;
  const float b = e.bias ? e.bias[col] : 0.f;
  // all 32 rows' loads in flight before the first store (one memory latency per chunk)
  constexpr int NB = KIND == EPI_RESID_DELTA ? 16 : 32;  // Delta: 32 would spill
#pragma unroll 1
  for (int r0 = 0; r0 < 32; r0 += NB) {
    float rv[NB], bv[NB];
#pragma unroll
    for (int q = 0; q < NB; ++q) {
      const int row = row0 + r0 + q;
      const size_t off = (size_t)row * e.ldo + col;
      rv[q] = row < M ? e.resid[off] : 0.f;
      if (KIND == EPI_RESID_DELTA) bv[q] = row < M ? e.base[off] : 0.f;
    }
#pragma unroll
    for (int q = 0; q < NB; ++q) {
      const int row = row0 + r0 + q;
      if (row < M) {
        const size_t off = (size_t)row * e.ldo + col;
        const float o = rv[q] + g * (stg[(r0 + q) * 33 + lane] + b);
        if (KIND == EPI_RESID_DELTA) e.delta[off] = __float2bfloat16_rn(o - bv[q]);
        reinterpret_cast<float*>(e.out)[off] = o;
      }
    }
  }
  __syncwarp();
}

template <int KIND>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(NUM_THREADS, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmW,
                    int M, int N, int K, GemmEpi epi, int* err) {
  using CC = C2Cfg<KIND>;
  constexpr int C2_STAGES = CC::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* epi_stage = reinterpret_cast<float*>(smem + C2_STAGES * C2_STAGE_BYTES);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C2_STAGES * C2_STAGE_BYTES + CC::EPI_BYTES);
  uint64_t* empty = full + C2_STAGES;
  uint64_t* tmem_full = empty + C2_STAGES;
  uint64_t* tmem_empty = tmem_full + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(tmem_empty + 2);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const uint32_t rank = cluster_ctarank();
  const int cluster = blockIdx.x >> 1, n_clusters = gridDim.x >> 1;
  const int n_mt = (M + 2 * BM - 1) / (2 * BM), n_nt = N / C2_BN, n_tiles = n_mt * n_nt;
  const int nk = K / BK;
  bool failed = false;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C2_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tmem_full[a], 1);
      mbar_init(&tmem_empty[a], 16);  // 8 epilogue warps x 2 CTAs
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmW);
  }
  if (warp == 1) tmem_alloc_cg2(tmem_holder, C2_TMEM_COLS);
  tc_fence_before();
  cluster_sync();  // both CTAs' barriers initialised, TMEM allocated
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // As in the 1-SM kernel: W tiles of the first tile's first stages before the wait.
  const int pre = (warp == 0 && lane == 0 && cluster < n_tiles)
                      ? (nk < C2_STAGES ? nk : C2_STAGES) : 0;
  for (int kb = 0; kb < pre; ++kb) {
    uint8_t* sa = smem + kb * C2_STAGE_BYTES;
    if (rank == 0) mbar_expect_tx(&full[kb], 2 * C2_STAGE_BYTES);
    tma_load_2d_cg2(sa + C2_HALF_BYTES, &tmW, mapa_shared(smem_u32(&full[kb]), 0), kb * BK,
                    (cluster % n_nt) * C2_BN + 128 * (int)rank);
  }
  griddep_wait();
  griddep_launch();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs) ----------------
      int stage = 0;
      uint32_t phase = 0;
      for (int tile = cluster; tile < n_tiles && !failed; tile += n_clusters) {
        const int m0 = (tile / n_nt) * 2 * BM, n0 = (tile % n_nt) * C2_BN;
        for (int kb = 0; kb < nk; ++kb) {
          uint8_t* sa = smem + stage * C2_STAGE_BYTES;
          const uint32_t fb = mapa_shared(smem_u32(&full[stage]), 0);
          if (tile == cluster && kb < pre) {  // W already requested before the wait
            tma_load_2d_cg2(sa, &tmA, fb, kb * BK, m0 + BM * (int)rank);
            if (++stage == C2_STAGES) { stage = 0; phase ^= 1u; }
            continue;
          }
          if (!mbar_wait(&empty[stage], phase ^ 1u, err)) { failed = true; break; }
          if (rank == 0) mbar_expect_tx(&full[stage], 2 * C2_STAGE_BYTES);
          tma_load_2d_cg2(sa, &tmA, fb, kb * BK, m0 + BM * (int)rank);
          tma_load_2d_cg2(sa + C2_HALF_BYTES, &tmW, fb, kb * BK, n0 + 128 * (int)rank);
          if (++stage == C2_STAGES) { stage = 0; phase ^= 1u; }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------- MMA issuer (even CTA) ----------------
      const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) |
                             ((uint32_t)(C2_BN >> 3) << 17) | ((uint32_t)((2 * BM) >> 4) << 24);
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int tile = cluster; tile < n_tiles && !failed; tile += n_clusters, ++it) {
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&tmem_empty[acc], acc_phase ^ 1u, err)) { failed = true; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * C2_BN;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&full[stage], phase, err)) { failed = true; break; }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * C2_STAGE_BYTES);
          const uint64_t adesc = sdesc_sw128(sa), bdesc = sdesc_sw128(sa + C2_HALF_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc_mma_f16_cg2(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb | k) ? 1u : 0u);
          tc_commit_mc(&empty[stage], 0x3);
          if (++stage == C2_STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!failed) tc_commit_mc(&tmem_full[acc], 0x3);
      }
    }
  } else {
    // ---------------- epilogue (warps 2..9 of both CTAs) ----------------
    const int quarter = warp & 3, half = (warp - 2) >> 2;
    const uint32_t te_remote = mapa_shared(smem_u32(&tmem_empty[0]), 0);
    int it = 0;
    for (int tile = cluster; tile < n_tiles; tile += n_clusters, ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const int m0 = (tile / n_nt) * 2 * BM, n0 = (tile % n_nt) * C2_BN;
      const int prow = m0 + BM * (int)rank + quarter * 32 + lane;
      // short-K tiles only: over a long mainloop the streamed operands evict the rows
      if (nk <= 48 && prow < M) epi_prefetch<KIND>(epi, prow, n0 + half * (C2_BN / 2), C2_BN / 2);
      const bool ok = mbar_wait(&tmem_full[acc], acc_phase, err);
      if (!__all_sync(0xffffffffu, ok)) { failed = true; break; }
      tc_fence_after();
      const int row0 = m0 + BM * (int)rank + quarter * 32;
      const int row = row0 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * C2_BN;
#pragma unroll 1
      for (int c = half * (C2_BN / 64); c < (half + 1) * (C2_BN / 64); ++c) {
        uint32_t r[32];
        tmem_ld32(taddr + c * 32, r);
        tmem_ld_wait();
        reg_fence32(r);
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
        if (CC::STAGED) {
          if (row0 < M)
            epi_resid_staged<KIND>(epi, epi_stage + (warp - 2) * EPI_STAGE_FLOATS, lane, row0,
                                   n0 + c * 32, M, v);
        } else if (row < M) {
          epi_apply32<KIND>(epi, row, n0 + c * 32, v);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(te_remote + acc * (uint32_t)sizeof(uint64_t));
    }
  }

  if (failed || *(volatile int*)err != 0) {
    // After a timeout, give TMA loads that may still be in flight time to land before
    // the shared memory they target is released (they complete within microseconds).
    const uint64_t t0 = fb_globaltimer();
    while (fb_globaltimer() - t0 < 100000ull) __nanosleep(1000);
  }
  tc_fence_before();
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_cg2(tmem_base, C2_TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor map over rows x cols (row stride ld elements), box box_rows x 64.
bool make_map(CUtensorMap* map, const bf16* ptr, int rows, int cols, int ld, int box_rows) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * sizeof(bf16)};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<bf16*>(ptr), dims,
                   strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN, int KIND>
cudaError_t launch(const GemmArgs& g, int* err, int num_sms, cudaStream_t st) {
  using C = TcCfg<BN>;
  CUtensorMap ma, mw;
  if (!make_map(&ma, g.A, g.M, g.K, g.lda, BM) || !make_map(&mw, g.W, g.N, g.K, g.ldw, BN))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, KIND>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  const int tiles = ((g.M + BM - 1) / BM) * (g.N / BN);
  const int grid = tiles < num_sms ? tiles : num_sms;
  return launch_k(gemm_tc_kernel<BN, KIND>, dim3(grid), dim3(NUM_THREADS), C::SMEM_BYTES, st, ma,
                  mw, g.M, g.N, g.K, g.epi, err);
}

template <int BN>
cudaError_t dispatch_kind(const GemmArgs& g, int* err, int num_sms, cudaStream_t st) {
  switch (g.kind) {
    case EPI_BF16: return launch<BN, EPI_BF16>(g, err, num_sms, st);
    case EPI_GELU_BF16: return launch<BN, EPI_GELU_BF16>(g, err, num_sms, st);
    case EPI_RESID: return launch<BN, EPI_RESID>(g, err, num_sms, st);
    case EPI_RESID_DELTA: return launch<BN, EPI_RESID_DELTA>(g, err, num_sms, st);
  }
  return cudaErrorInvalidValue;
}

template <int KIND>
cudaError_t launch2(const GemmArgs& g, int* err, int num_sms, cudaStream_t st) {
  CUtensorMap ma, mw;
  if (!make_map(&ma, g.A, g.M, g.K, g.lda, BM) || !make_map(&mw, g.W, g.N, g.K, g.ldw, 128))
    return cudaErrorInvalidValue;
  constexpr int C2_SMEM_BYTES = C2Cfg<KIND>::SMEM_BYTES;
  cudaError_t e = cudaFuncSetAttribute(gemm_tc2_kernel<KIND>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C2_SMEM_BYTES);
  if (e != cudaSuccess) return e;
  // as many clusters as can be resident at once (pairs must share a GPC)
  static int max_clusters[4] = {0, 0, 0, 0};
  int& mc = max_clusters[KIND];
  if (mc == 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(num_sms, 1, 1);
    cfg.blockDim = dim3(NUM_THREADS, 1, 1);
    cfg.dynamicSmemBytes = C2_SMEM_BYTES;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tc2_kernel<KIND>, &cfg) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = num_sms / 2;
    }
    mc = n < num_sms / 2 ? n : num_sms / 2;
  }
  const int tiles = ((g.M + 2 * BM - 1) / (2 * BM)) * (g.N / C2_BN);
  const int clusters = tiles < mc ? tiles : mc;
  return launch_k(gemm_tc2_kernel<KIND>, dim3(2 * clusters), dim3(NUM_THREADS), C2_SMEM_BYTES, st,
                  ma, mw, g.M, g.N, g.K, g.epi, err);
}

cudaError_t dispatch2(const GemmArgs& g, int* err, int num_sms, cudaStream_t st) {
  switch (g.kind) {
    case EPI_BF16: return launch2<EPI_BF16>(g, err, num_sms, st);
    case EPI_GELU_BF16: return launch2<EPI_GELU_BF16>(g, err, num_sms, st);
    case EPI_RESID: return launch2<EPI_RESID>(g, err, num_sms, st);
    case EPI_RESID_DELTA: return launch2<EPI_RESID_DELTA>(g, err, num_sms, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

bool gemm_tc_supported(const GemmArgs& g) {
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  return g.M >= 1 && g.N % 128 == 0 && g.K % BK == 0 && g.K >= BK && g.lda % 8 == 0 &&
         g.ldw % 8 == 0 && g.epi.ldo % 8 == 0 && al16(g.A) && al16(g.W) && al16(g.epi.out);
}

cudaError_t gemm_tc(const GemmArgs& g, int* err, int num_sms, cudaStream_t st, bool force_1sm) {
  if (!gemm_tc_supported(g)) return cudaErrorInvalidValue;
  // 2-SM 256 x 256 tiles whenever N allows; otherwise 1-SM 128 x BN tiles, BN = 256
  // when that still gives every SM a tile.
  if (g.N % C2_BN == 0 && !force_1sm && num_sms >= 2) return dispatch2(g, err, num_sms, st);
  const int mt = (g.M + BM - 1) / BM;
  if (g.N % 256 == 0 && mt * (g.N / 256) >= num_sms) return dispatch_kind<256>(g, err, num_sms, st);
  return dispatch_kind<128>(g, err, num_sms, st);
}
