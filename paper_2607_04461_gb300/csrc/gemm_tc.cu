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

#include <atomic>
#include <string.h>

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
                   fb_globaltimer() - t0 < fb_wait_limit()) {
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
// Epilogues. bf16 outputs and the fp32 gated residual go through shared memory and TMA:
// each epilogue warp owns two 32 x 32 tiles (bf16 64-byte rows with the 64-byte swizzle,
// or fp32 128-byte rows with the 128-byte swizzle, so that one row per lane is read and
// written at full shared-memory bandwidth), writes its results there and stores them with
// a TMA bulk store that runs while it computes the next chunk; the fp32 residual tiles of
// a chunk are loaded by TMA into the same tile, two chunks ahead, the first two before
// the accumulator is ready. The residual + contribution epilogue (Delta) stages each
// chunk in a [32][33] float tile per warp and moves whole 128-byte rows with plain loads
// and stores. The epilogue space comes out of the operand ring where needed.
constexpr int EPI_STAGE_FLOATS = 32 * 33;
template <int KIND>
struct C2Cfg {
  static constexpr bool TMA_EPI = KIND != EPI_RESID_DELTA;
  static constexpr bool STAGED = KIND == EPI_RESID_DELTA;
  static constexpr int STAGES = KIND == EPI_BF16 || KIND == EPI_GELU_BF16 ? 6 : 5;
  static constexpr int TILE_BYTES = KIND == EPI_RESID ? 32 * 32 * 4 : 32 * 32 * 2;
  static constexpr int EPI_BYTES = TMA_EPI ? 8 * 2 * TILE_BYTES : 8 * EPI_STAGE_FLOATS * 4;
  static constexpr int SMEM_BYTES = STAGES * C2_STAGE_BYTES + EPI_BYTES + 1024 + 512;
};
static_assert(C2Cfg<EPI_BF16>::SMEM_BYTES <= 232448 && C2Cfg<EPI_RESID>::SMEM_BYTES <= 232448 &&
                  C2Cfg<EPI_RESID_DELTA>::SMEM_BYTES <= 232448,
              "2-SM GEMM shared memory");

// byte offset of row r, 16-byte column chunk q in a TMA tile of 128-byte rows (128-byte
// swizzle: chunk bits 4-6 of the address XOR bits 7-9) or 64-byte rows (64-byte swizzle:
// bits 4-5 XOR bits 7-8); tiles start on 1024-byte boundaries
__device__ __forceinline__ uint32_t swz128(int r, int q) { return r * 128 + ((q ^ (r & 7)) << 4); }
__device__ __forceinline__ uint32_t swz64(int r, int q) { return r * 64 + ((q ^ ((r >> 1) & 3)) << 4); }

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

// ---- work split of the 2-SM kernel --------------------------------------------------
// Data-parallel: cluster c computes whole tiles c, c + G, c + 2G, ... (G clusters).
// Stream-K: the U = tiles x nk (tile, K-block) units, tile-major, are cut into G
// contiguous ranges of floor(c U / G) .. floor((c + 1) U / G); a cluster walks its range
// as segments (one tile, K-blocks kb0..kb1). A tile cut between clusters c_lo..c_hi is
// finished by c_lo, which holds its first K blocks as the last segment of its range; the
// others reach it as the first segment of theirs. Each of their epilogue warps writes its
// part of an fp32 partial to the workspace and counts itself on the tile's counter; c_lo's
// matching warp waits (bounded) for the count, adds the partials in contributor (= K)
// order, so the sum does not depend on arrival order, runs the epilogue and resets the
// counter to zero. With U >= G every range is non-empty, so c_hi - c_lo + 1 clusters
// contribute.
struct Seg {
  int tile, kb0, kb1;
};
struct WorkIter {
  long long u, u1;
  int tile, n_tiles, nk, G;
  bool sk;
  __device__ WorkIter(bool sk_, int c, int G_, int n_tiles_, int nk_)
      : tile(c), n_tiles(n_tiles_), nk(nk_), G(G_), sk(sk_) {
    const long long U = (long long)n_tiles_ * nk_;
    u = (long long)c * U / G_;
    u1 = (long long)(c + 1) * U / G_;
  }
  __device__ bool next(Seg& g) {
    if (!sk) {
      if (tile >= n_tiles) return false;
      g.tile = tile;
      g.kb0 = 0;
      g.kb1 = nk;
      tile += G;
      return true;
    }
    if (u >= u1) return false;
    g.tile = (int)(u / nk);
    g.kb0 = (int)(u % nk);
    const long long rest = u1 - u;
    g.kb1 = rest < nk - g.kb0 ? g.kb0 + (int)rest : nk;
    u += g.kb1 - g.kb0;
    return true;
  }
};
// the cluster whose stream-K range holds unit u
__device__ __forceinline__ int sk_owner(long long u, long long U, int G) {
  return (int)(((u + 1) * G - 1) / U);
}
// Workspace slot of cluster c's segment of `tile`: 2c for the first segment of its range,
// 2c + 1 for the last (a range meets at most two cut tiles). Per slot and CTA of the pair,
// 8 epilogue warps x 4096 floats: [chunk 4][j/4 8][lane 32][4], 32 rows x 128 columns.
__device__ __forceinline__ float* sk_part(float* ws, int c, int tile, long long U, int G, int nk,
                                          int rank, int we) {
  const int first_tile = (int)(((long long)c * U / G) / nk);
  const int slot = 2 * c + (tile == first_tile ? 0 : 1);
  return ws + ((size_t)(slot * 2 + rank) * 8 + we) * 4096;
}

template <int KIND>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(NUM_THREADS, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmW,
                    const __grid_constant__ CUtensorMap tmO, const __grid_constant__ CUtensorMap tmR,
                    int M, int N, int K, GemmEpi epi, SkArgs sk, int* err) {
  using CC = C2Cfg<KIND>;
  constexpr int C2_STAGES = CC::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* epi_smem = smem + C2_STAGES * C2_STAGE_BYTES;
  float* epi_stage = reinterpret_cast<float*>(epi_smem);
  uint64_t* full = reinterpret_cast<uint64_t*>(epi_smem + CC::EPI_BYTES);
  uint64_t* empty = full + C2_STAGES;
  uint64_t* tmem_full = empty + C2_STAGES;
  uint64_t* tmem_empty = tmem_full + 2;
  uint64_t* rload = tmem_empty + 2;  // residual tile loads: 2 per epilogue warp
  uint64_t* pload = rload + 16;     // stream-K finisher: one partial prefetch per epilogue warp
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(pload + 8);

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
    for (int b = 0; b < 16; ++b) mbar_init(&rload[b], 1);
    for (int b = 0; b < 8; ++b) mbar_init(&pload[b], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmW);
    if (CC::TMA_EPI) tma_prefetch_desc(&tmO);
    if (KIND == EPI_RESID) tma_prefetch_desc(&tmR);
  }
  if (warp == 1) tmem_alloc_cg2(tmem_holder, C2_TMEM_COLS);
  tc_fence_before();
  cluster_sync();  // both CTAs' barriers initialised, TMEM allocated
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const bool use_sk = sk.on != 0;
  const long long U = (long long)n_tiles * nk;
  // As in the 1-SM kernel: W tiles of the first segment's first stages before the wait.
  Seg first{0, 0, 0};
  int pre = 0;
  if (warp == 0 && lane == 0) {
    WorkIter w0(use_sk, cluster, n_clusters, n_tiles, nk);
    if (w0.next(first)) {
      const int len = first.kb1 - first.kb0;
      pre = len < C2_STAGES ? len : C2_STAGES;
    }
  }
  for (int i = 0; i < pre; ++i) {
    uint8_t* sa = smem + i * C2_STAGE_BYTES;
    if (rank == 0) mbar_expect_tx(&full[i], 2 * C2_STAGE_BYTES);
    tma_load_2d_cg2(sa + C2_HALF_BYTES, &tmW, mapa_shared(smem_u32(&full[i]), 0),
                    (first.kb0 + i) * BK, (first.tile % n_nt) * C2_BN + 128 * (int)rank);
  }
  griddep_wait();
  // Dependents may start once every CTA of this grid has passed here: with the stream-K
  // split all contributors are then resident, so a finisher's wait cannot be starved.
  griddep_launch();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs) ----------------
      int stage = 0;
      uint32_t phase = 0;
      WorkIter wi(use_sk, cluster, n_clusters, n_tiles, nk);
      Seg sg;
      for (int it = 0; !failed && wi.next(sg); ++it) {
        const int m0 = (sg.tile / n_nt) * 2 * BM, n0 = (sg.tile % n_nt) * C2_BN;
        for (int kb = sg.kb0; kb < sg.kb1; ++kb) {
          uint8_t* sa = smem + stage * C2_STAGE_BYTES;
          const uint32_t fb = mapa_shared(smem_u32(&full[stage]), 0);
          if (it == 0 && kb - sg.kb0 < pre) {  // W already requested before the wait
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
      WorkIter wi(use_sk, cluster, n_clusters, n_tiles, nk);
      Seg sg;
      for (int it = 0; !failed && wi.next(sg); ++it) {
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!mbar_wait(&tmem_empty[acc], acc_phase ^ 1u, err)) { failed = true; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * C2_BN;
        for (int kb = sg.kb0; kb < sg.kb1; ++kb) {
          if (!mbar_wait(&full[stage], phase, err)) { failed = true; break; }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * C2_STAGE_BYTES);
          const uint64_t adesc = sdesc_sw128(sa), bdesc = sdesc_sw128(sa + C2_HALF_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc_mma_f16_cg2(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc,
                           (kb > sg.kb0 || k > 0) ? 1u : 0u);
          tc_commit_mc(&empty[stage], 0x3);
          if (++stage == C2_STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!failed) tc_commit_mc(&tmem_full[acc], 0x3);
      }
    }
  } else {
    // ---------------- epilogue (warps 2..9 of both CTAs) ----------------
    const int quarter = warp & 3, half = (warp - 2) >> 2, we = warp - 2;
    const uint32_t te_remote = mapa_shared(smem_u32(&tmem_empty[0]), 0);
    uint8_t* wtiles = epi_smem + we * 2 * CC::TILE_BYTES;  // this warp's two TMA tiles
    uint32_t rl_phase = 0;                                 // bit b: parity of tile b's load
    WorkIter wi(use_sk, cluster, n_clusters, n_tiles, nk);
    Seg sg;
    for (int it = 0; wi.next(sg); ++it) {
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const int tile = sg.tile;
      const bool whole = sg.kb0 == 0 && sg.kb1 == nk;
      const int m0 = (tile / n_nt) * 2 * BM, n0 = (tile % n_nt) * C2_BN;
      const int prow = m0 + BM * (int)rank + quarter * 32 + lane;
      const int row0 = m0 + BM * (int)rank + quarter * 32;
      // residual chunk cc of this warp's rows into tile cc % 2 (one lane)
      auto rload_issue = [&](int cc) {
        const int b = cc & 1;
        mbar_expect_tx(&rload[2 * we + b], CC::TILE_BYTES);
        tma_load_2d(wtiles + b * CC::TILE_BYTES, &tmR, &rload[2 * we + b],
                    n0 + (half * 4 + cc) * 32, row0);
      };
      // bias and gate of this warp's four chunks, one column per lane, requested before
      // the accumulator is ready (the chunks broadcast them with shuffles)
      const int ecol = n0 + half * 128 + lane;
      const float eb0 = epi.bias ? __ldg(epi.bias + ecol) : 0.f;
      const float eb1 = epi.bias ? __ldg(epi.bias + ecol + 32) : 0.f;
      const float eb2 = epi.bias ? __ldg(epi.bias + ecol + 64) : 0.f;
      const float eb3 = epi.bias ? __ldg(epi.bias + ecol + 96) : 0.f;
      const bool has_gate = KIND == EPI_RESID && epi.gate;
      const float eg0 = has_gate ? __ldg(epi.gate + ecol) : 1.f;
      const float eg1 = has_gate ? __ldg(epi.gate + ecol + 32) : 1.f;
      const float eg2 = has_gate ? __ldg(epi.gate + ecol + 64) : 1.f;
      const float eg3 = has_gate ? __ldg(epi.gate + ecol + 96) : 1.f;
      // the cluster holding K blocks 0.. of a cut tile finishes it (see the work split)
      const bool head = !whole && sg.kb0 == 0;
      // tiles this cluster finishes: the first two residual chunks load during the mainloop
      const bool has_r = KIND == EPI_RESID && epi.resid != nullptr;
      const bool early = has_r && (whole || head) && row0 < M;
      if (early) {
        if (lane == 0) {
          bulk_wait_read<0>();
          rload_issue(0);
          rload_issue(1);
        }
        __syncwarp();
      }
      // Delta epilogue, short-K tiles only: the rows into L2 (over a long mainloop the
      // streamed operands would evict them)
      if (CC::STAGED && whole && nk <= 48 && prow < M)
        epi_prefetch<KIND>(epi, prow, n0 + half * (C2_BN / 2), C2_BN / 2);
      const bool ok = mbar_wait(&tmem_full[acc], acc_phase, err);
      if (!__all_sync(0xffffffffu, ok)) { failed = true; break; }
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + acc * C2_BN;
      bool finish = whole;
      int c_lo = 0, n_c = 1;
      if (!whole) {
        c_lo = sk_owner((long long)tile * nk, U, n_clusters);
        n_c = sk_owner((long long)(tile + 1) * nk - 1, U, n_clusters) - c_lo + 1;
        int* ctr = sk.ctr + ((size_t)c_lo * 2 + rank) * 8 + we;
        if (!head) {
          // a later part of a cut tile: publish this warp's partial and count in
          float* part = sk_part(sk.ws, cluster, tile, U, n_clusters, nk, (int)rank, we);
#pragma unroll 1
          for (int cc = 0; cc < 4; ++cc) {
            uint32_t r[32];
            tmem_ld32(taddr + (half * 4 + cc) * 32, r);
            tmem_ld_wait();
            reg_fence32(r);
            float4* dst = reinterpret_cast<float4*>(part + cc * 1024) + lane;
#pragma unroll
            for (int j4 = 0; j4 < 8; ++j4)
              dst[j4 * 32] = make_float4(__uint_as_float(r[4 * j4]),
                                         __uint_as_float(r[4 * j4 + 1]),
                                         __uint_as_float(r[4 * j4 + 2]),
                                         __uint_as_float(r[4 * j4 + 3]));
          }
          __threadfence();
          __syncwarp();
          if (lane == 0) atomicAdd(ctr, 1);
        } else {
          // the finisher: wait (bounded) until the other contributors' warps have counted
          // in. They computed their parts at the start of their ranges, or over ranges no
          // longer than this one, so the wait is short. Every contributor gets an SM: the
          // grid is at most the resident-cluster count, and a dependent grid starts only
          // after all of this grid's CTAs have started.
          bool ok2 = true;
          if (lane == 0) {
            const uint64_t t0 = fb_globaltimer();
            while (*(volatile int*)ctr < n_c - 1) {
              if (*(volatile int*)err != 0) { ok2 = false; break; }
              if (fb_globaltimer() - t0 > fb_wait_limit()) {
                atomicExch(err, FB_DEVERR_WAIT_TIMEOUT);
                ok2 = false;
                break;
              }
              __nanosleep(64);
            }
            if (ok2) *(volatile int*)ctr = 0;  // every contributor is in: ready for reuse
          }
          ok2 = __shfl_sync(0xffffffffu, ok2, 0);
          if (!ok2) { failed = true; break; }
          __threadfence();
          // The next contributor's partial (16 KB for this warp) into this warp's part of
          // the operand ring, idle now: a head segment is the last of the cluster's range,
          // so every MMA that read the ring has completed and no load follows. One bulk
          // copy instead of a round trip per chunk below. Only for rows the chunk loop
          // handles: that loop waits for the copy before the CTA can leave.
          if (lane == 0 && row0 < M) {
            fence_proxy_async_global();
            mbar_expect_tx(&pload[we], 16384);
            bulk_load_1d(smem + we * 16384,
                         sk_part(sk.ws, c_lo + 1, tile, U, n_clusters, nk, (int)rank, we), 16384,
                         &pload[we]);
          }
          __syncwarp();
          finish = true;
        }
      }
      if (finish && row0 < M) {
        if (has_r && !early) {
          if (lane == 0) {
            bulk_wait_read<0>();
            for (int cc = 0; cc < 2; ++cc) rload_issue(cc);
          }
          __syncwarp();
        }
#pragma unroll 1
        for (int cc = 0; cc < 4; ++cc) {
          const int c = half * 4 + cc;
          float v[32];
          if (whole) {
            uint32_t r[32];
            tmem_ld32(taddr + c * 32, r);
            tmem_ld_wait();
            reg_fence32(r);
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
          } else {
            // the contributors' partials summed in K order, this cluster's from TMEM, the
            // next one's from the copy in shared memory (waited for once, at chunk 0)
            if (cc == 0) {
              const bool pok = mbar_wait(&pload[we], 0, err);
              if (!__all_sync(0xffffffffu, pok)) { failed = true; break; }
            }
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.f;
#pragma unroll 1
            for (int q = 0; q < n_c; ++q) {
              const int cq = c_lo + q;
              if (cq == cluster) {
                uint32_t r[32];
                tmem_ld32(taddr + c * 32, r);
                tmem_ld_wait();
                reg_fence32(r);
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] += __uint_as_float(r[j]);
              } else if (cq == c_lo + 1) {  // shared memory: generic loads
                const float4* src = reinterpret_cast<const float4*>(
                                        reinterpret_cast<const float*>(smem + we * 16384) +
                                        cc * 1024) + lane;
#pragma unroll
                for (int j4 = 0; j4 < 8; ++j4) {
                  const float4 f = src[j4 * 32];
                  v[4 * j4] += f.x;
                  v[4 * j4 + 1] += f.y;
                  v[4 * j4 + 2] += f.z;
                  v[4 * j4 + 3] += f.w;
                }
              } else {
                const float4* src = reinterpret_cast<const float4*>(
                                        sk_part(sk.ws, cq, tile, U, n_clusters, nk, (int)rank, we) +
                                        cc * 1024) + lane;
#pragma unroll
                for (int j4 = 0; j4 < 8; ++j4) {
                  const float4 f = __ldcg(src + j4 * 32);
                  v[4 * j4] += f.x;
                  v[4 * j4 + 1] += f.y;
                  v[4 * j4 + 2] += f.z;
                  v[4 * j4 + 3] += f.w;
                }
              }
            }
          }
          const int col0 = n0 + c * 32;
          if (CC::STAGED) {
            epi_resid_staged<KIND>(epi, epi_stage + we * EPI_STAGE_FLOATS, lane, row0, col0, M, v);
            continue;
          }
          const int b = cc & 1;
          uint8_t* tile_b = wtiles + b * CC::TILE_BYTES;
          // this chunk's bias / gate (lane j holds column j; see eb / eg)
          const float bl = cc == 0 ? eb0 : cc == 1 ? eb1 : cc == 2 ? eb2 : eb3;
          const float gl = cc == 0 ? eg0 : cc == 1 ? eg1 : cc == 2 ? eg2 : eg3;
          if (KIND == EPI_RESID) {
            float4 rr[8];
            if (has_r) {
              const bool lok = mbar_wait(&rload[2 * we + b], (rl_phase >> b) & 1u, err);
              rl_phase ^= 1u << b;
              if (!__all_sync(0xffffffffu, lok)) { failed = true; break; }
              // all eight residual loads first: a load after a store to the same tile
              // would otherwise wait for it
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4)
                rr[j4] = *reinterpret_cast<const float4*>(tile_b + swz128(lane, j4));
            } else {
              // no residual: only the store issued from this tile two chunks ago must
              // have left shared memory
              if (lane == 0) bulk_wait_read<1>();
              __syncwarp();
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4) rr[j4] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int j4 = 0; j4 < 8; ++j4) {
              float bb[4], gg[4];
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                bb[q] = __shfl_sync(0xffffffffu, bl, 4 * j4 + q);
                gg[q] = __shfl_sync(0xffffffffu, gl, 4 * j4 + q);
              }
              rr[j4].x += gg[0] * (v[4 * j4] + bb[0]);
              rr[j4].y += gg[1] * (v[4 * j4 + 1] + bb[1]);
              rr[j4].z += gg[2] * (v[4 * j4 + 2] + bb[2]);
              rr[j4].w += gg[3] * (v[4 * j4 + 3] + bb[3]);
            }
#pragma unroll
            for (int j4 = 0; j4 < 8; ++j4)
              *reinterpret_cast<float4*>(tile_b + swz128(lane, j4)) = rr[j4];
          } else {
            // the store issued from this tile two chunks ago has left shared memory (the
            // one outstanding group allowed is the other tile's, one chunk ago)
            if (lane == 0) bulk_wait_read<1>();
            __syncwarp();
            // bias by shuffle; GELU on packed fp32 pairs
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              uint32_t w[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                float y0 = v[8 * q + 2 * i] + __shfl_sync(0xffffffffu, bl, 8 * q + 2 * i);
                float y1 = v[8 * q + 2 * i + 1] + __shfl_sync(0xffffffffu, bl, 8 * q + 2 * i + 1);
                if (KIND == EPI_GELU_BF16) gelu_tanh_f2(y0, y1);
                w[i] = pack_bf16x2(y0, y1);
              }
              *reinterpret_cast<uint4*>(tile_b + swz64(lane, q)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&tmO, smem_u32(tile_b), col0, row0);
            bulk_commit();
            if (has_r && cc + 2 < 4) {
              bulk_wait_read<0>();  // the tile is free again: next residual chunk into it
              rload_issue(cc + 2);
            }
          }
          __syncwarp();
        }
        if (failed) break;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(te_remote + acc * (uint32_t)sizeof(uint64_t));
    }
  }

  if (CC::TMA_EPI && warp >= 2 && lane == 0) bulk_wait<0>();  // own TMA stores complete
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
  // looked up once; a function-local static is initialised thread-safely (the bench
  // drives two models from two host threads)
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    cudaGetLastError();
    return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
  }();
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

// 2-D map over an epilogue matrix [rows][cols] (row stride ld elements) with 32 x 32
// boxes: fp32 with the 128-byte swizzle, bf16 with the 64-byte swizzle.
bool make_epi_map(CUtensorMap* map, const void* ptr, bool f32, int rows, int cols, int ld) {
  auto enc = get_encode();
  if (!enc) return false;
  const size_t es = f32 ? 4 : 2;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * es};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                   2, const_cast<void*>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE,
                   f32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int KIND>
cudaError_t launch2(const GemmArgs& g, int* err, int num_sms, cudaStream_t st) {
  CUtensorMap ma, mw, mo, mr;
  memset(&mo, 0, sizeof(mo));
  memset(&mr, 0, sizeof(mr));
  if (!make_map(&ma, g.A, g.M, g.K, g.lda, BM) || !make_map(&mw, g.W, g.N, g.K, g.ldw, 128))
    return cudaErrorInvalidValue;
  if (C2Cfg<KIND>::TMA_EPI &&
      !make_epi_map(&mo, g.epi.out, KIND == EPI_RESID, g.M, g.N, g.epi.ldo))
    return cudaErrorInvalidValue;
  mr = CUtensorMap{};  // unused without a residual
  if (KIND == EPI_RESID && g.epi.resid &&
      !make_epi_map(&mr, g.epi.resid, true, g.M, g.N, g.epi.ldo))
    return cudaErrorInvalidValue;
  constexpr int C2_SMEM_BYTES = C2Cfg<KIND>::SMEM_BYTES;
  cudaError_t e = cudaFuncSetAttribute(gemm_tc2_kernel<KIND>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C2_SMEM_BYTES);
  if (e != cudaSuccess) return e;
  // as many clusters as can be resident at once (pairs must share a GPC), and no more than
  // the num_sms SMs this launch may use allow
  static std::atomic<int> occ_clusters[4];  // zero until a launch has asked (any thread)
  int occ = occ_clusters[KIND].load(std::memory_order_relaxed);
  if (occ == 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(num_sms, 1, 1);
    cfg.blockDim = dim3(NUM_THREADS, 1, 1);
    cfg.dynamicSmemBytes = C2_SMEM_BYTES;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tc2_kernel<KIND>, &cfg) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = num_sms / 2;
    }
    occ = n;
    occ_clusters[KIND].store(n, std::memory_order_relaxed);
  }
  const int mc = occ < num_sms / 2 ? occ : num_sms / 2;
  const int tiles = ((g.M + 2 * BM - 1) / (2 * BM)) * (g.N / C2_BN);
  const int nk = g.K / BK;
  SkArgs sk{0, g.sk_ws, g.sk_ctr};
  // Stream-K automatically only for a few rounds of tiles (<= 4) whose last round leaves
  // at least 24 K blocks' worth of work per pair idle ((rounds - tiles / pairs) * nk >=
  // 24), with A and W together within half of L2. There the idle pairs' share of the K
  // loop outweighs writing and summing the partials of cut tiles. Measured on all 76
  // pairs: 1560 x 1536 x 8960 gains (43.2 vs 47.9 us); a short K (1560 x 1536 x 1536:
  // 22.9 vs 15.8 us) and 1560 x 8960 x 1536 (3.2 rounds: 41.4 vs 37.6 us) lose. The
  // contiguous unit ranges spread each round over far-apart tiles, so operands larger
  // than L2 are read several times: 8192 x 1536 x 8960 (2.5 rounds, A 147 MB) took 203
  // us and 1.07 GB of DRAM reads against 156 us and 0.34 GB over whole tiles. On a
  // partition of 20 pairs the 1560 x 1536 x 8960 shape's 42 tiles take 3 rounds, the
  // last 90 % empty.
  const long long U = (long long)tiles * nk;
  const bool sk_ok = g.sk_ws && g.sk_ctr && mc <= g.sk_clusters && U >= 4LL * mc;
  const int rounds = (tiles + mc - 1) / mc;
  const double operand_bytes = 2.0 * ((double)g.M + g.N) * g.K;
  const bool sk_pays = rounds <= 4 && ((long long)rounds * mc - tiles) * nk >= 24LL * mc &&
                       operand_bytes <= 64.0 * 1024 * 1024;
  if (g.sk_mode == 2) {
    if (!sk_ok) return cudaErrorInvalidValue;
    sk.on = 1;
  } else if (g.sk_mode == 0 && sk_ok && sk_pays) {
    sk.on = 1;
  }
  const int clusters = sk.on ? mc : (tiles < mc ? tiles : mc);
  return launch_k(gemm_tc2_kernel<KIND>, dim3(2 * clusters), dim3(NUM_THREADS), C2_SMEM_BYTES, st,
                  ma, mw, mo, mr, g.M, g.N, g.K, g.epi, sk, err);
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
         g.ldw % 8 == 0 && g.epi.ldo % 8 == 0 && al16(g.A) && al16(g.W) && al16(g.epi.out) &&
         (g.kind < EPI_RESID || al16(g.epi.resid)) && (g.kind != EPI_RESID_DELTA || g.epi.resid) &&
         (g.kind != EPI_RESID_DELTA || (al16(g.epi.base) && al16(g.epi.delta)));
}

cudaError_t gemm_tc_set_wait_limit(unsigned long long ns) { return fb_set_wait_limit_tu(ns); }

cudaError_t gemm_tc(const GemmArgs& g, int* err, int num_sms, cudaStream_t st, bool force_1sm) {
  if (!gemm_tc_supported(g)) return cudaErrorInvalidValue;
  // 2-SM 256 x 256 tiles whenever N allows; otherwise 1-SM 128 x BN tiles, BN = 256
  // when that still gives every SM a tile.
  if (g.N % C2_BN == 0 && !force_1sm && num_sms >= 2) return dispatch2(g, err, num_sms, st);
  if (g.sk_mode == 2) return cudaErrorInvalidValue;  // stream-K exists in the 2-SM kernel only
  const int mt = (g.M + BM - 1) / BM;
  if (g.N % 256 == 0 && mt * (g.N / 256) >= num_sms) return dispatch_kind<256>(g, err, num_sms, st);
  return dispatch_kind<128>(g, err, num_sms, st);
}
