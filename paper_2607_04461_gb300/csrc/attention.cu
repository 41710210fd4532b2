// Flash-style attention O = softmax(Q K^T / sqrt(dh)) V for the DiT block's
// self-attention (K, V per candidate) and cross-attention (K, V of the projected text,
// shared by all candidates). Non-causal; ragged Lq / Lkv tails are masked.
//
// One CTA = 4 warps = 64 query rows of one (batch, head); each warp owns 16 rows and
// keeps its Q fragments, the running row max / sum and the O accumulator in
// registers (online softmax, base-2 exponentials with the 1/sqrt(dh) scale folded in).
// K/V tiles of 64 keys are double-buffered in shared memory with cp.async (16-byte
// chunks, XOR-swizzled so ldmatrix reads are conflict-free); S = Q K^T and O += P V use
// bf16 m16n8k16 tensor-core MMAs with fp32 accumulation.
#include "kernels.h"

namespace {
constexpr int BQ = 64, BKV = 64, NT = 128;

__device__ __forceinline__ int swz(int row, int col, int dh) {
  // element offset of (row, col) in a [rows][dh] bf16 tile, 16-byte chunks XOR row%8
  const int chunk = (col >> 3) ^ (row & 7);
  return row * dh + (chunk << 3) + (col & 7);
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Loads rows [r0, r0 + 64) of a [L][ld] bf16 matrix (columns col0..col0+DH) into a
// swizzled tile; rows >= L are zero-filled.
template <int DH>
__device__ __forceinline__ void load_tile(bf16* tile, const bf16* base, int ld, int r0, int L) {
  constexpr int CH = DH / 8;  // 16-byte chunks per row
  for (int i = threadIdx.x; i < 64 * CH; i += NT) {
    const int r = i / CH, ch = i % CH;
    const bool ok = (r0 + r) < L;
    const bf16* src = base + (size_t)(ok ? r0 + r : 0) * ld + ch * 8;
    cp_async16(tile + swz(r, ch * 8, DH), src, ok);
  }
}

template <int DH>
__global__ void __launch_bounds__(NT) flash_attn_kernel(AttnArgs a, float scale_log2) {
  griddep_wait();
  griddep_launch();
  extern __shared__ __align__(128) uint8_t smem_raw[];
  bf16* Qs = reinterpret_cast<bf16*>(smem_raw);
  bf16* Ks = Qs + BQ * DH;        // [2][BKV][DH]
  bf16* Vs = Ks + 2 * BKV * DH;   // [2][BKV][DH]

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int g = lane >> 2, c = lane & 3;
  const int q0 = blockIdx.x * BQ, h = blockIdx.y, b = blockIdx.z;
  const bf16* Qb = a.Q + (size_t)b * a.Lq * a.ldq + h * DH;
  const bf16* Kb = a.K + (size_t)b * a.kv_batch_rows * a.ldk + h * DH;
  const bf16* Vb = a.V + (size_t)b * a.kv_batch_rows * a.ldv + h * DH;
  bf16* Ob = a.O + (size_t)b * a.Lq * a.ldo + h * DH;
  const int n_tiles = (a.Lkv + BKV - 1) / BKV;

  load_tile<DH>(Qs, Qb, a.ldq, q0, a.Lq);
  load_tile<DH>(Ks, Kb, a.ldk, 0, a.Lkv);
  load_tile<DH>(Vs, Vb, a.ldv, 0, a.Lkv);
  cp_commit();
  cp_wait<0>();
  __syncthreads();

  uint32_t qf[DH / 16][4];
#pragma unroll
  for (int kk = 0; kk < DH / 16; ++kk) {
    const int row = warp * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
    const int col = kk * 16 + 8 * (lane >> 4);
    ldsm_x4(qf[kk], Qs + swz(row, col, DH));
  }

  float o[DH / 8][4];
#pragma unroll
  for (int j = 0; j < DH / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};

  for (int it = 0; it < n_tiles; ++it) {
    const int buf = it & 1;
    if (it + 1 < n_tiles) {
      load_tile<DH>(Ks + (buf ^ 1) * BKV * DH, Kb, a.ldk, (it + 1) * BKV, a.Lkv);
      load_tile<DH>(Vs + (buf ^ 1) * BKV * DH, Vb, a.ldv, (it + 1) * BKV, a.Lkv);
      cp_commit();
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    const bf16* Kt = Ks + buf * BKV * DH;
    const bf16* Vt = Vs + buf * BKV * DH;

    // S = Q K^T for this warp's 16 rows x 64 keys
    float s[BKV / 8][4];
#pragma unroll
    for (int j = 0; j < BKV / 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DH / 16; ++kk) {
#pragma unroll
      for (int j = 0; j < BKV / 8; j += 2) {
        uint32_t kb[4];
        const int key = j * 8 + (lane & 7) + 8 * (lane >> 4);
        const int col = kk * 16 + 8 * ((lane >> 3) & 1);
        ldsm_x4(kb, Kt + swz(key, col, DH));
        mma16816(s[j], qf[kk], kb[0], kb[1]);
        mma16816(s[j + 1], qf[kk], kb[2], kb[3]);
      }
    }
    // scale, mask the ragged tail, online softmax
    const int kv0 = it * BKV;
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int j = 0; j < BKV / 8; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kv0 + j * 8 + 2 * c + (e & 1);
        float v = s[j][e] * scale_log2;
        if (key >= a.Lkv) v = -INFINITY;
        s[j][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    float alpha[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      const float m_new = fmaxf(m_run[r], mx[r]);
      alpha[r] = exp2f(m_run[r] - m_new);
      m_run[r] = m_new;
      l_run[r] *= alpha[r];
    }
#pragma unroll
    for (int j = 0; j < BKV / 8; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(s[j][e] - m_run[e >> 1]);
        s[j][e] = p;
        l_run[e >> 1] += p;
      }
#pragma unroll
    for (int j = 0; j < DH / 8; ++j) {
      o[j][0] *= alpha[0]; o[j][1] *= alpha[0];
      o[j][2] *= alpha[1]; o[j][3] *= alpha[1];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < BKV / 16; ++kk) {
      uint32_t pf[4];
      pf[0] = pack_bf16x2(s[2 * kk][0], s[2 * kk][1]);
      pf[1] = pack_bf16x2(s[2 * kk][2], s[2 * kk][3]);
      pf[2] = pack_bf16x2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pf[3] = pack_bf16x2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int jd = 0; jd < DH / 8; jd += 2) {
        uint32_t vb[4];
        const int key = kk * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
        const int col = jd * 8 + 8 * (lane >> 4);
        ldsm_x4_t(vb, Vt + swz(key, col, DH));
        mma16816(o[jd], pf, vb[0], vb[1]);
        mma16816(o[jd + 1], pf, vb[2], vb[3]);
      }
    }
    __syncthreads();
  }

  // normalise and store
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
  }
  const float inv0 = 1.f / l_run[0], inv1 = 1.f / l_run[1];
  const int row0 = q0 + warp * 16 + g, row1 = row0 + 8;
#pragma unroll
  for (int j = 0; j < DH / 8; ++j) {
    const int col = j * 8 + 2 * c;
    if (row0 < a.Lq)
      *reinterpret_cast<uint32_t*>(Ob + (size_t)row0 * a.ldo + col) =
          pack_bf16x2(o[j][0] * inv0, o[j][1] * inv0);
    if (row1 < a.Lq)
      *reinterpret_cast<uint32_t*>(Ob + (size_t)row1 * a.ldo + col) =
          pack_bf16x2(o[j][2] * inv1, o[j][3] * inv1);
  }
}

template <int DH>
cudaError_t launch(const AttnArgs& a, cudaStream_t st) {
  const int smem = (BQ + 4 * BKV) * DH * (int)sizeof(bf16);
  cudaError_t e = cudaFuncSetAttribute(flash_attn_kernel<DH>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.Lq + BQ - 1) / BQ, a.heads, a.batch);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
  cudaError_t le = launch_k(flash_attn_kernel<DH>, grid, dim3(NT), smem, st, a, scale_log2);
  if (le != cudaSuccess) return le;
  return cudaGetLastError();
}
}  // namespace

cudaError_t attention(const AttnArgs& a, cudaStream_t st) {
  if (a.Lq < 1 || a.Lkv < 1 || a.batch < 1 || a.heads < 1) return cudaErrorInvalidValue;
  if (a.ldq % 8 || a.ldk % 8 || a.ldv % 8 || a.ldo % 8) return cudaErrorInvalidValue;
  if (a.head_dim == 128) return launch<128>(a, st);
  if (a.head_dim == 64) return launch<64>(a, st);
  return cudaErrorInvalidValue;
}
