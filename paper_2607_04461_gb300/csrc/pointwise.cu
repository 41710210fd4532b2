// Memory-bound and small kernels of the draft path:
//  ln_mod       adaLN: LayerNorm (no affine) * (1 + scale) + shift, or affine LN; fp32 in,
//               bf16 out (feeds the next GEMM). Row held in registers: one HBM read.
//  qk_norm_rope RMSNorm of q / k over the model width, then 2-D axial RoPE, in place.
//  proxy_add    activation proxy (Eqs. 3-5 as a linear combination of cached block
//               contributions): h += sum_t c_t Delta_t, one read and write of h per run.
//  patch_embed  2x2 patchify + linear (D x C p p), writes the fp32 residual stream.
//  head_euler   output projection D -> C p p, unpatchify and the Euler step
//               z += (t' - t) v of dx = v dt, fused (CUDA cores, any C p p).
//  patchify     z -> bf16 patch rows, the A operand of the tensor-core patch embedding.
//  euler_step   the step of head_euler from the tensor-core head GEMM's output.
//  gemv, timestep_sincos, mod_prepare, f32_to_bf16: per-step conditioning, conversions.
#include "kernels.h"

namespace {

template <int THREADS>
__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if (THREADS > 32) {
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    v = 0.f;
#pragma unroll
    for (int w = 0; w < THREADS / 32; ++w) v += red[w];
  }
  return v;
}

// ---------------------------------------------------------------------------------
// ln_mod: THREADS threads per row, VPT float4 per thread (D = 4 * VPT * THREADS), ROWS
// rows per block (ROWS > 1 only with one warp per row).
template <int THREADS, int VPT, int ROWS = 1>
__global__ void __launch_bounds__(THREADS * ROWS) ln_mod_kernel(const float* __restrict__ x,
                                                                bf16* __restrict__ out, int rows,
                                                                int D, float eps, float mul_base,
                                                                const float* __restrict__ mul,
                                                                const float* __restrict__ add) {
  static_assert(ROWS == 1 || THREADS == 32, "several rows per block need one warp per row");
  griddep_wait();
  griddep_launch();
  __shared__ float red[THREADS / 32 > 0 ? THREADS / 32 : 1];
  const size_t row = (size_t)blockIdx.x * ROWS + threadIdx.x / THREADS;
  if (row >= (size_t)rows) return;
  const int tid = threadIdx.x % THREADS;
  const float* xr = x + row * D;
  float4 v[VPT];
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    v[i] = *reinterpret_cast<const float4*>(xr + (i * THREADS + tid) * 4);
    s += v[i].x + v[i].y + v[i].z + v[i].w;
  }
  const float mean = block_sum<THREADS>(s, red) / D;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    const float a = v[i].x - mean, b = v[i].y - mean, c = v[i].z - mean, d = v[i].w - mean;
    q += a * a + b * b + c * c + d * d;
  }
  const float rstd = rsqrtf(block_sum<THREADS>(q, red) / D + eps);
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    const int col = (i * THREADS + tid) * 4;
    const float4 m = *reinterpret_cast<const float4*>(mul + col);
    const float4 ad = *reinterpret_cast<const float4*>(add + col);
    const float y0 = (v[i].x - mean) * rstd * (mul_base + m.x) + ad.x;
    const float y1 = (v[i].y - mean) * rstd * (mul_base + m.y) + ad.y;
    const float y2 = (v[i].z - mean) * rstd * (mul_base + m.z) + ad.z;
    const float y3 = (v[i].w - mean) * rstd * (mul_base + m.w) + ad.w;
    uint2 u;
    u.x = pack_bf16x2(y0, y1);
    u.y = pack_bf16x2(y2, y3);
    *reinterpret_cast<uint2*>(out + row * D + col) = u;
  }
}

template <int THREADS, int VPT, int ROWS = 1>
cudaError_t ln_mod_launch(const float* x, bf16* out, int rows, int D, float eps, float mb,
                          const float* mul, const float* add, cudaStream_t st) {
  return launch_k(ln_mod_kernel<THREADS, VPT, ROWS>, dim3((rows + ROWS - 1) / ROWS),
                  dim3(THREADS * ROWS), 0, st, x, out, rows, D, eps, mb, mul, add);
}

// ---------------------------------------------------------------------------------
// qk_norm_rope: THREADS threads per (row, segment), VPT chunks of 4 bf16 per thread, ROWS
// rows per block (ROWS > 1 only with one warp per row).
__device__ __forceinline__ void load_bf16x4(const bf16* p, float* v) {
  uint2 u = *reinterpret_cast<const uint2*>(p);
  float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
  v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
}
__device__ __forceinline__ void store_bf16x4(bf16* p, const float* v) {
  uint2 u;
  u.x = pack_bf16x2(v[0], v[1]);
  u.y = pack_bf16x2(v[2], v[3]);
  *reinterpret_cast<uint2*>(p) = u;
}

template <int THREADS, int VPT, int ROWS>
__global__ void __launch_bounds__(THREADS * ROWS) qk_norm_rope_kernel(
    bf16* __restrict__ x, int rows, int ld, int D, int col0, const float* __restrict__ w0,
    int col1, const float* __restrict__ w1, float eps, const float2* __restrict__ rope,
    int tokens, int head_dim) {
  static_assert(ROWS == 1 || THREADS == 32, "several rows per block need one warp per row");
  griddep_wait();
  griddep_launch();
  __shared__ float red[THREADS / 32 > 0 ? THREADS / 32 : 1];
  const size_t row = (size_t)blockIdx.x * ROWS + threadIdx.x / THREADS;
  if (row >= (size_t)rows) return;
  const int tid = threadIdx.x % THREADS;
  const int seg = blockIdx.y;
  const int col0s = seg ? col1 : col0;
  const float* w = seg ? w1 : w0;
  bf16* xr = x + row * ld + col0s;
  float v[VPT][4];
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    load_bf16x4(xr + (i * THREADS + tid) * 4, v[i]);
#pragma unroll
    for (int j = 0; j < 4; ++j) ss += v[i][j] * v[i][j];
  }
  const float r = rsqrtf(block_sum<THREADS>(ss, red) / D + eps);
  const float2* rp = rope ? rope + (size_t)(row % tokens) * (head_dim / 2) : nullptr;
#pragma unroll
  for (int i = 0; i < VPT; ++i) {
    const int col = (i * THREADS + tid) * 4;
    const float4 wv = *reinterpret_cast<const float4*>(w + col);
    v[i][0] *= r * wv.x; v[i][1] *= r * wv.y; v[i][2] *= r * wv.z; v[i][3] *= r * wv.w;
    if (rp) {
      const int d0 = col % head_dim;  // a chunk never straddles a head (head_dim % 4 == 0)
#pragma unroll
      for (int j = 0; j < 4; j += 2) {
        const float2 cs = rp[(d0 + j) >> 1];
        const float a = v[i][j], b = v[i][j + 1];
        v[i][j] = a * cs.x - b * cs.y;
        v[i][j + 1] = a * cs.y + b * cs.x;
      }
    }
    store_bf16x4(xr + col, v[i]);
  }
}

template <int THREADS, int VPT, int ROWS = 1>
cudaError_t qkn_launch(bf16* x, int rows, int ld, int D, int nseg, int col0, const float* w0,
                       int col1, const float* w1, float eps, const float2* rope, int tokens,
                       int head_dim, cudaStream_t st) {
  dim3 grid((rows + ROWS - 1) / ROWS, nseg);
  return launch_k(qk_norm_rope_kernel<THREADS, VPT, ROWS>, grid, dim3(THREADS * ROWS), 0, st, x,
                  rows, ld, D, col0, w0, col1, w1, eps, rope, tokens, head_dim);
}

// ---------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) proxy_add_kernel(float* __restrict__ h, size_t n8,
                                                        ProxyTerms t) {
  griddep_wait();
  griddep_launch();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n8;
       i += (size_t)gridDim.x * blockDim.x) {
    float acc[8];
    load_f32x8(h + i * 8, acc);
    for (int k = 0; k < t.n; ++k) {
      float a[8];
      load_bf16x8(t.ptr[k] + i * 8, a);
      const float c = t.coef[k];
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] += c * a[j];
    }
    store_f32x8(h + i * 8, acc);
  }
}

// ---------------------------------------------------------------------------------
// patch_embed: 32 tokens per CTA, 256 threads; thread owns output columns n = tid + 256 k.
constexpr int PE_TOK = 32;
__global__ void __launch_bounds__(256) patch_embed_kernel(const float* __restrict__ z, int n,
                                                          int C, int H, int W, int p,
                                                          const bf16* __restrict__ Wp,
                                                          const float* __restrict__ bp, int D,
                                                          float* __restrict__ h) {
  griddep_wait();
  griddep_launch();
  extern __shared__ float xs[];  // [PE_TOK][PD]
  const int PD = C * p * p, gw = W / p, P = (H / p) * gw;
  const int M = n * P;
  const int tok0 = blockIdx.x * PE_TOK;
  for (int i = threadIdx.x; i < PE_TOK * PD; i += blockDim.x) {
    const int t = i / PD, k = i % PD;
    const int tok = tok0 + t;
    float val = 0.f;
    if (tok < M) {
      const int b = tok / P, pt = tok % P, r = pt / gw, cc = pt % gw;
      const int ch = k / (p * p), dy = (k / p) % p, dx = k % p;
      val = z[(((size_t)b * C + ch) * H + r * p + dy) * W + cc * p + dx];
    }
    xs[i] = val;
  }
  __syncthreads();
  for (int col = threadIdx.x; col < D; col += blockDim.x) {
    float acc[PE_TOK];
    const float bias = bp[col];
#pragma unroll
    for (int t = 0; t < PE_TOK; ++t) acc[t] = bias;
    for (int k0 = 0; k0 < PD; k0 += 8) {
      float wv[8];
      load_bf16x8(Wp + (size_t)col * PD + k0, wv);
#pragma unroll
      for (int t = 0; t < PE_TOK; ++t)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[t] += wv[j] * xs[t * PD + k0 + j];
    }
#pragma unroll
    for (int t = 0; t < PE_TOK; ++t)
      if (tok0 + t < M) h[(size_t)(tok0 + t) * D + col] = acc[t];
  }
}

// ---------------------------------------------------------------------------------
// patchify: the patch rows of z in bf16, the A operand of the tensor-core patch
// embedding. Thread -> 8 consecutive columns (ch, dy, dx) of one row (b P + token).
__global__ void __launch_bounds__(256) patchify_kernel(const float* __restrict__ z, int n, int C,
                                                       int H, int W, int p,
                                                       bf16* __restrict__ out) {
  griddep_wait();
  griddep_launch();
  const int PD = C * p * p, gw = W / p, P = (H / p) * gw, pp = p * p;
  const size_t total = (size_t)n * P * (PD / 8);
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    const size_t row = i / (PD / 8);
    const int k0 = (int)(i % (PD / 8)) * 8;
    const int b = (int)(row / P), pt = (int)(row % P), r = pt / gw, cc = pt % gw;
    float v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int k = k0 + j, ch = k / pp, dy = (k / p) % p, dx = k % p;
      v[j] = z[(((size_t)b * C + ch) * H + r * p + dy) * W + cc * p + dx];
    }
    store_bf16x8(out + row * PD + k0, v);
  }
}

// euler_step: the guidance combination and the ODE / SDE step of head_euler, from the
// head output v[row][o] (bias included) of the tensor-core head GEMM, fused with the next
// step's conditioning inputs: the bf16 patch rows of the updated z (the A operand of the
// next patch embedding) and the sinusoidal embedding of the next t. One block per token
// row (p latent rows) of one candidate: threads walk the latent in memory order (each
// element reads output o = (ch, y % p, x % p) of token x / p), then the updated values
// leave through a shared-memory tile [token][o] as whole 16-byte patch-row chunks.
__device__ __forceinline__ void sincos_entry(float t, int k, int half, float* emb) {
  // f_k = 10000^(-k/half); the argument is formed in double for accuracy at 1000 t
  const double f = exp(-9.210340371976184 * (double)k / (double)half);
  const double arg = 1000.0 * (double)t * f;
  emb[k] = (float)cos(arg);
  emb[half + k] = (float)sin(arg);
}

__global__ void __launch_bounds__(256) euler_step_kernel(const float* __restrict__ v, int ldv,
                                                         int n, int C, int H, int W, int p,
                                                         HeadStep hs, float* __restrict__ z) {
  extern __shared__ float tile[];  // [W / p tokens][C p p] when hs.patch_next
  griddep_wait();
  griddep_launch();
  const int PD = C * p * p, gw = W / p, gh = H / p, P = gh * gw;
  const int r = blockIdx.x % gh, b = blockIdx.x / gh;  // token row r of candidate b
  if (hs.emb_next && blockIdx.x == 0) {
    const int half = hs.freq_dim / 2;
    for (int k = threadIdx.x; k < half; k += blockDim.x)
      sincos_entry(hs.t_next, k, half, hs.emb_next);
  }
  const size_t tok0 = (size_t)b * P + (size_t)r * gw;  // first token of the row
  const int row_elems = C * p * W;                      // (ch, dy, x) of the p latent rows
  for (int e = threadIdx.x; e < row_elems; e += blockDim.x) {
    const int x = e % W, dy = (e / W) % p, ch = e / (W * p);
    const size_t zi = (((size_t)b * C + ch) * H + (size_t)r * p + dy) * W + x;
    const int tok = x / p, o = (ch * p + dy) * p + x % p;
    float vv = v[(tok0 + tok) * ldv + o];
    if (hs.uncond_rows) {
      const float vu = v[(tok0 + tok + hs.uncond_rows) * ldv + o];
      vv = vu + hs.w * (vv - vu);
    }
    const float zo = z[zi];
    const float zn = hs.noise ? zo + (vv + hs.sde_c * (zo + (1.f - hs.t) * vv)) * hs.dt +
                                    hs.nscale * hs.noise[zi]
                              : zo + hs.dt * vv;
    z[zi] = zn;
    if (hs.patch_next) tile[tok * PD + o] = zn;
  }
  if (!hs.patch_next) return;
  __syncthreads();
  for (int c = threadIdx.x; c < gw * (PD / 8); c += blockDim.x) {
    const int tok = c / (PD / 8), o0 = (c % (PD / 8)) * 8;
    store_bf16x8(hs.patch_next + (tok0 + tok) * PD + o0, tile + tok * PD + o0);
  }
}

// ---------------------------------------------------------------------------------
// head_euler: 32 tokens per CTA, 256 threads; K staged through shared memory in
// chunks of 64. Thread -> output o = tid % PD and TPT = 32 PD / 256 consecutive tokens.
// With guidance each thread also accumulates the unconditional row of its tokens.
constexpr int HE_TOK = 32, HE_KC = 64;
template <int PD, bool GUIDED>
__global__ void __launch_bounds__(256) head_euler_kernel(const bf16* __restrict__ a, int n,
                                                         int C, int H, int W, int p,
                                                         const bf16* __restrict__ Wh,
                                                         const float* __restrict__ bh, int D,
                                                         HeadStep hs, float* __restrict__ z) {
  griddep_wait();
  griddep_launch();
  constexpr int TPT = HE_TOK * PD / 256;
  __shared__ float as[2][HE_TOK][HE_KC + 1];
  __shared__ float ws[PD][HE_KC + 1];
  const int gw = W / p, P = (H / p) * gw, M = n * P;
  constexpr bool guided = GUIDED;
  const int tok0 = blockIdx.x * HE_TOK;
  const int o = threadIdx.x % PD, grp = threadIdx.x / PD;
  float acc[TPT], accu[TPT];
#pragma unroll
  for (int i = 0; i < TPT; ++i) acc[i] = accu[i] = 0.f;
  for (int k0 = 0; k0 < D; k0 += HE_KC) {
    __syncthreads();
    for (int i = threadIdx.x; i < (GUIDED ? 2 : 1) * HE_TOK * HE_KC / 8; i += 256) {
      const int u = i / (HE_TOK * HE_KC / 8), rem = i % (HE_TOK * HE_KC / 8);
      const int t = rem / (HE_KC / 8), kc = (rem % (HE_KC / 8)) * 8;
      float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      if ((u == 0 || guided) && tok0 + t < M && k0 + kc < D)
        load_bf16x8(a + (size_t)(tok0 + t + u * hs.uncond_rows) * D + k0 + kc, v);
#pragma unroll
      for (int j = 0; j < 8; ++j) as[u][t][kc + j] = v[j];
    }
    for (int i = threadIdx.x; i < PD * HE_KC / 8; i += 256) {
      const int r = i / (HE_KC / 8), kc = (i % (HE_KC / 8)) * 8;
      float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      if (k0 + kc < D) load_bf16x8(Wh + (size_t)r * D + k0 + kc, v);
#pragma unroll
      for (int j = 0; j < 8; ++j) ws[r][kc + j] = v[j];
    }
    __syncthreads();
#pragma unroll 4
    for (int k = 0; k < HE_KC; ++k) {
      const float wv = ws[o][k];
#pragma unroll
      for (int i = 0; i < TPT; ++i) {
        acc[i] += wv * as[0][grp * TPT + i][k];
        if (GUIDED) accu[i] += wv * as[1][grp * TPT + i][k];
      }
    }
  }
  const float bias = bh[o];
  const int ch = o / (p * p), dy = (o / p) % p, dx = o % p;
#pragma unroll
  for (int i = 0; i < TPT; ++i) {
    const int tok = tok0 + grp * TPT + i;
    if (tok < M) {
      float v = acc[i] + bias;
      if (guided) {
        const float vu = accu[i] + bias;
        v = vu + hs.w * (v - vu);
      }
      const int b = tok / P, pt = tok % P, r = pt / gw, cc = pt % gw;
      const size_t zi = (((size_t)b * C + ch) * H + r * p + dy) * W + cc * p + dx;
      const float zo = z[zi];
      if (hs.noise)
        z[zi] = zo + (v + hs.sde_c * (zo + (1.f - hs.t) * v)) * hs.dt + hs.nscale * hs.noise[zi];
      else
        z[zi] = zo + hs.dt * v;
    }
  }
}

// ---------------------------------------------------------------------------------
// gemv: one warp per output row.
__global__ void __launch_bounds__(256) gemv_kernel(const bf16* __restrict__ W,
                                                   const float* __restrict__ b,
                                                   const float* __restrict__ x,
                                                   float* __restrict__ y, int O, int K,
                                                   int act_in, int act_out) {
  griddep_wait();
  griddep_launch();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) / 32, lane = threadIdx.x % 32;
  if (warp >= O) return;
  const bf16* wr = W + (size_t)warp * K;
  float acc = 0.f;
  for (int k = lane * 8; k < K; k += 32 * 8) {
    float wv[8], xv[8];
    load_bf16x8(wr + k, wv);
    load_f32x8(x + k, xv);
#pragma unroll
    for (int j = 0; j < 8; ++j) acc += wv[j] * (act_in ? silu_f(xv[j]) : xv[j]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) {
    float v = acc + (b ? b[warp] : 0.f);
    y[warp] = act_out ? silu_f(v) : v;
  }
}

__global__ void timestep_sincos_kernel(float t, int dim, float* emb) {
  griddep_wait();
  griddep_launch();
  const int half = dim / 2;
  for (int k = threadIdx.x; k < half; k += blockDim.x) sincos_entry(t, k, half, emb);
}

__global__ void mod_prepare_kernel(const float* __restrict__ mod,
                                   const float* __restrict__ tables, int L, int D,
                                   float* __restrict__ modl, const float* __restrict__ htab,
                                   const float* __restrict__ temb, float* __restrict__ head_mod) {
  griddep_wait();
  griddep_launch();
  const size_t n6 = 6 * (size_t)D;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < (size_t)L * n6;
       i += (size_t)gridDim.x * blockDim.x)
    modl[i] = mod[i % n6] + tables[i];
  if (blockIdx.x == 0)
    for (int i = threadIdx.x; i < 2 * D; i += blockDim.x) head_mod[i] = htab[i] + temb[i % D];
}

__global__ void f32_to_bf16_kernel(const float* __restrict__ x, bf16* __restrict__ y, size_t n) {
  griddep_wait();
  griddep_launch();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x)
    y[i] = __float2bfloat16_rn(x[i]);
}

int grid_for(size_t work, int threads) {
  size_t g = (work + threads - 1) / threads;
  const size_t cap = 152 * 16;
  return (int)(g < 1 ? 1 : (g > cap ? cap : g));
}

}  // namespace

// ---- launchers --------------------------------------------------------------------

cudaError_t ln_mod(const float* x, bf16* out, int rows, int D, float eps, float mul_base,
                   const float* mul, const float* add, cudaStream_t st) {
  if (rows == 0) return cudaSuccess;
  switch (D) {  // threads * 4 * VPT == D
    case 128: return ln_mod_launch<32, 1>(x, out, rows, D, eps, mul_base, mul, add, st);
    case 256: return ln_mod_launch<64, 1>(x, out, rows, D, eps, mul_base, mul, add, st);
    case 512: return ln_mod_launch<128, 1>(x, out, rows, D, eps, mul_base, mul, add, st);
    case 1024: return ln_mod_launch<128, 2>(x, out, rows, D, eps, mul_base, mul, add, st);
    // one warp per row, two rows per block, reductions by shuffles only: 5.93 TB/s against
    // 5.44 with 128 threads per row on the 16-candidate probe (24960 rows)
    case 1536: return ln_mod_launch<32, 12, 2>(x, out, rows, D, eps, mul_base, mul, add, st);
    case 2048: return ln_mod_launch<128, 4>(x, out, rows, D, eps, mul_base, mul, add, st);
    case 3072: return ln_mod_launch<256, 3>(x, out, rows, D, eps, mul_base, mul, add, st);
    case 4096: return ln_mod_launch<256, 4>(x, out, rows, D, eps, mul_base, mul, add, st);
    case 5120: return ln_mod_launch<256, 5>(x, out, rows, D, eps, mul_base, mul, add, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t qk_norm_rope(bf16* x, int rows, int ld, int D, int nseg, int col0, const float* w0,
                         int col1, const float* w1, float eps, const float2* rope, int tokens,
                         int head_dim, cudaStream_t st) {
  if (rows == 0) return cudaSuccess;
#define QKN(T, V, ...) \
  qkn_launch<T, V, ##__VA_ARGS__>(x, rows, ld, D, nseg, col0, w0, col1, w1, eps, rope, tokens, head_dim, st)
  switch (D) {  // threads * 4 * VPT == D
    case 128: return QKN(32, 1);
    case 256: return QKN(64, 1);
    case 512: return QKN(128, 1);
    case 1024: return QKN(128, 2);
    // one warp per row (96 bytes in flight per thread), four rows per block: on the
    // 16-candidate probe (24960 rows x 2 x 1536) 5.04 TB/s against 4.90 with two rows
    // per block and 4.60 with eight (at 49920 rows two rows per block gave 6.1 TB/s, one
    // row 5.4)
    case 1536: return QKN(32, 12, 4);
    case 2048: return QKN(128, 4);
    case 3072: return QKN(256, 3);
    case 4096: return QKN(256, 4);
    case 5120: return QKN(256, 5);
  }
#undef QKN
  return cudaErrorInvalidValue;
}

cudaError_t patchify(const float* z, int n, int C, int H, int W, int p, bf16* out,
                     cudaStream_t st) {
  const int PD = C * p * p;
  if (PD % 8 || H % p || W % p) return cudaErrorInvalidValue;
  const size_t work = (size_t)n * (H / p) * (W / p) * (PD / 8);
  if (work == 0) return cudaSuccess;
  return launch_k(patchify_kernel, dim3(grid_for(work, 256)), dim3(256), 0, st, z, n, C, H, W, p,
                  out);
}

cudaError_t euler_step(const float* v, int ldv, int n, int C, int H, int W, int p,
                       const HeadStep& hs, float* z, cudaStream_t st) {
  const int PD = C * p * p;
  if (H % p || W % p || ldv < PD || PD % 8) return cudaErrorInvalidValue;
  const size_t smem = hs.patch_next ? (size_t)(W / p) * PD * sizeof(float) : 0;
  if (smem > 48 * 1024) return cudaErrorInvalidValue;  // one token row's tile
  if (n == 0) return cudaSuccess;
  return launch_k(euler_step_kernel, dim3(n * (H / p)), dim3(256), smem, st, v, ldv, n, C, H, W, p,
                  hs, z);
}

cudaError_t proxy_add(float* h, size_t n_elems, const ProxyTerms& t, cudaStream_t st) {
  if (n_elems == 0 || t.n == 0) return cudaSuccess;
  if (n_elems % 8) return cudaErrorInvalidValue;
  const size_t n8 = n_elems / 8;
  return launch_k(proxy_add_kernel, dim3(grid_for(n8, 256)), dim3(256), 0, st, h, n8, t);
}

cudaError_t patch_embed(const float* z, int n, int C, int H, int W, int p, const bf16* Wp,
                        const float* bp, int D, float* h, cudaStream_t st) {
  const int PD = C * p * p, M = n * (H / p) * (W / p);
  if (M == 0) return cudaSuccess;
  if (PD % 8 || PD > 64) return cudaErrorInvalidValue;
  return launch_k(patch_embed_kernel, dim3((M + PE_TOK - 1) / PE_TOK), dim3(256),
                  PE_TOK * PD * sizeof(float), st, z, n, C, H, W, p, Wp, bp, D, h);
}

cudaError_t head_euler(const bf16* a, int n, int C, int H, int W, int p, const bf16* Wh,
                       const float* bh, int D, const HeadStep& hs, float* z, cudaStream_t st) {
  const int PD = C * p * p, M = n * (H / p) * (W / p);
  if (M == 0) return cudaSuccess;
  if (D % 8) return cudaErrorInvalidValue;
  const dim3 grid((M + HE_TOK - 1) / HE_TOK);
#define HE(PD)                                                                              \
  (hs.uncond_rows > 0                                                                      \
       ? launch_k(head_euler_kernel<PD, true>, grid, dim3(256), 0, st, a, n, C, H, W, p, Wh, \
                  bh, D, hs, z)                                                            \
       : launch_k(head_euler_kernel<PD, false>, grid, dim3(256), 0, st, a, n, C, H, W, p,   \
                  Wh, bh, D, hs, z))
  switch (PD) {
    case 8: return HE(8);
    case 16: return HE(16);
    case 32: return HE(32);
    case 64: return HE(64);
    default: return cudaErrorInvalidValue;
  }
#undef HE
}

cudaError_t gemv(const bf16* W, const float* b, const float* x, float* y, int O, int K,
                 int act_in, int act_out, cudaStream_t st) {
  if (K % 8) return cudaErrorInvalidValue;
  return launch_k(gemv_kernel, dim3((O * 32 + 255) / 256), dim3(256), 0, st, W, b, x, y, O, K,
                  act_in, act_out);
}

cudaError_t timestep_sincos(float t, int dim, float* emb, cudaStream_t st) {
  return launch_k(timestep_sincos_kernel, dim3(1), dim3(128), 0, st, t, dim, emb);
}

cudaError_t mod_prepare(const float* mod, const float* tables, int L, int D, float* modl,
                        const float* htab, const float* temb, float* head_mod, cudaStream_t st) {
  return launch_k(mod_prepare_kernel, dim3(grid_for((size_t)L * 6 * D, 256)), dim3(256), 0, st, mod,
                  tables, L, D, modl, htab, temb, head_mod);
}

cudaError_t f32_to_bf16(const float* x, bf16* y, size_t n, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  return launch_k(f32_to_bf16_kernel, dim3(grid_for(n, 256)), dim3(256), 0, st, x, y, n);
}
