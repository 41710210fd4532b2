// CUDA-core GEMM: out[M][N] = epilogue(A[M][K] * W[N][K]^T), for shapes the tcgen05
// kernel does not tile (N not a multiple of 128 or K not a multiple of 64). Any M and K;
// N a multiple of 8. 64 x 64 output tile per CTA, 256 threads, each 2 rows x 8 columns.
#include "kernels.h"

namespace {
constexpr int TM = 64, TN = 64, TK = 32;

template <int KIND>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const bf16* __restrict__ A, int lda,
                                                        const bf16* __restrict__ W, int ldw,
                                                        int M, int N, int K, GemmEpi epi) {
  griddep_wait();
  griddep_launch();
  __shared__ float As[TK][TM + 1];
  __shared__ float Ws[TK][TN + 1];
  const int tid = threadIdx.x;
  const int ty = tid / 8, tx = tid % 8;  // rows ty, ty + 32; columns tx*8 .. tx*8+7
  const int m0 = blockIdx.y * TM, n0 = blockIdx.x * TN;
  float acc[2][8] = {};
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int i = tid; i < TM * TK; i += 256) {
      const int r = i / TK, k = i % TK;
      const int gm = m0 + r, gk = k0 + k;
      As[k][r] = (gm < M && gk < K) ? __bfloat162float(A[(size_t)gm * lda + gk]) : 0.f;
      const int gn = n0 + r;
      Ws[k][r] = (gn < N && gk < K) ? __bfloat162float(W[(size_t)gn * ldw + gk]) : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int k = 0; k < TK; ++k) {
      const float a0 = As[k][ty], a1 = As[k][ty + 32];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float w = Ws[k][tx * 8 + j];
        acc[0][j] += a0 * w;
        acc[1][j] += a1 * w;
      }
    }
    __syncthreads();
  }
  const int col = n0 + tx * 8;
  if (col >= N) return;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int row = m0 + ty + 32 * i;
    if (row < M) epi_apply8<KIND>(epi, row, col, acc[i]);
  }
}
}  // namespace

cudaError_t gemm_simt(const GemmArgs& g, cudaStream_t st) {
  if (g.N % 8 != 0 || g.M < 1 || g.K < 1) return cudaErrorInvalidValue;
  dim3 grid((g.N + TN - 1) / TN, (g.M + TM - 1) / TM);
  switch (g.kind) {
    case EPI_BF16:
      return launch_k(gemm_simt_kernel<EPI_BF16>, grid, dim3(256), 0, st, g.A, g.lda, g.W, g.ldw, g.M, g.N, g.K, g.epi);
      break;
    case EPI_GELU_BF16:
      return launch_k(gemm_simt_kernel<EPI_GELU_BF16>, grid, dim3(256), 0, st, g.A, g.lda, g.W, g.ldw, g.M, g.N, g.K, g.epi);
      break;
    case EPI_RESID:
      return launch_k(gemm_simt_kernel<EPI_RESID>, grid, dim3(256), 0, st, g.A, g.lda, g.W, g.ldw, g.M, g.N, g.K, g.epi);
      break;
    case EPI_RESID_DELTA:
      return launch_k(gemm_simt_kernel<EPI_RESID_DELTA>, grid, dim3(256), 0, st, g.A, g.lda, g.W, g.ldw, g.M, g.N, g.K, g.epi);
      break;
    default:
      return cudaErrorInvalidValue;
  }
}
