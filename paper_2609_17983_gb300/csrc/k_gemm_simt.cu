// k_gemm_simt.cu -- FFMA GEMM Y[M][N] (+)= X[M][K] W[N][K]^T (+ bias), fp32
// accumulation.  Serves the fp32 model (whose 1e-4 parity rules out TF32
// tensor cores) and shapes the tensor-core GEMM does not take.
#include "kvr_internal.cuh"

namespace kvr {
namespace {

template <typename T>
__device__ __forceinline__ float ldv(const T *p, size_t i);
template <>
__device__ __forceinline__ float ldv<float>(const float *p, size_t i) { return p[i]; }
template <>
__device__ __forceinline__ float ldv<__nv_bfloat16>(const __nv_bfloat16 *p, size_t i) {
  return __bfloat162float(p[i]);
}

constexpr int BM = 64, BN = 64, BK = 32;

// 256 threads; thread (ty, tx) of a 16x16 grid owns a 4x4 block of outputs.
template <typename T>
__global__ void __launch_bounds__(256)
    k_gemm_simt(const T *X, const T *W, const float *bias, float *Y, int M, int N, int K, int ldx,
                int ldy, int accumulate) {
  __shared__ float Xs[BK][BM + 4];
  __shared__ float Ws[BK][BN + 4];
  int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += BK) {
    for (int e = threadIdx.x; e < BM * BK; e += 256) {
      int r = e / BK, kk = e % BK, m = m0 + r, k = k0 + kk;
      Xs[kk][r] = (m < M && k < K) ? ldv(X, (size_t)m * ldx + k) : 0.f;
    }
    for (int e = threadIdx.x; e < BN * BK; e += 256) {
      int r = e / BK, kk = e % BK, n = n0 + r, k = k0 + kk;
      Ws[kk][r] = (n < N && k < K) ? ldv(W, (size_t)n * K + k) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < BK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = Xs[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Ws[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] += a[i] * b[j];
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int m = m0 + ty * 4 + i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int n = n0 + tx * 4 + j;
      if (n >= N) continue;
      float v = acc[i][j] + (bias ? bias[n] : 0.f);
      float *y = Y + (size_t)m * ldy + n;
      *y = accumulate ? *y + v : v;
    }
  }
}

}  // namespace

void launch_gemm_simt(const GemmArgs &g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return;
  dim3 grid((g.N + BN - 1) / BN, (g.M + BM - 1) / BM);
  if (g.dtype == KVR_DTYPE_BF16)
    k_gemm_simt<<<grid, 256, 0, s>>>((const __nv_bfloat16 *)g.X, (const __nv_bfloat16 *)g.W,
                                     g.bias, g.Y, g.M, g.N, g.K, g.ldx, g.ldy, g.accumulate);
  else
    k_gemm_simt<<<grid, 256, 0, s>>>((const float *)g.X, (const float *)g.W, g.bias, g.Y, g.M,
                                     g.N, g.K, g.ldx, g.ldy, g.accumulate);
}

}  // namespace kvr
