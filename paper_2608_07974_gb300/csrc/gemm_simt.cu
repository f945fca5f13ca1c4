// CUDA-core GEMM with fp32 accumulation: the fp32 path (the tiny fp32 workload needs fp32
// accuracy, which rules out TF32 tensor cores) and the reference the tensor-core GEMM is tested
// against. Row-major operands; the three modes of ops.h.
#include <type_traits>

#include "common.cuh"
#include "ops.h"

namespace zl {

namespace {
constexpr int BM = 64, BN = 64, BK = 16;

template <typename T, int MODE>
__device__ __forceinline__ float ldA(const T* A, int M, int K, int m, int k) {
  if (m >= M || k >= K) return 0.f;
  return MODE == 2 ? to_f(A[(size_t)k * M + m]) : to_f(A[(size_t)m * K + k]);
}
template <typename T, int MODE>
__device__ __forceinline__ float ldB(const T* B, int N, int K, int k, int n) {
  if (n >= N || k >= K) return 0.f;
  return MODE == 0 ? to_f(B[(size_t)n * K + k]) : to_f(B[(size_t)k * N + n]);
}

template <typename T, typename TC, int MODE>
__global__ void __launch_bounds__(256) gemm_simt_k(int M, int N, int K, const T* __restrict__ A,
                                                   const T* __restrict__ B, TC* C,
                                                   const float* __restrict__ bias, const TC* R, float alpha,
                                                   int rmode) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int bm = blockIdx.y * BM, bn = blockIdx.x * BN;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += BK) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int e = tid + 256 * r;
      if (MODE == 2) { const int k = e / BM, m = e % BM; As[k][m] = ldA<T, MODE>(A, M, K, bm + m, k0 + k); }
      else { const int m = e / BK, k = e % BK; As[k][m] = ldA<T, MODE>(A, M, K, bm + m, k0 + k); }
      if (MODE == 0) { const int n = e / BK, k = e % BK; Bs[k][n] = ldB<T, MODE>(B, N, K, k0 + k, bn + n); }
      else { const int k = e / BN, n = e % BN; Bs[k][n] = ldB<T, MODE>(B, N, K, k0 + k, bn + n); }
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < BK; ++k) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = As[k][ty + 16 * i]; b[i] = Bs[k][tx + 16 * i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = bm + ty + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = bn + tx + 16 * j;
      if (n >= N) continue;
      const size_t o = (size_t)m * N + n;
      float v = alpha * acc[i][j];
      if (MODE == 2) {
        reinterpret_cast<float*>(C)[o] += v;
      } else {
        if (bias) v += bias[n];
        if (R) v = rmode ? v * gelu_tanh_grad(to_f(R[o]), std::is_same<TC, bf16>::value) : v + to_f(R[o]);
        C[o] = from_f<TC>(v);
      }
    }
  }
}

template <typename T>
void gemm_simt_t(int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias,
                 const void* R, cudaStream_t s, float alpha, int rmode) {
  dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM), block(256);
  if (mode == 0)
    gemm_simt_k<T, T, 0><<<grid, block, 0, s>>>(M, N, K, (const T*)A, (const T*)B, (T*)C, bias, (const T*)R, alpha,
                                                 rmode);
  else if (mode == 1)
    gemm_simt_k<T, T, 1><<<grid, block, 0, s>>>(M, N, K, (const T*)A, (const T*)B, (T*)C, bias, (const T*)R,
                                                 alpha, rmode);
  else
    gemm_simt_k<T, float, 2><<<grid, block, 0, s>>>(M, N, K, (const T*)A, (const T*)B, (float*)C, nullptr, nullptr,
                                                    alpha, 0);
}
}  // namespace

void gemm_simt(int dt, int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias,
               const void* R, cudaStream_t s, float alpha, int rmode) {
  note_launch(1);
  if (M <= 0 || N <= 0) return;
  if (dt == BF16) gemm_simt_t<bf16>(mode, M, N, K, A, B, C, bias, R, s, alpha, rmode);
  else gemm_simt_t<float>(mode, M, N, K, A, B, C, bias, R, s, alpha, rmode);
}

}  // namespace zl

namespace zl {
// GEMM dispatch: the tensor-core kernel where it applies, else the CUDA-core kernel.
void gemm(int dt, int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias,
          const void* R, cudaStream_t s, unsigned* err, cudaMemPool_t pool, float alpha, int rmode) {
  if (dt == BF16 && gemm_tc(mode, M, N, K, A, B, C, bias, R, err, s, pool, alpha, rmode)) return;
  gemm_simt(dt, mode, M, N, K, A, B, C, bias, R, s, alpha, rmode);
}
}  // namespace zl
