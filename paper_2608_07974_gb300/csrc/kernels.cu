// Memory-bound kernels of the ZeroLock local step: embedding gather, norms, RoPE, activations,
// the fused local objective (Eq. 3-5) and the per-chunk AdamW update.
#include <math.h>

#include <algorithm>
#include <stdlib.h>

#include <type_traits>

#include "common.cuh"
#include "ops.h"

namespace zl {

static inline int grid_for(size_t work, int threads, int max_blocks = 152 * 16) {
  size_t b = (work + threads - 1) / threads;
  if (b < 1) b = 1;
  return (int)(b > (size_t)max_blocks ? (size_t)max_blocks : b);
}

// ------------------------------------------------------------------------------------------
// Embedding gather (Eq. 1: h_0 = E(x)); frozen E (and learned positions P for GPT-2).
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void embed_k(const int32_t* __restrict__ ids, const T* __restrict__ E, const T* __restrict__ P,
                        T* __restrict__ h, int N, int S, int d, int V, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int nv = d / 8;
  const long total = (long)N * nv;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < total; i += (long)gridDim.x * blockDim.x) {
    const int n = (int)(i / nv), c = (int)(i % nv) * 8;
    const int id = ids[n];
    T* dst = h + (size_t)n * d + c;
    if (id < 0 || id >= V) {
      if (c == 0) atomicOr(err, ZL_DEVERR_BAD_ID);
      float f[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      Vec8<T>::store(dst, f);
      continue;
    }
    const T* src = E + (size_t)id * d + c;
    if (P == nullptr) {               // bit-exact row copy
      const uint4* s4 = reinterpret_cast<const uint4*>(src);
      uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
      for (int q = 0; q < (int)(sizeof(T) * 8 / 16); ++q) d4[q] = s4[q];
    } else {
      float a[8], b[8];
      Vec8<T>::load(src, a);
      Vec8<T>::load(P + (size_t)(n % S) * d + c, b);
#pragma unroll
      for (int q = 0; q < 8; ++q) a[q] += b[q];
      Vec8<T>::store(dst, a);
    }
  }
}

void launch_embed(int dt, const int32_t* ids, const void* E, const void* P, void* h, int N, int S, int d,
                  int V, unsigned* err, cudaStream_t s) {
  note_launch(1);
  const int th = 256, g = grid_for((size_t)N * (d / 8), th);
  if (dt == BF16)
    launch_pdl(embed_k<bf16>, g, th, 0, s, ids, (const bf16*)E, (const bf16*)P, (bf16*)h, N, S, d, V, err);
  else
    launch_pdl(embed_k<float>, g, th, 0, s, ids, (const float*)E, (const float*)P, (float*)h, N, S, d, V, err);
}

// ------------------------------------------------------------------------------------------
// RMSNorm / LayerNorm forward and backward (one warp per row, 8-wide vector access, fp32 math).
// ------------------------------------------------------------------------------------------
// 8 consecutive fp32 values (32-byte aligned) as two 16-byte loads.
__device__ __forceinline__ void load8f(const float* p, float* f) {
  const float4 u = reinterpret_cast<const float4*>(p)[0], v = reinterpret_cast<const float4*>(p)[1];
  f[0] = u.x; f[1] = u.y; f[2] = u.z; f[3] = u.w; f[4] = v.x; f[5] = v.y; f[6] = v.z; f[7] = v.w;
}

// Row held in registers (d <= 256 * VPL), one warp per row: one read of x; every load of the row, its
// gains and biases is issued before the reductions, so a warp waits for memory once.
template <typename T, bool LN, int VPL>
__global__ void norm_fwd_reg_k(const T* __restrict__ x, const float* __restrict__ g, const float* __restrict__ b,
                               T* __restrict__ y, float* __restrict__ rstd_o, float* __restrict__ mean_o, int N, int d,
                               float eps) {
  pdl_wait();
  pdl_trigger();
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= N) return;
  const T* xr = x + (size_t)row * d;
  float f[VPL][8], gv[VPL][8], bv[VPL][8];
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane * 8 + v * 256;
    if (c < d) {
      Vec8<T>::load(xr + c, f[v]);
      if (g) load8f(g + c, gv[v]);
      if (LN && b) load8f(b + c, bv[v]);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) f[v][i] = 0.f;
    }
  }
  float s = 0.f;
#pragma unroll
  for (int v = 0; v < VPL; ++v)
#pragma unroll
    for (int i = 0; i < 8; ++i) s += f[v][i];
  const float mean = LN ? warp_sum(s) / d : 0.f;
  float q = 0.f;
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane * 8 + v * 256;
    if (c < d) {
#pragma unroll
      for (int i = 0; i < 8; ++i) { const float t = f[v][i] - mean; q += t * t; }
    }
  }
  const float rstd = 1.f / sqrtf(warp_sum(q) / d + eps);
  T* yr = y + (size_t)row * d;
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane * 8 + v * 256;
    if (c >= d) continue;
    float o[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      o[i] = (f[v][i] - mean) * rstd * (g ? gv[v][i] : 1.f);
      if (LN && b) o[i] += bv[v][i];
    }
    Vec8<T>::store(yr + c, o);
  }
  if (lane == 0) {
    if (rstd_o) rstd_o[row] = rstd;
    if (LN && mean_o) mean_o[row] = mean;
  }
}

// dx = rstd * (dyh - mean(dyh) [LN] - xhat * mean(dyh * xhat)) (+ dres), dyh = g * dy; one warp per row.
template <typename T, bool LN, int VPL>
__global__ void norm_bwd_dx_reg_k(const T* __restrict__ x, const float* __restrict__ g,
                                  const float* __restrict__ rstd, const float* __restrict__ mean,
                                  const T* __restrict__ dy, const T* __restrict__ dres, T* __restrict__ dx, int N,
                                  int d) {
  pdl_wait();
  pdl_trigger();
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= N) return;
  const size_t o = (size_t)row * d;
  const float r = rstd[row], mu = LN ? mean[row] : 0.f;
  float fx[VPL][8], fd[VPL][8], fr[VPL][8];
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane * 8 + v * 256;
    if (c < d) {
      Vec8<T>::load(x + o + c, fx[v]);
      Vec8<T>::load(dy + o + c, fd[v]);
      if (dres) Vec8<T>::load(dres + o + c, fr[v]);
      if (g) {
        float gv[8];
        load8f(g + c, gv);
#pragma unroll
        for (int i = 0; i < 8; ++i) fd[v][i] *= gv[i];
      }
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) fx[v][i] = fd[v][i] = 0.f;
    }
  }
  float s1 = 0.f, s2 = 0.f;
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane * 8 + v * 256;
    if (c >= d) continue;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      fx[v][i] = (fx[v][i] - mu) * r;         // xhat
      s1 += fd[v][i];
      s2 += fd[v][i] * fx[v][i];
    }
  }
  s1 = warp_sum(s1) / d;
  s2 = warp_sum(s2) / d;
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane * 8 + v * 256;
    if (c >= d) continue;
    float out[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      out[i] = r * (fd[v][i] - (LN ? s1 : 0.f) - fx[v][i] * s2);
      if (dres) out[i] += fr[v][i];
    }
    Vec8<T>::store(dx + o + c, out);
  }
}

// One block per row (1024 < d <= 16384): thread t holds vectors t + j * blockDim.x, j < VPT, of the
// row, every load issued before the block reductions.
template <typename T, bool LN, int VPT>
__global__ void __launch_bounds__(512) norm_fwd_blk_k(const T* __restrict__ x, const float* __restrict__ g,
                                                      const float* __restrict__ b, T* __restrict__ y,
                                                      float* __restrict__ rstd_o, float* __restrict__ mean_o, int N,
                                                      int d, float eps) {
  pdl_wait();
  pdl_trigger();
  __shared__ float sh[32];
  const size_t o = (size_t)blockIdx.x * d;
  float f[VPT][8], gv[VPT][8], bv[VPT][8];
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int c = (threadIdx.x + j * blockDim.x) * 8;
    if (c < d) {
      Vec8<T>::load(x + o + c, f[j]);
      if (g) load8f(g + c, gv[j]);
      if (LN && b) load8f(b + c, bv[j]);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) f[j][i] = 0.f;
    }
  }
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < VPT; ++j)
#pragma unroll
    for (int i = 0; i < 8; ++i) sum += f[j][i];
  const float mean = LN ? block_sum(sum, sh) / d : 0.f;
  float q = 0.f;
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    if ((int)(threadIdx.x + j * blockDim.x) * 8 >= d) continue;
#pragma unroll
    for (int i = 0; i < 8; ++i) { const float t = f[j][i] - mean; q += t * t; }
  }
  const float rstd = 1.f / sqrtf(block_sum(q, sh) / d + eps);
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int c = (threadIdx.x + j * blockDim.x) * 8;
    if (c >= d) continue;
    float out[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      out[i] = (f[j][i] - mean) * rstd * (g ? gv[j][i] : 1.f);
      if (LN && b) out[i] += bv[j][i];
    }
    Vec8<T>::store(y + o + c, out);
  }
  if (threadIdx.x == 0) {
    if (rstd_o) rstd_o[blockIdx.x] = rstd;
    if (LN && mean_o) mean_o[blockIdx.x] = mean;
  }
}

template <typename T, bool LN, int VPT>
__global__ void __launch_bounds__(512) norm_bwd_dx_blk_k(const T* __restrict__ x, const float* __restrict__ g,
                                                         const float* __restrict__ rstd,
                                                         const float* __restrict__ mean, const T* __restrict__ dy,
                                                         const T* __restrict__ dres, T* __restrict__ dx, int N,
                                                         int d) {
  pdl_wait();
  pdl_trigger();
  __shared__ float sh[32];
  const size_t o = (size_t)blockIdx.x * d;
  const float r = rstd[blockIdx.x], mu = LN ? mean[blockIdx.x] : 0.f;
  float fx[VPT][8], fd[VPT][8], fr[VPT][8];
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int c = (threadIdx.x + j * blockDim.x) * 8;
    if (c < d) {
      Vec8<T>::load(x + o + c, fx[j]);
      Vec8<T>::load(dy + o + c, fd[j]);
      if (dres) Vec8<T>::load(dres + o + c, fr[j]);
      if (g) {
        float gv[8];
        load8f(g + c, gv);
#pragma unroll
        for (int i = 0; i < 8; ++i) fd[j][i] *= gv[i];
      }
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) fx[j][i] = fd[j][i] = 0.f;
    }
  }
  float s1 = 0.f, s2 = 0.f;
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    if ((int)(threadIdx.x + j * blockDim.x) * 8 >= d) continue;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      fx[j][i] = (fx[j][i] - mu) * r;
      s1 += fd[j][i];
      s2 += fd[j][i] * fx[j][i];
    }
  }
  s1 = LN ? block_sum(s1, sh) / d : 0.f;
  s2 = block_sum(s2, sh) / d;
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int c = (threadIdx.x + j * blockDim.x) * 8;
    if (c >= d) continue;
    float out[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      out[i] = r * (fd[j][i] - s1 - fx[j][i] * s2);
      if (dres) out[i] += fr[j][i];
    }
    Vec8<T>::store(dx + o + c, out);
  }
}

// Threads per block (<= 512) and vectors per thread of the block-per-row kernels: the fewest vectors
// per thread (at most four) that keep a block within `target` threads. The forward takes 128 (small
// blocks: every row of a 2048-row, d = 4096 batch resident at once; 9.7 against 11.0 us), the backward
// 512 (one vector of x, dy and the residual per thread; with four, 18.7 against 14.0 us).
static void blk_shape(int d, int target, int& threads, int& vpt) {
  const int nvec = d / 8;
  vpt = 1;
  while (vpt < 4 && (nvec + vpt - 1) / vpt > target) vpt *= 2;
  threads = ((nvec + vpt - 1) / vpt + 31) / 32 * 32;
}

void launch_norm_fwd(int dt, bool ln, const void* x, const float* g, const float* b, void* y, float* rstd,
                     float* mean, int N, int d, float eps, cudaStream_t s) {
  note_launch(1);
  const int th = 256, blocks = (N * 32 + th - 1) / th;
  const int vpl = (d + 255) / 256;
#define NFR(T, L, V) launch_pdl(norm_fwd_reg_k<T, L, V>, blocks, th, 0, s, (const T*)x, g, b, (T*)y, rstd, mean, N, d, eps)
#define NFV(T, L)                     \
  if (vpl == 1) NFR(T, L, 1);         \
  else if (vpl == 2) NFR(T, L, 2);    \
  else if (vpl == 3) NFR(T, L, 3);    \
  else NFR(T, L, 4);
#define NFB(T, L, V) launch_pdl(norm_fwd_blk_k<T, L, V>, N, bt, 0, s, (const T*)x, g, b, (T*)y, rstd, mean, N, d, eps)
#define NF(T, L)                      \
  if (vpt == 1) NFB(T, L, 1);         \
  else if (vpt == 2) NFB(T, L, 2);    \
  else NFB(T, L, 4);
  if (vpl <= 4) {
    if (dt == BF16) { if (ln) { NFV(bf16, true) } else { NFV(bf16, false) } }
    else { if (ln) { NFV(float, true) } else { NFV(float, false) } }
  } else {
    int bt, vpt;
    blk_shape(d, 128, bt, vpt);
    if (dt == BF16) { if (ln) { NF(bf16, true) } else { NF(bf16, false) } }
    else { if (ln) { NF(float, true) } else { NF(float, false) } }
  }
#undef NF
#undef NFB
#undef NFV
#undef NFR
}

void launch_norm_bwd_dx(int dt, bool ln, const void* x, const float* g, const float* rstd, const float* mean,
                        const void* dy, const void* dres, void* dx, int N, int d, cudaStream_t s) {
  note_launch(1);
  const int th = 256, blocks = (N * 32 + th - 1) / th;
  const int vpl = (d + 255) / 256;
#define NBR(T, L, V)                                                                                             \
  launch_pdl(norm_bwd_dx_reg_k<T, L, V>, blocks, th, 0, s, (const T*)x, g, rstd, mean, (const T*)dy, (const T*)dres, (T*)dx, \
                                                   N, d)
#define NBV(T, L)                     \
  if (vpl == 1) NBR(T, L, 1);         \
  else if (vpl == 2) NBR(T, L, 2);    \
  else if (vpl == 3) NBR(T, L, 3);    \
  else NBR(T, L, 4);
#define NBB(T, L, V)                                                                                          \
  launch_pdl(norm_bwd_dx_blk_k<T, L, V>, N, bt, 0, s, (const T*)x, g, rstd, mean, (const T*)dy, (const T*)dres, (T*)dx, N, d)
#define NB(T, L)                      \
  if (vpt == 1) NBB(T, L, 1);         \
  else if (vpt == 2) NBB(T, L, 2);    \
  else NBB(T, L, 4);
  if (vpl <= 4) {
    if (dt == BF16) { if (ln) { NBV(bf16, true) } else { NBV(bf16, false) } }
    else { if (ln) { NBV(float, true) } else { NBV(float, false) } }
  } else {
    int bt, vpt;
    blk_shape(d, 512, bt, vpt);
    if (dt == BF16) { if (ln) { NB(bf16, true) } else { NB(bf16, false) } }
    else { if (ln) { NB(float, true) } else { NB(float, false) } }
  }
#undef NB
#undef NBB
#undef NBV
#undef NBR
}

static constexpr int kColRows = 64;   // rows per partial-sum block
static constexpr int kColLanes = 8;   // row lanes per block: each thread sums kColRows / kColLanes rows
int colsum_blocks(int N) { return (N + kColRows - 1) / kColRows; }
int colsum_groups(int d) { return (d + 255) / 256; }

// block (32, 8): 32 threads x 8 columns each (256 columns, 16-byte loads) x 8 row lanes;
// grid (colsum_groups(d), colsum_blocks(N)). Requires d % 8 == 0.
// Every row load of a thread is issued before the first add (8 rows, 16 B each, in flight at once).
// After its partial sums, the last block of each 256-column group (one ticket counter per group)
// adds sum_b part[b][c], b in increasing order, into the outputs and re-arms its counter:
// deterministic, one launch, and the final sums of the groups run in parallel.
template <typename T, bool NORM, bool LN>
__global__ void __launch_bounds__(256) colsum_k(const T* __restrict__ A, const T* __restrict__ x,
                                                const float* __restrict__ rstd, const float* __restrict__ mean,
                                                float* __restrict__ part_g, float* __restrict__ part_b, int N,
                                                int d, float* __restrict__ out_g, float* __restrict__ out_b,
                                                unsigned* __restrict__ counters) {
  pdl_wait();
  pdl_trigger();
  constexpr int R = kColRows / kColLanes;
  __shared__ unsigned ticket;
  __shared__ float sg[kColLanes][256], sb[kColLanes][256];
  const int c0 = blockIdx.x * 256 + threadIdx.x * 8;
  const int rb = blockIdx.y * kColRows + threadIdx.y;
  float ag[8] = {0, 0, 0, 0, 0, 0, 0, 0}, ab[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  if (c0 < d) {
    float a[R][8];
#pragma unroll
    for (int j = 0; j < R; ++j) {
      const int r = rb + j * kColLanes;
      if (r < N) Vec8<T>::load(A + (size_t)r * d + c0, a[j]);
      else {
#pragma unroll
        for (int i = 0; i < 8; ++i) a[j][i] = 0.f;
      }
    }
    if (NORM) {
      float xs[R][8], mu[R], rs[R];
#pragma unroll
      for (int j = 0; j < R; ++j) {
        const int r = rb + j * kColLanes;
        if (r < N) {
          Vec8<T>::load(x + (size_t)r * d + c0, xs[j]);
          mu[j] = LN ? mean[r] : 0.f;
          rs[j] = rstd[r];
        } else {
          mu[j] = 0.f;
          rs[j] = 0.f;
#pragma unroll
          for (int i = 0; i < 8; ++i) xs[j][i] = 0.f;
        }
      }
#pragma unroll
      for (int j = 0; j < R; ++j)
#pragma unroll
        for (int i = 0; i < 8; ++i) ag[i] = fmaf(a[j][i], (xs[j][i] - mu[j]) * rs[j], ag[i]);
    }
#pragma unroll
    for (int j = 0; j < R; ++j)
#pragma unroll
      for (int i = 0; i < 8; ++i) ab[i] += a[j][i];
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    sg[threadIdx.y][threadIdx.x * 8 + i] = ag[i];
    sb[threadIdx.y][threadIdx.x * 8 + i] = ab[i];
  }
  __syncthreads();
  const int t = threadIdx.y * 32 + threadIdx.x;   // 256 threads, one column each
  const int c = blockIdx.x * 256 + t;
  if (c < d) {
    float tg = 0.f, tb = 0.f;
#pragma unroll
    for (int i = 0; i < kColLanes; ++i) { tg += sg[i][t]; tb += sb[i][t]; }
    if (NORM) {
      part_g[(size_t)blockIdx.y * d + c] = tg;
      if (LN) part_b[(size_t)blockIdx.y * d + c] = tb;
    } else {
      part_b[(size_t)blockIdx.y * d + c] = tb;
    }
  }
  __threadfence();
  __syncthreads();
  if (t == 0) ticket = atomicAdd(counters + blockIdx.x, 1u);
  __syncthreads();
  if (ticket != gridDim.y - 1) return;
  __threadfence();
  if (c < d) {
    const int nb = gridDim.y;
    float a = 0.f, bsum = 0.f;
    int bb = 0;
    for (; bb + 16 <= nb; bb += 16) {   // 16 loads in flight, added in increasing b
      float vg[16], vb[16];
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        if (NORM) vg[q] = __ldcg(part_g + (size_t)(bb + q) * d + c);
        if (!NORM || LN) vb[q] = __ldcg(part_b + (size_t)(bb + q) * d + c);
      }
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        if (NORM) a += vg[q];
        if (!NORM || LN) bsum += vb[q];
      }
    }
    for (; bb < nb; ++bb) {
      if (NORM) a += __ldcg(part_g + (size_t)bb * d + c);
      if (!NORM || LN) bsum += __ldcg(part_b + (size_t)bb * d + c);
    }
    if (NORM) {
      out_g[c] += a;
      if (LN) out_b[c] += bsum;
    } else {
      out_b[c] += bsum;
    }
  }
  if (t == 0) counters[blockIdx.x] = 0u;
}

void launch_norm_bwd_dparam(int dt, bool ln, const void* x, const float* rstd, const float* mean,
                            const void* dy, float* part_g, float* part_b, int N, int d, float* out_g, float* out_b,
                            unsigned* counters, cudaStream_t s) {
  note_launch(1);
  dim3 grid(colsum_groups(d), colsum_blocks(N)), block(32, kColLanes);
#define CS(T, L)                                                                                             \
  launch_pdl(colsum_k<T, true, L>, grid, block, 0, s, (const T*)dy, (const T*)x, rstd, mean, part_g, part_b, N, d, out_g, \
                                              out_b, counters)
  if (dt == BF16) { if (ln) CS(bf16, true); else CS(bf16, false); }
  else { if (ln) CS(float, true); else CS(float, false); }
#undef CS
}

void launch_colsum(int dt, const void* A, float* part, int N, int d, float* out, unsigned* counters, cudaStream_t s) {
  note_launch(1);
  dim3 grid(colsum_groups(d), colsum_blocks(N)), block(32, kColLanes);
  if (dt == BF16)
    launch_pdl(colsum_k<bf16, false, false>, grid, block, 0, s, (const bf16*)A, nullptr, nullptr, nullptr, nullptr, part, N, d,
                                                        nullptr, out, counters);
  else
    launch_pdl(colsum_k<float, false, false>, grid, block, 0, s, (const float*)A, nullptr, nullptr, nullptr, nullptr, part, N,
                                                         d, nullptr, out, counters);
}

__global__ void partials_add_k(const float* __restrict__ part, int nb, int d, float* __restrict__ out) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= d) return;
  float acc = 0.f;
  for (int b = 0; b < nb; ++b) acc += part[(size_t)b * d + c];
  out[c] += acc;
}

void launch_partials_add(const float* part, int nb, int d, float* out, cudaStream_t s) {
  note_launch(1);
  partials_add_k<<<(d + 255) / 256, 256, 0, s>>>(part, nb, d, out);
}

// ------------------------------------------------------------------------------------------
// RoPE (rotate-half), SwiGLU, GELU(tanh)
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void rope_k(T* __restrict__ qkv, const float2* __restrict__ cs, int N, int S, int nh, int hd,
                       int ld, int inverse) {
  pdl_wait();
  pdl_trigger();
  const int half = hd / 2;
  const long total = (long)N * nh * half;
  for (long idx = blockIdx.x * (long)blockDim.x + threadIdx.x; idx < total;
       idx += (long)gridDim.x * blockDim.x) {
    const int i = (int)(idx % half);
    const int hh = (int)((idx / half) % nh);
    const int n = (int)(idx / ((long)half * nh));
    const float2 c = cs[(size_t)(n % S) * half + i];
    const float sn = inverse ? -c.y : c.y;
    T* p = qkv + (size_t)n * ld + (size_t)hh * hd;
    const float x1 = to_f(p[i]), x2 = to_f(p[i + half]);
    float y1, y2;
    rope_rot(x1, x2, c.x, sn, y1, y2);
    p[i] = from_f<T>(y1);
    p[i + half] = from_f<T>(y2);
  }
}

// Head dims with hd / 2 a multiple of 8: one thread per 8 rotation pairs (16-byte loads of both halves and
// 64 bytes of the (cos, sin) table), blocks striding over token rows, no 64-bit index divisions.
template <typename T>
__global__ void rope8_k(T* __restrict__ qkv, const float2* __restrict__ cs, int N, int S, int nh, int hd, int ld,
                        int inverse) {
  pdl_wait();
  pdl_trigger();
  const int half = hd / 2, g8 = half / 8, per_row = nh * g8;
  const float sg = inverse ? -1.f : 1.f;
  for (int n = blockIdx.x; n < N; n += gridDim.x) {
    const float2* c = cs + (size_t)(n % S) * half;
    T* row = qkv + (size_t)n * ld;
    for (int w = threadIdx.x; w < per_row; w += blockDim.x) {
      const int hh = w / g8, i0 = (w - hh * g8) * 8;
      T* p = row + hh * hd + i0;
      float x1[8], x2[8], y1[8], y2[8];
      Vec8<T>::load(p, x1);
      Vec8<T>::load(p + half, x2);
      const float4* c4 = reinterpret_cast<const float4*>(c + i0);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float4 t = c4[j];   // (cos, sin) of pairs i0 + 2j and i0 + 2j + 1
        const float co[2] = {t.x, t.z}, sn[2] = {sg * t.y, sg * t.w};
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int q = 2 * j + e;
          rope_rot(x1[q], x2[q], co[e], sn[e], y1[q], y2[q]);
        }
      }
      Vec8<T>::store(p, y1);
      Vec8<T>::store(p + half, y2);
    }
  }
}

void launch_rope(int dt, void* qkv, const float* cs, int N, int S, int H, int Hkv, int hd, int inverse,
                 cudaStream_t s) {
  launch_rope_heads(dt, qkv, cs, N, S, H + Hkv, hd, (H + 2 * Hkv) * hd, inverse, s);
}

void launch_rope_heads(int dt, void* qkv, const float* cs, int N, int S, int nh, int hd, int ld, int inverse,
                       cudaStream_t s) {
  note_launch(1);
  if (hd % 16 == 0) {
    const int th = 128, g = std::min(N, 152 * 16);
    if (dt == BF16) launch_pdl(rope8_k<bf16>, g, th, 0, s, (bf16*)qkv, (const float2*)cs, N, S, nh, hd, ld, inverse);
    else launch_pdl(rope8_k<float>, g, th, 0, s, (float*)qkv, (const float2*)cs, N, S, nh, hd, ld, inverse);
    return;
  }
  const int th = 256, g = grid_for((size_t)N * nh * (hd / 2), th);
  if (dt == BF16) launch_pdl(rope_k<bf16>, g, th, 0, s, (bf16*)qkv, (const float2*)cs, N, S, nh, hd, ld, inverse);
  else launch_pdl(rope_k<float>, g, th, 0, s, (float*)qkv, (const float2*)cs, N, S, nh, hd, ld, inverse);
}

__device__ __forceinline__ float sigmoidf_(float x) { return 1.f / (1.f + expf(-x)); }

template <typename T>
__global__ void swiglu_fwd_k(const T* __restrict__ gu, T* __restrict__ a, int N, int f) {
  pdl_wait();
  pdl_trigger();
  const int nv = f / 8;
  const long total = (long)N * nv;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < total; i += (long)gridDim.x * blockDim.x) {
    const int n = (int)(i / nv), c = (int)(i % nv) * 8;
    float g[8], u[8];
    Vec8<T>::load(gu + (size_t)n * 2 * f + c, g);
    Vec8<T>::load(gu + (size_t)n * 2 * f + f + c, u);
#pragma unroll
    for (int q = 0; q < 8; ++q) g[q] = g[q] * sigmoidf_(g[q]) * u[q];
    Vec8<T>::store(a + (size_t)n * f + c, g);
  }
}

template <typename T>
__global__ void swiglu_bwd_k(const T* __restrict__ gu, const T* __restrict__ da, T* __restrict__ dgu, int N,
                             int f) {
  pdl_wait();
  pdl_trigger();
  const int nv = f / 8;
  const long total = (long)N * nv;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < total; i += (long)gridDim.x * blockDim.x) {
    const int n = (int)(i / nv), c = (int)(i % nv) * 8;
    float g[8], u[8], d[8], dg[8], du[8];
    Vec8<T>::load(gu + (size_t)n * 2 * f + c, g);
    Vec8<T>::load(gu + (size_t)n * 2 * f + f + c, u);
    Vec8<T>::load(da + (size_t)n * f + c, d);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float sg = sigmoidf_(g[q]);
      du[q] = d[q] * g[q] * sg;
      dg[q] = d[q] * u[q] * sg * (1.f + g[q] * (1.f - sg));
    }
    Vec8<T>::store(dgu + (size_t)n * 2 * f + c, dg);
    Vec8<T>::store(dgu + (size_t)n * 2 * f + f + c, du);
  }
}

void launch_swiglu_fwd(int dt, const void* gu, void* a, int N, int f, cudaStream_t s) {
  note_launch(1);
  const int th = 256, g = grid_for((size_t)N * (f / 8), th);
  if (dt == BF16) launch_pdl(swiglu_fwd_k<bf16>, g, th, 0, s, (const bf16*)gu, (bf16*)a, N, f);
  else launch_pdl(swiglu_fwd_k<float>, g, th, 0, s, (const float*)gu, (float*)a, N, f);
}
void launch_swiglu_bwd(int dt, const void* gu, const void* da, void* dgu, int N, int f, cudaStream_t s) {
  note_launch(1);
  const int th = 256, g = grid_for((size_t)N * (f / 8), th);
  if (dt == BF16) launch_pdl(swiglu_bwd_k<bf16>, g, th, 0, s, (const bf16*)gu, (const bf16*)da, (bf16*)dgu, N, f);
  else launch_pdl(swiglu_bwd_k<float>, g, th, 0, s, (const float*)gu, (const float*)da, (float*)dgu, N, f);
}

__device__ __forceinline__ float gelu_inner(float x) { return 0.7978845608028654f * (x + 0.044715f * x * x * x); }
// tanh for the GELU of bf16 activations: the SFU's tanh.approx (relative error about 2^-11, below the
// 2^-8 of the bf16 result); fp32 activations keep the accurate tanhf.
template <typename T>
__device__ __forceinline__ float gelu_tanh(float v) {
  if constexpr (std::is_same<T, bf16>::value) {
    float y;
    asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(v));
    return y;
  } else {
    return tanhf(v);
  }
}

template <typename T>
__global__ void gelu_fwd_k(const T* __restrict__ x, T* __restrict__ y, size_t n8) {
  pdl_wait();
  pdl_trigger();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n8; i += (size_t)gridDim.x * blockDim.x) {
    float f[8];
    Vec8<T>::load(x + i * 8, f);
#pragma unroll
    for (int q = 0; q < 8; ++q) f[q] = 0.5f * f[q] * (1.f + gelu_tanh<T>(gelu_inner(f[q])));
    Vec8<T>::store(y + i * 8, f);
  }
}

template <typename T>
__global__ void gelu_bwd_k(const T* __restrict__ x, const T* __restrict__ dy, T* __restrict__ dx, size_t n8) {
  pdl_wait();
  pdl_trigger();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n8; i += (size_t)gridDim.x * blockDim.x) {
    float f[8], d[8];
    Vec8<T>::load(x + i * 8, f);
    Vec8<T>::load(dy + i * 8, d);
#pragma unroll
    for (int q = 0; q < 8; ++q) d[q] *= gelu_tanh_grad(f[q], std::is_same<T, bf16>::value);
    Vec8<T>::store(dx + i * 8, d);
  }
}

void launch_gelu_fwd(int dt, const void* x, void* y, size_t n, cudaStream_t s) {
  note_launch(1);
  const int th = 256, g = grid_for(n / 8, th);
  if (dt == BF16) launch_pdl(gelu_fwd_k<bf16>, g, th, 0, s, (const bf16*)x, (bf16*)y, n / 8);
  else launch_pdl(gelu_fwd_k<float>, g, th, 0, s, (const float*)x, (float*)y, n / 8);
}
void launch_gelu_bwd(int dt, const void* x, const void* dy, void* dx, size_t n, cudaStream_t s) {
  note_launch(1);
  const int th = 256, g = grid_for(n / 8, th);
  if (dt == BF16) launch_pdl(gelu_bwd_k<bf16>, g, th, 0, s, (const bf16*)x, (const bf16*)dy, (bf16*)dx, n / 8);
  else launch_pdl(gelu_bwd_k<float>, g, th, 0, s, (const float*)x, (const float*)dy, (float*)dx, n / 8);
}

// ------------------------------------------------------------------------------------------
// Local objective (Eq. 3-5), fused: per row i in Omega with p = softmax(z_i), q = softmax(t_i):
//   CE_i = lse_z - z_y;  KL_i = sum_j p_j (z_j - t_j) - lse_z + lse_t       (kl_dir 0: KL(p||q))
//                        KL_i = sum_j q_j (t_j - z_j) - lse_t + lse_z       (kl_dir 1: KL(q||p))
//   dz_j = (1/|Omega|) [alpha (p_j - [j = y]) + (1 - alpha) g_j],
//   g_j = p_j ((z_j - t_j) - (lse_z - lse_t) - KL_i)   (kl_dir 0),   g_j = p_j - q_j   (kl_dir 1).
// One block per row; pass 1 keeps online (max, sum) pairs, pass 2 writes dz. No probability
// tensor is stored.
// ------------------------------------------------------------------------------------------
constexpr float kL2e = 1.4426950408889634f, kLn2 = 0.6931471805599453f;

// 2^x by the SFU's ex2.approx (relative error about 2^-22; flushes subnormal results to zero,
// which only affects probabilities below 1e-38).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}


struct Lse3 { float m, s, a; };   // running max (log2 units), sum 2^(x-m), sum 2^(x-m) * w

__device__ __forceinline__ Lse3 lse_merge(Lse3 x, Lse3 y) {
  const float M = fmaxf(x.m, y.m);
  if (M == -INFINITY) return x;
  const float ex = ex2(x.m - M), ey = ex2(y.m - M);
  return Lse3{M, x.s * ex + y.s * ey, x.a * ex + y.a * ey};
}

__device__ __forceinline__ Lse3 warp_merge(Lse3 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Lse3 w{__shfl_xor_sync(0xffffffffu, v.m, o), __shfl_xor_sync(0xffffffffu, v.s, o),
           __shfl_xor_sync(0xffffffffu, v.a, o)};
    v = lse_merge(v, w);
  }
  return v;
}


// Online base-2 log-sum-exp of 8 raw logits x (the running max A.m is kept in log2 units, x * log2 e),
// optionally with the cross term sum 2^(x log2 e - m) * w. nvalid < 8 only for the last, partial
// vector of a row. The scale by log2 e is folded into the exponent's FMA.
template <bool FULL>
__device__ __forceinline__ void lse_add8(Lse3& A, const float* x, const float* w, int nvalid) {
  float mx = -INFINITY;
#pragma unroll
  for (int i = 0; i < 8; ++i)
    if (FULL || i < nvalid) mx = fmaxf(mx, x[i]);
  mx *= kL2e;
  if (mx > A.m) {
    const float sc = ex2(A.m - mx);
    A.s *= sc;
    A.a *= sc;
    A.m = mx;
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if (FULL || i < nvalid) {
      const float e = ex2(fmaf(x[i], kL2e, -A.m));
      A.s += e;
      if (w) A.a = fmaf(e, w[i], A.a);
    }
  }
}

template <typename T, bool TEACHER, int KLDIR, bool FULL>
__device__ __forceinline__ void loss_pass1_vec(const T* zp, const T* tp, Lse3& Z, Lse3& Q, int nv) {
  float zs[8], ts[8], w[8];
  Vec8<T>::load(zp, zs);
  if (TEACHER) {
    Vec8<T>::load(tp, ts);
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = KLDIR == 0 ? zs[i] - ts[i] : ts[i] - zs[i];   // natural units
    lse_add8<FULL>(Z, zs, KLDIR == 0 ? w : nullptr, nv);
    lse_add8<FULL>(Q, ts, KLDIR == 0 ? nullptr : w, nv);
  } else {
    lse_add8<FULL>(Z, zs, nullptr, nv);
  }
}

// bf16 vectors in packed form: the running sums in two lanes (fp32 pairs), the block maximum from the
// raw bf16 pairs (exact), every FMA / add on pairs. Same terms as lse_add8, about a third fewer
// instructions per element.
struct Lse2 { float m; uint64_t s, a; };   // running max (log2 units), two-lane sum 2^(x-m), cross sum

__device__ __forceinline__ Lse3 lse2_fold(const Lse2& A) {
  const float2 s = uf2(A.s), a = uf2(A.a);
  return Lse3{A.m, s.x + s.y, a.x + a.y};
}

__device__ __forceinline__ void lse2_add8(Lse2& A, const uint4& raw, const uint64_t* x2, const uint64_t* w2) {
  const uint32_t mm = bf2_max(bf2_max(raw.x, raw.y), bf2_max(raw.z, raw.w));
  const float mx = fmaxf(__uint_as_float(mm << 16), __uint_as_float(mm & 0xffff0000u)) * kL2e;
  if (mx > A.m) {
    const float sc = ex2(A.m - mx);
    const uint64_t sc2 = f2(sc, sc);
    A.s = mul2(A.s, sc2);
    if (w2) A.a = mul2(A.a, sc2);
    A.m = mx;
  }
  const uint64_t l2 = f2(kL2e, kL2e), nm = f2(-A.m, -A.m);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 x = uf2(fma2(x2[i], l2, nm));
    const uint64_t e = f2(ex2(x.x), ex2(x.y));
    A.s = add2(A.s, e);
    if (w2) A.a = fma2(e, w2[i], A.a);
  }
}

template <bool TEACHER, int KLDIR>
__device__ __forceinline__ void loss_pass1_bf16(const bf16* zp, const bf16* tp, Lse2& Z, Lse2& Q) {
  const uint4 zr = *reinterpret_cast<const uint4*>(zp);
  const uint64_t z2[4] = {bf2_to_f2(zr.x), bf2_to_f2(zr.y), bf2_to_f2(zr.z), bf2_to_f2(zr.w)};
  if (TEACHER) {
    const uint4 tr = *reinterpret_cast<const uint4*>(tp);
    const uint64_t t2[4] = {bf2_to_f2(tr.x), bf2_to_f2(tr.y), bf2_to_f2(tr.z), bf2_to_f2(tr.w)};
    uint64_t w2[4];   // natural units
#pragma unroll
    for (int i = 0; i < 4; ++i) w2[i] = KLDIR == 0 ? sub2(z2[i], t2[i]) : sub2(t2[i], z2[i]);
    lse2_add8(Z, zr, z2, KLDIR == 0 ? w2 : nullptr);
    lse2_add8(Q, tr, t2, KLDIR == 0 ? nullptr : w2);
  } else {
    lse2_add8(Z, zr, z2, nullptr);
  }
}

// One block per row of logits. Pass 1: base-2 online log-sum-exp of z and t and the KL cross term
// (two full vectors per trip for loads in flight); pass 2 (the row is still in L2) writes dz. dz may be
// z itself (in place): every element is read before it is written, by the same thread.
template <typename T, bool TEACHER, int KLDIR>
__device__ __forceinline__ void local_loss_row(const T* z, const T* __restrict__ t,
                                               const int32_t* __restrict__ labels, int V, int ldz, float alpha,
                                               const int* __restrict__ count, T* dz,
                                               float* __restrict__ row_loss) {
  pdl_wait();
  pdl_trigger();
  __shared__ Lse3 shz[32], sht[32];
  __shared__ float sh_stats[4];
  const int row = blockIdx.x;
  const T* zr = z + (size_t)row * ldz;
  const T* tr = TEACHER ? t + (size_t)row * ldz : nullptr;
  T* dr = dz + (size_t)row * ldz;
  const int y = labels[row];
  const int step = blockDim.x * 8;
  if (!(y >= 0 && y < V)) {   // rows outside Omega: no loss, zero gradient
    float f[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int c = threadIdx.x * 8; c < ldz; c += step) Vec8<T>::store(dr + c, f);
    if (threadIdx.x == 0) row_loss[row] = 0.f;
    return;
  }
  Lse3 Z{-INFINITY, 0.f, 0.f}, Q{-INFINITY, 0.f, 0.f};
  int c = threadIdx.x * 8;
  if constexpr (std::is_same<T, bf16>::value) {
    Lse2 Z2{-INFINITY, 0ull, 0ull}, Q2{-INFINITY, 0ull, 0ull};   // (0ull is the pair (+0, +0))
    for (; c + step + 8 <= V; c += 2 * step) {
      loss_pass1_bf16<TEACHER, KLDIR>(zr + c, tr + c, Z2, Q2);
      loss_pass1_bf16<TEACHER, KLDIR>(zr + c + step, tr + c + step, Z2, Q2);
    }
    for (; c + 8 <= V; c += step) loss_pass1_bf16<TEACHER, KLDIR>(zr + c, tr + c, Z2, Q2);
    if (c < V) loss_pass1_vec<T, TEACHER, KLDIR, false>(zr + c, tr + c, Z, Q, V - c);
    Z = lse_merge(lse2_fold(Z2), Z);
    if (TEACHER) Q = lse_merge(lse2_fold(Q2), Q);
  } else {
    for (; c + step + 8 <= V; c += 2 * step) {
      loss_pass1_vec<T, TEACHER, KLDIR, true>(zr + c, tr + c, Z, Q, 8);
      loss_pass1_vec<T, TEACHER, KLDIR, true>(zr + c + step, tr + c + step, Z, Q, 8);
    }
    for (; c < V; c += step) {
      if (c + 8 <= V) loss_pass1_vec<T, TEACHER, KLDIR, true>(zr + c, tr + c, Z, Q, 8);
      else loss_pass1_vec<T, TEACHER, KLDIR, false>(zr + c, tr + c, Z, Q, V - c);
    }
  }
  Z = warp_merge(Z);
  if (TEACHER) Q = warp_merge(Q);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (lane == 0) { shz[wid] = Z; sht[wid] = Q; }
  __syncthreads();
  if (threadIdx.x == 0) {
    Lse3 a = shz[0], b = sht[0];
    for (int i = 1; i < nw; ++i) { a = lse_merge(a, shz[i]); if (TEACHER) b = lse_merge(b, sht[i]); }
    const float lse_z = (a.m + log2f(a.s)) * kLn2;
    float lse_t = 0.f, kl = 0.f;
    if (TEACHER) {
      lse_t = (b.m + log2f(b.s)) * kLn2;
      kl = KLDIR == 0 ? a.a / a.s - lse_z + lse_t : b.a / b.s - lse_t + lse_z;
    }
    row_loss[row] = alpha * (lse_z - to_f(zr[y])) + (TEACHER ? (1.f - alpha) * kl : 0.f);
    sh_stats[0] = lse_z;
    sh_stats[1] = lse_t;
    sh_stats[2] = kl;
  }
  __syncthreads();
  const float lse_z = sh_stats[0], lse_t = sh_stats[1], kl = sh_stats[2];
  const float lz2 = lse_z * kL2e, lt2 = lse_t * kL2e, shift = (lse_z - lse_t) + kl;
  const int cnt = *count;
  const float inv_n = cnt > 0 ? 1.f / (float)cnt : 0.f;
  const float wt = inv_n * alpha, wc = inv_n * (1.f - alpha);
  //   kl_dir 0: dz = p (wt + wc ((z - t) - shift));  kl_dir 1: dz = (wt + wc) p - wc q;  no teacher: wt p
  const float k0 = wt - wc * shift, wtc = wt + wc;
  const uint64_t L2 = f2(kL2e, kL2e), NLZ = f2(-lz2, -lz2), NLT = f2(-lt2, -lt2), WT = f2(wt, wt), WC = f2(wc, wc),
                 K0 = f2(k0, k0), WTC = f2(wtc, wtc), NWC = f2(-wc, -wc);
  // dz of one 8-wide vector at column c from its raw z (and t) words (bf16 rows)
  auto emit_bf16 = [&](int cc, const uint4& zr4, const uint4& tr4) {
    const uint32_t zw[4] = {zr4.x, zr4.y, zr4.z, zr4.w}, tw[4] = {tr4.x, tr4.y, tr4.z, tr4.w};
    float o[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint64_t z2 = bf2_to_f2(zw[i]);
      const float2 x = uf2(fma2(z2, L2, NLZ));
      const uint64_t p = f2(ex2(x.x), ex2(x.y));
      uint64_t r;
      if (!TEACHER) {
        r = mul2(WT, p);
      } else if (KLDIR == 0) {
        r = mul2(p, fma2(WC, sub2(z2, bf2_to_f2(tw[i])), K0));
      } else {
        const float2 xt = uf2(fma2(bf2_to_f2(tw[i]), L2, NLT));
        r = fma2(WTC, p, mul2(NWC, f2(ex2(xt.x), ex2(xt.y))));
      }
      const float2 rf = uf2(r);
      o[2 * i] = rf.x;
      o[2 * i + 1] = rf.y;
    }
    if (y >= cc && y < cc + 8) o[y - cc] -= wt;   // the one-hot of the task term
    if (cc + 8 > V) {
#pragma unroll
      for (int i = 0; i < 8; ++i)
        if (cc + i >= V) o[i] = 0.f;   // padding columns
    }
    Vec8<T>::store(dr + cc, o);
  };
  c = threadIdx.x * 8;
  if constexpr (std::is_same<T, bf16>::value) {
    const uint4 zero4 = make_uint4(0u, 0u, 0u, 0u);
    for (; c + step < ldz; c += 2 * step) {   // two vectors' loads in flight per trip
      const uint4 za = *reinterpret_cast<const uint4*>(zr + c), zb = *reinterpret_cast<const uint4*>(zr + c + step);
      const uint4 ta = TEACHER ? *reinterpret_cast<const uint4*>(tr + c) : zero4;
      const uint4 tb = TEACHER ? *reinterpret_cast<const uint4*>(tr + c + step) : zero4;
      emit_bf16(c, za, ta);
      emit_bf16(c + step, zb, tb);
    }
    if (c < ldz) emit_bf16(c, *reinterpret_cast<const uint4*>(zr + c),
                           TEACHER ? *reinterpret_cast<const uint4*>(tr + c) : zero4);
  } else {
    for (; c < ldz; c += step) {
      float fz[8], ft[8], o[8];
      Vec8<T>::load(zr + c, fz);
      if (TEACHER) Vec8<T>::load(tr + c, ft);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float p = ex2(fmaf(fz[i], kL2e, -lz2));
        if (!TEACHER) o[i] = wt * p;
        else if (KLDIR == 0) o[i] = p * fmaf(wc, fz[i] - ft[i], k0);
        else o[i] = fmaf(wtc, p, -wc * ex2(fmaf(ft[i], kL2e, -lt2)));
      }
      if (y >= c && y < c + 8) o[y - c] -= wt;   // the one-hot of the task term
      if (c + 8 > V) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if (c + i >= V) o[i] = 0.f;   // padding columns
      }
      Vec8<T>::store(dr + c, o);
    }
  }
}

// Two rows per SM (the compiler's own register choice) and three rows per SM (at most 40 registers).
template <typename T, bool TEACHER, int KLDIR>
__global__ void __launch_bounds__(1024) local_loss_k(const T* z, const T* __restrict__ t,
                                                     const int32_t* __restrict__ labels, int V, int ldz,
                                                     float alpha, const int* __restrict__ count,
                                                     T* dz, float* __restrict__ row_loss) {
  local_loss_row<T, TEACHER, KLDIR>(z, t, labels, V, ldz, alpha, count, dz, row_loss);
}
template <typename T, bool TEACHER, int KLDIR>
__global__ void __launch_bounds__(512, 3) local_loss3_k(const T* z, const T* __restrict__ t,
                                                        const int32_t* __restrict__ labels, int V, int ldz,
                                                        float alpha, const int* __restrict__ count,
                                                        T* dz, float* __restrict__ row_loss) {
  local_loss_row<T, TEACHER, KLDIR>(z, t, labels, V, ldz, alpha, count, dz, row_loss);
}

void launch_local_loss(int dt, const void* z, const void* t, const int32_t* labels, int N, int V, int ldz,
                       float alpha, int kl_dir, const int* count, void* dz, float* row_loss, cudaStream_t s) {
  note_launch(1);
  if (N <= 0) return;
  // up to 512 threads per row (one 8-wide vector each): several rows in flight per SM, and the rows
  // being read still fit in L2 for the second pass. Three rows per SM (40 registers) where the rows in
  // flight on every SM stay well inside L2 (V = 32000: 58 MB), two otherwise (V = 50257: three would
  // hold 92 MB, and pass 2 would go back to DRAM: 293 against 260 us at 4096 rows).
  int th = 32;
  while (th < 512 && th * 8 < ldz) th *= 2;
  const size_t row_bytes = (size_t)ldz * dt_size(dt) * (t ? 2 : 1);
  const bool three = dt == BF16 && 3ull * 152 * row_bytes <= (64ull << 20);
#define LL2(T, TE, KD)                                                                                            \
  launch_pdl(local_loss_k<T, TE, KD>, N, th, 0, s, (const T*)z, (const T*)t, labels, V, ldz, alpha, count, (T*)dz, \
             row_loss)
#define LL(T, TE, KD)                                                                                           \
  if (three)                                                                                                    \
    launch_pdl(local_loss3_k<T, TE, KD>, N, th, 0, s, (const T*)z, (const T*)t, labels, V, ldz, alpha, count,   \
               (T*)dz, row_loss);                                                                               \
  else                                                                                                          \
    LL2(T, TE, KD);
  if (dt == BF16) {
    if (!t) { LL(bf16, false, 0) }
    else if (kl_dir == 0) { LL(bf16, true, 0) }
    else { LL(bf16, true, 1) }
  } else {   // fp32 rows: two per SM
    if (!t) LL2(float, false, 0);
    else if (kl_dir == 0) LL2(float, true, 0);
    else LL2(float, true, 1);
  }
#undef LL
#undef LL2
}

__global__ void count_valid_k(const int32_t* __restrict__ labels, int N, int V, int* count, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  __shared__ float sh[32];
  float c = 0.f;
  bool bad = false;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    const int y = labels[i];
    if (y >= 0 && y < V) c += 1.f;
    if (y < -1 || y >= V) bad = true;
  }
  if (bad) atomicOr(err, ZL_DEVERR_BAD_LABEL);
  c = block_sum(c, sh);
  if (threadIdx.x == 0) *count = (int)(c + 0.5f);
}

void launch_count_valid(const int32_t* labels, int N, int V, int* count, unsigned* err, cudaStream_t s) {
  note_launch(1);
  launch_pdl(count_valid_k, 1, 1024, 0, s, labels, N, V, count, err);
}

__global__ void loss_reduce_k(const float* __restrict__ rl, int N, const int* count, float* out) {
  pdl_wait();
  pdl_trigger();
  __shared__ double sh[1024];
  double acc = 0.0;
  for (int i0 = threadIdx.x; i0 < N; i0 += 4 * blockDim.x) {   // 4 loads in flight, added in index order
    float v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = i0 + q * (int)blockDim.x < N ? rl[i0 + q * blockDim.x] : 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (i0 + q * (int)blockDim.x < N) acc += (double)v[q];
  }
  sh[threadIdx.x] = acc;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {
    if ((int)threadIdx.x < o) sh[threadIdx.x] += sh[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const int c = *count;
    *out = c > 0 ? (float)(sh[0] / (double)c) : 0.f;
  }
}

void launch_loss_reduce(const float* row_loss, int N, const int* count, float* out, cudaStream_t s) {
  note_launch(1);
  launch_pdl(loss_reduce_k, 1, 1024, 0, s, row_loss, N, count, out);
}

// ------------------------------------------------------------------------------------------
// AdamW over one chunk's contiguous parameter slab (decoupled weight decay, bias correction).
// ------------------------------------------------------------------------------------------
// Advances a chunk's optimizer step count t (device memory, so a replayed CUDA graph keeps counting)
// and writes this step's learning rate and bias corrections: hp = {lr_t, 1 - beta1^t, 1 - beta2^t}.
__global__ void adamw_tick_k(long long* __restrict__ t, float* __restrict__ hp, float lr0, int schedule,
                             float gamma, float b1, float b2) {
  pdl_wait();
  pdl_trigger();
  const long long tt = *t + 1;
  *t = tt;
  const double lr = schedule == 1 ? (double)lr0 / sqrt((double)(tt - 1) + (double)gamma) : (double)lr0;
  hp[0] = (float)lr;
  hp[1] = (float)(1.0 - pow((double)b1, (double)tt));
  hp[2] = (float)(1.0 - pow((double)b2, (double)tt));
}

__global__ void adamw_k(float4* __restrict__ th, float4* __restrict__ g, float4* __restrict__ m,
                        float4* __restrict__ v, __nv_bfloat162* __restrict__ comp, size_t n4,
                        const float* __restrict__ hp, float b1, float b2, float eps, float wd, float gscale) {
  pdl_wait();
  pdl_trigger();
  const AdamHP h = adam_hp(hp, b1, b2, eps, wd);
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4; i += (size_t)gridDim.x * blockDim.x) {
    float4 t = th[i], gg = g[i], mm = m[i], vv = v[i];
    float* tp = &t.x; float* gp = &gg.x; float* mp = &mm.x; float* vp = &vv.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) adamw_elem(tp[q], mp[q], vp[q], __fmul_rn(gp[q], gscale), h);
    th[i] = t; m[i] = mm; v[i] = vv;
    g[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (comp) {
      comp[2 * i] = __floats2bfloat162_rn(t.x, t.y);
      comp[2 * i + 1] = __floats2bfloat162_rn(t.z, t.w);
    }
  }
}

void launch_adamw_tick(long long* t, float* hp, float lr0, int schedule, float gamma, float b1, float b2,
                       cudaStream_t s) {
  note_launch(1);
  launch_pdl(adamw_tick_k, 1, 1, 0, s, t, hp, lr0, schedule, gamma, b1, b2);
}

void launch_adamw(float* theta, float* g, float* m, float* v, void* comp, size_t n, long long* t, float* hp,
                  float lr0, int schedule, float gamma, float b1, float b2, float eps, float wd, float gscale,
                  cudaStream_t s) {
  launch_adamw_tick(t, hp, lr0, schedule, gamma, b1, b2, s);
  note_launch(1);
  const size_t n4 = n / 4;   // slabs are padded to a multiple of 64 elements
  if (n4 == 0) return;
  const int th = 256, gr = grid_for(n4, th, 152 * 8);
  launch_pdl(adamw_k, gr, th, 0, s, (float4*)theta, (float4*)g, (float4*)m, (float4*)v, (__nv_bfloat162*)comp, n4,
             (const float*)hp, b1, b2, eps, wd, gscale);
}

void launch_adamw_span(float* theta, float* g, float* m, float* v, void* comp, size_t n, const float* hp, float b1,
                       float b2, float eps, float wd, float gscale, cudaStream_t s) {
  const size_t n4 = n / 4;
  if (n4 == 0) return;
  note_launch(1);
  const int th = 256, gr = grid_for(n4, th, 152 * 8);
  launch_pdl(adamw_k, gr, th, 0, s, (float4*)theta, (float4*)g, (float4*)m, (float4*)v, (__nv_bfloat162*)comp, n4,
             hp, b1, b2, eps, wd, gscale);
}

// AdamW over a list of ranges of one slab (offsets and lengths in floats, multiples of 4), with this
// step's lr and bias corrections already in hp (no tick): the parameters the weight-gradient GEMMs did
// not update in their epilogue. blockIdx.y is the range.
__global__ void adamw_ranges_k(float* __restrict__ th, float* __restrict__ g, float* __restrict__ m,
                               float* __restrict__ v, bf16* __restrict__ comp, const long long* __restrict__ ranges,
                               const float* __restrict__ hp, float b1, float b2, float eps, float wd, float gscale) {
  pdl_wait();
  pdl_trigger();
  const AdamHP h = adam_hp(hp, b1, b2, eps, wd);
  const size_t off = (size_t)ranges[2 * blockIdx.y], n4 = (size_t)ranges[2 * blockIdx.y + 1] / 4;
  float4* th4 = reinterpret_cast<float4*>(th + off);
  float4* g4 = reinterpret_cast<float4*>(g + off);
  float4* m4 = reinterpret_cast<float4*>(m + off);
  float4* v4 = reinterpret_cast<float4*>(v + off);
  __nv_bfloat162* c2 = comp ? reinterpret_cast<__nv_bfloat162*>(comp + off) : nullptr;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4; i += (size_t)gridDim.x * blockDim.x) {
    float4 t = th4[i], gg = g4[i], mm = m4[i], vv = v4[i];
    float* tp = &t.x; float* gp = &gg.x; float* mp = &mm.x; float* vp = &vv.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) adamw_elem(tp[q], mp[q], vp[q], __fmul_rn(gp[q], gscale), h);
    th4[i] = t; m4[i] = mm; v4[i] = vv;
    g4[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c2) {
      c2[2 * i] = __floats2bfloat162_rn(t.x, t.y);
      c2[2 * i + 1] = __floats2bfloat162_rn(t.z, t.w);
    }
  }
}

void launch_adamw_ranges(float* theta, float* g, float* m, float* v, void* comp, const long long* ranges,
                         int nranges, size_t max_len, const float* hp, float b1, float b2, float eps, float wd,
                         float gscale, cudaStream_t s) {
  if (nranges <= 0) return;
  note_launch(1);
  const int th = 256;
  const unsigned bx = (unsigned)std::max<size_t>(1, std::min<size_t>((max_len / 4 + th - 1) / th, 64));
  launch_pdl(adamw_ranges_k, dim3(bx, (unsigned)nranges), th, 0, s, theta, g, m, v, (bf16*)comp, ranges, hp, b1,
             b2, eps, wd, gscale);
}

// One thread per four consecutive columns of one row (contiguous in both layouts).
__global__ void adamw_blk_k(float* __restrict__ th, float* __restrict__ g, float* __restrict__ m,
                            float* __restrict__ v, __nv_bfloat162* __restrict__ comp, int M, int N,
                            const float* __restrict__ hp, float b1, float b2, float eps, float wd, float gscale) {
  pdl_wait();
  pdl_trigger();
  const AdamHP h = adam_hp(hp, b1, b2, eps, wd);
  const size_t n4 = (size_t)M * N / 4;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4; i += (size_t)gridDim.x * blockDim.x) {
    const size_t e = 4 * i, b = blk_index(e / N, e % N, N);
    float4 t = *reinterpret_cast<float4*>(th + b), gg = *reinterpret_cast<float4*>(g + e),
           mm = *reinterpret_cast<float4*>(m + b), vv = *reinterpret_cast<float4*>(v + b);
    float* tp = &t.x; float* gp = &gg.x; float* mp = &mm.x; float* vp = &vv.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) adamw_elem(tp[q], mp[q], vp[q], __fmul_rn(gp[q], gscale), h);
    *reinterpret_cast<float4*>(th + b) = t;
    *reinterpret_cast<float4*>(m + b) = mm;
    *reinterpret_cast<float4*>(v + b) = vv;
    *reinterpret_cast<float4*>(g + e) = make_float4(0.f, 0.f, 0.f, 0.f);
    if (comp) {
      comp[2 * i] = __floats2bfloat162_rn(t.x, t.y);
      comp[2 * i + 1] = __floats2bfloat162_rn(t.z, t.w);
    }
  }
}

void launch_adamw_span_blk(float* theta, float* g, float* m, float* v, void* comp, int M, int N, const float* hp,
                           float b1, float b2, float eps, float wd, float gscale, cudaStream_t s) {
  const size_t n4 = (size_t)M * N / 4;
  if (n4 == 0) return;
  note_launch(1);
  const int th = 256, gr = grid_for(n4, th, 152 * 8);
  launch_pdl(adamw_blk_k, gr, th, 0, s, theta, g, m, v, (__nv_bfloat162*)comp, M, N, hp, b1, b2, eps, wd, gscale);
}

__global__ void blk_permute_k(const float* __restrict__ src, float* __restrict__ dst, int M, int N, int to_blk) {
  const size_t n4 = (size_t)M * N / 4;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4; i += (size_t)gridDim.x * blockDim.x) {
    const size_t e = 4 * i, b = blk_index(e / N, e % N, N);
    if (to_blk) *reinterpret_cast<float4*>(dst + b) = *reinterpret_cast<const float4*>(src + e);
    else *reinterpret_cast<float4*>(dst + e) = *reinterpret_cast<const float4*>(src + b);
  }
}

void launch_blk_permute(const float* src, float* dst, int M, int N, int to_blk, cudaStream_t s) {
  const size_t n4 = (size_t)M * N / 4;
  if (n4 == 0) return;
  note_launch(1);
  blk_permute_k<<<grid_for(n4, 256), 256, 0, s>>>(src, dst, M, N, to_blk);
}

__global__ void f32_to_bf16_k(const float* __restrict__ a, bf16* __restrict__ b, size_t n) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
    b[i] = __float2bfloat16_rn(a[i]);
}

void launch_f32_to_bf16(const float* src, void* dst, size_t n, cudaStream_t s) {
  note_launch(1);
  f32_to_bf16_k<<<grid_for(n, 256), 256, 0, s>>>(src, (bf16*)dst, n);
}

}  // namespace zl
