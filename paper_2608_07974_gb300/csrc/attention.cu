// Causal softmax attention with grouped KV heads, forward and backward, CUDA-core version:
// one warp per query (or key) row, fp32 online softmax. Query head h reads KV head
// h / (H / Hkv). Scale 1/sqrt(hd). The forward saves the row log-sum-exp for the backward.
#include <math.h>

#include "common.cuh"
#include "ops.h"

namespace zl {

namespace {
constexpr int R = 4;   // dims per lane: head_dim <= 128

template <typename T>
__device__ __forceinline__ void load_row(const T* p, int hd, int lane, float* v, float scale) {
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int d = lane + 32 * r;
    v[r] = d < hd ? to_f(p[d]) * scale : 0.f;
  }
}
template <typename T>
__device__ __forceinline__ float dot_row(const T* p, int hd, int lane, const float* v) {
  float s = 0.f;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int d = lane + 32 * r;
    if (d < hd) s += v[r] * to_f(p[d]);
  }
  return warp_sum(s);
}

template <typename T>
__global__ void attn_fwd_k(const T* __restrict__ qkv, T* __restrict__ out, float* __restrict__ lse, int B, int S,
                           int H, int Hkv, int hd, float scale) {
  const long gw = (blockIdx.x * (long)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (long)B * H * S) return;
  const int i = S - 1 - (int)(gw % S);              // long rows first
  const int h = (int)((gw / S) % H), b = (int)(gw / ((long)S * H));
  const int ld = (H + 2 * Hkv) * hd, kvh = h / (H / Hkv);
  float q[R], o[R] = {0.f, 0.f, 0.f, 0.f};
  load_row(qkv + (size_t)(b * S + i) * ld + h * hd, hd, lane, q, scale);
  float m = -INFINITY, l = 0.f;
  const T* kb = qkv + (size_t)b * S * ld + (H + kvh) * hd;
  const T* vb = qkv + (size_t)b * S * ld + (H + Hkv + kvh) * hd;
  for (int j = 0; j <= i; ++j) {
    const float s = dot_row(kb + (size_t)j * ld, hd, lane, q);
    const float mn = fmaxf(m, s);
    const float corr = expf(m - mn), p = expf(s - mn);
    l = l * corr + p;
    const T* vr = vb + (size_t)j * ld;
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int d = lane + 32 * r;
      o[r] = o[r] * corr + (d < hd ? p * to_f(vr[d]) : 0.f);
    }
    m = mn;
  }
  T* orow = out + (size_t)(b * S + i) * H * hd + h * hd;
  const float inv = 1.f / l;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int d = lane + 32 * r;
    if (d < hd) orow[d] = from_f<T>(o[r] * inv);
  }
  if (lane == 0) lse[((size_t)b * H + h) * S + i] = m + logf(l);
}

// D_i = sum_d dO_i[d] * O_i[d]
template <typename T>
__global__ void attn_bwd_d_k(const T* __restrict__ out, const T* __restrict__ dout, float* __restrict__ D, int B,
                             int S, int H, int hd) {
  const long gw = (blockIdx.x * (long)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (long)B * H * S) return;
  const int i = (int)(gw % S), h = (int)((gw / S) % H), b = (int)(gw / ((long)S * H));
  const size_t o = (size_t)(b * S + i) * H * hd + h * hd;
  float v[R];
  load_row(out + o, hd, lane, v, 1.f);
  const float s = dot_row(dout + o, hd, lane, v);
  if (lane == 0) D[((size_t)b * H + h) * S + i] = s;
}

template <typename T>
__global__ void attn_bwd_dq_k(const T* __restrict__ qkv, const T* __restrict__ dout, const float* __restrict__ lse,
                              const float* __restrict__ D, T* __restrict__ dqkv, int B, int S, int H, int Hkv, int hd,
                              float scale) {
  const long gw = (blockIdx.x * (long)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (long)B * H * S) return;
  const int i = S - 1 - (int)(gw % S), h = (int)((gw / S) % H), b = (int)(gw / ((long)S * H));
  const int ld = (H + 2 * Hkv) * hd, kvh = h / (H / Hkv);
  float q[R], dO[R], dq[R] = {0.f, 0.f, 0.f, 0.f};
  load_row(qkv + (size_t)(b * S + i) * ld + h * hd, hd, lane, q, scale);
  load_row(dout + (size_t)(b * S + i) * H * hd + h * hd, hd, lane, dO, 1.f);
  const size_t si = ((size_t)b * H + h) * S + i;
  const float L = lse[si], Di = D[si];
  const T* kb = qkv + (size_t)b * S * ld + (H + kvh) * hd;
  const T* vb = qkv + (size_t)b * S * ld + (H + Hkv + kvh) * hd;
  for (int j = 0; j <= i; ++j) {
    const T* kr = kb + (size_t)j * ld;
    const float p = expf(dot_row(kr, hd, lane, q) - L);
    const float dp = dot_row(vb + (size_t)j * ld, hd, lane, dO);
    const float ds = p * (dp - Di);
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int d = lane + 32 * r;
      if (d < hd) dq[r] += ds * to_f(kr[d]);
    }
  }
  T* dr = dqkv + (size_t)(b * S + i) * ld + h * hd;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int d = lane + 32 * r;
    if (d < hd) dr[d] = from_f<T>(dq[r] * scale);
  }
}

template <typename T>
__global__ void attn_bwd_dkv_k(const T* __restrict__ qkv, const T* __restrict__ dout, const float* __restrict__ lse,
                               const float* __restrict__ D, T* __restrict__ dqkv, int B, int S, int H, int Hkv, int hd,
                               float scale) {
  const long gw = (blockIdx.x * (long)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (long)B * Hkv * S) return;
  const int j = (int)(gw % S), kvh = (int)((gw / S) % Hkv), b = (int)(gw / ((long)S * Hkv));
  const int ld = (H + 2 * Hkv) * hd, rep = H / Hkv;
  float k[R], v[R], dk[R] = {0.f, 0.f, 0.f, 0.f}, dv[R] = {0.f, 0.f, 0.f, 0.f};
  load_row(qkv + (size_t)(b * S + j) * ld + (H + kvh) * hd, hd, lane, k, scale);
  load_row(qkv + (size_t)(b * S + j) * ld + (H + Hkv + kvh) * hd, hd, lane, v, 1.f);
  for (int hh = 0; hh < rep; ++hh) {
    const int h = kvh * rep + hh;
    for (int i = j; i < S; ++i) {
      const T* qr = qkv + (size_t)(b * S + i) * ld + h * hd;
      const T* dor = dout + (size_t)(b * S + i) * H * hd + h * hd;
      const size_t si = ((size_t)b * H + h) * S + i;
      const float p = expf(dot_row(qr, hd, lane, k) - lse[si]);
      const float dp = dot_row(dor, hd, lane, v);
      const float ds = p * (dp - D[si]);
#pragma unroll
      for (int r = 0; r < R; ++r) {
        const int d = lane + 32 * r;
        if (d < hd) { dv[r] += p * to_f(dor[d]); dk[r] += ds * to_f(qr[d]); }
      }
    }
  }
  T* dkr = dqkv + (size_t)(b * S + j) * ld + (H + kvh) * hd;
  T* dvr = dqkv + (size_t)(b * S + j) * ld + (H + Hkv + kvh) * hd;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int d = lane + 32 * r;
    if (d < hd) { dkr[d] = from_f<T>(dk[r] * scale); dvr[d] = from_f<T>(dv[r]); }
  }
}

inline int warps_grid(long rows) { return (int)((rows * 32 + 255) / 256); }

// Head padding for the tcgen05 kernels (head dims 64 and 128): dst [N, nh * hp] from src [N, nh * hd] with
// each head's columns hd .. hp - 1 zero (pad), or src [N, nh * hp] back to dst [N, nh * hd] (unpad).
// Zero query and key columns add nothing to Q K^T, zero value columns give zero output columns, and the
// gradients of the padding columns are zero, so the padded products are the unpadded ones. bf16 pairs.
__global__ void heads_pad_k(const __nv_bfloat162* __restrict__ src, __nv_bfloat162* __restrict__ dst, int N, int nh,
                            int hd, int hp, int pad) {
  pdl_wait();
  pdl_trigger();
  const int h2 = hd / 2, p2 = hp / 2;
  const int src_w = (pad ? h2 : p2) * nh, dst_w = (pad ? p2 : h2) * nh, cols = nh * (pad ? p2 : h2);
  const __nv_bfloat162 zero = __floats2bfloat162_rn(0.f, 0.f);
  for (int n = blockIdx.x; n < N; n += gridDim.x) {
    const __nv_bfloat162* sr = src + (size_t)n * src_w;
    __nv_bfloat162* dr = dst + (size_t)n * dst_w;
    for (int c = threadIdx.x; c < cols; c += blockDim.x) {
      if (pad) {
        const int h = c / p2, e = c - h * p2;
        dr[c] = e < h2 ? sr[h * h2 + e] : zero;
      } else {
        const int h = c / h2, e = c - h * h2;
        dr[c] = sr[h * p2 + e];
      }
    }
  }
}

void heads_pad(const void* src, void* dst, int N, int nh, int hd, int hp, bool pad, cudaStream_t s) {
  note_launch(1);
  launch_pdl(heads_pad_k, std::min(N, 152 * 16), 256, 0, s, (const __nv_bfloat162*)src, (__nv_bfloat162*)dst, N, nh, hd,
             hp, pad ? 1 : 0);
}

// The tcgen05 head dim a bf16 head of hd columns is padded to, or 0 when it runs as it is (64, 128) or
// on the mma.sync kernels (odd, or above 128).
int padded_hd(int hd) {
  if (hd == 64 || hd == 128 || hd % 2 != 0 || hd > 128) return 0;
  return hd < 64 ? 64 : 128;
}

void* scratch(size_t bytes, cudaStream_t s, cudaMemPool_t pool) {
  void* p = nullptr;
  const cudaError_t e = pool ? cudaMallocFromPoolAsync(&p, bytes, pool, s) : cudaMallocAsync(&p, bytes, s);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return p;
}
}  // namespace

bool attn_fwd_tc(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s);
bool attn_fwd_tcgen05(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s,
                      unsigned* err, float scale);
bool attn_bwd_tc(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv, int B, int S,
                 int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool);
bool attn_bwd_tcgen05(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv,
                      int B, int S, int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool, unsigned* err,
                      float scale);

namespace {
// bf16 heads of a dim the tcgen05 kernels do not take: zero-padded copies through them (padded_hd).
bool attn_fwd_padded(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s,
                     unsigned* err, cudaMemPool_t pool) {
  const int hp = padded_hd(hd), N = B * S, nh = H + 2 * Hkv;
  if (!hp) return false;
  void* qp = scratch((size_t)N * nh * hp * 2, s, pool);
  void* op = qp ? scratch((size_t)N * H * hp * 2, s, pool) : nullptr;
  bool ok = op != nullptr;
  if (ok) {
    heads_pad(qkv, qp, N, nh, hd, hp, true, s);
    ok = attn_fwd_tcgen05(qp, op, lse, B, S, H, Hkv, hp, s, err, 1.f / sqrtf((float)hd));
    if (ok) heads_pad(op, out, N, H, hd, hp, false, s);
  }
  if (op) cudaFreeAsync(op, s);
  if (qp) cudaFreeAsync(qp, s);
  return ok;
}

bool attn_bwd_padded(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv, int B,
                     int S, int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool, unsigned* err) {
  const int hp = padded_hd(hd), N = B * S, nh = H + 2 * Hkv;
  if (!hp) return false;
  const size_t wq = (size_t)N * nh * hp * 2, wo = (size_t)N * H * hp * 2;
  void* buf = scratch(2 * wq + 2 * wo, s, pool);
  if (!buf) return false;
  char* qp = (char*)buf;
  char* dqp = qp + wq;
  char* op = dqp + wq;
  char* dop = op + wo;
  heads_pad(qkv, qp, N, nh, hd, hp, true, s);
  heads_pad(out, op, N, H, hd, hp, true, s);
  heads_pad(dout, dop, N, H, hd, hp, true, s);
  const bool ok = attn_bwd_tcgen05(qp, op, dop, lse, D, dqp, B, S, H, Hkv, hp, s, pool, err, 1.f / sqrtf((float)hd));
  if (ok) heads_pad(dqp, dqkv, N, nh, hd, hp, false, s);
  cudaFreeAsync(buf, s);
  return ok;
}
}  // namespace

void attn_fwd(int dt, const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s,
              unsigned* err, cudaMemPool_t pool) {
  if (dt == BF16 && attn_fwd_tcgen05(qkv, out, lse, B, S, H, Hkv, hd, s, err, 1.f / sqrtf((float)hd))) return;
  if (dt == BF16 && attn_fwd_padded(qkv, out, lse, B, S, H, Hkv, hd, s, err, pool)) return;
  note_launch(1);
  if (dt == BF16 && attn_fwd_tc(qkv, out, lse, B, S, H, Hkv, hd, s)) return;
  const float scale = 1.f / sqrtf((float)hd);
  const int g = warps_grid((long)B * H * S);
  if (dt == BF16) attn_fwd_k<bf16><<<g, 256, 0, s>>>((const bf16*)qkv, (bf16*)out, lse, B, S, H, Hkv, hd, scale);
  else attn_fwd_k<float><<<g, 256, 0, s>>>((const float*)qkv, (float*)out, lse, B, S, H, Hkv, hd, scale);
}

void attn_bwd(int dt, const void* qkv, const void* out, const void* dout, const float* lse, float* Dbuf, void* dqkv,
              int B, int S, int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool, unsigned* err) {
  note_launch(dt == BF16 ? (H > Hkv ? 3 : 2) : 3);
  const float scale = 1.f / sqrtf((float)hd);
  const int gq = warps_grid((long)B * H * S), gk = warps_grid((long)B * Hkv * S);
  if (dt == BF16 && attn_bwd_tcgen05(qkv, out, dout, lse, Dbuf, dqkv, B, S, H, Hkv, hd, s, pool, err, scale)) return;
  if (dt == BF16 && attn_bwd_padded(qkv, out, dout, lse, Dbuf, dqkv, B, S, H, Hkv, hd, s, pool, err)) return;
  if (dt == BF16 && attn_bwd_tc(qkv, out, dout, lse, Dbuf, dqkv, B, S, H, Hkv, hd, s, pool)) return;
  if (dt == BF16) {
    attn_bwd_d_k<bf16><<<gq, 256, 0, s>>>((const bf16*)out, (const bf16*)dout, Dbuf, B, S, H, hd);
    attn_bwd_dq_k<bf16><<<gq, 256, 0, s>>>((const bf16*)qkv, (const bf16*)dout, lse, Dbuf, (bf16*)dqkv, B, S, H, Hkv,
                                           hd, scale);
    attn_bwd_dkv_k<bf16><<<gk, 256, 0, s>>>((const bf16*)qkv, (const bf16*)dout, lse, Dbuf, (bf16*)dqkv, B, S, H,
                                            Hkv, hd, scale);
  } else {
    attn_bwd_d_k<float><<<gq, 256, 0, s>>>((const float*)out, (const float*)dout, Dbuf, B, S, H, hd);
    attn_bwd_dq_k<float><<<gq, 256, 0, s>>>((const float*)qkv, (const float*)dout, lse, Dbuf, (float*)dqkv, B, S, H,
                                            Hkv, hd, scale);
    attn_bwd_dkv_k<float><<<gk, 256, 0, s>>>((const float*)qkv, (const float*)dout, lse, Dbuf, (float*)dqkv, B, S,
                                             H, Hkv, hd, scale);
  }
}

}  // namespace zl
