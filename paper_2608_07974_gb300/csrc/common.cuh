// Shared device helpers of the ZeroLock engine (sm_103a).
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <utility>

typedef __nv_bfloat16 bf16;

// Device-side error bits (ZL_DEVERR_*, declared with the C ABI), OR-ed into the context's error word
// and reported by zl_synchronize.
#include "zerolock.h"

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Sum over the block; every thread gets the result. `sh` holds >= 32 floats.
__device__ __forceinline__ float block_sum(float v, float* sh) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) sh[w] = v;
  __syncthreads();
  float r = lane < nw ? sh[lane] : 0.f;
  r = warp_sum(r);
  return r;
}

// 8 consecutive values of T as floats (16 B of bf16 or 2 x 16 B of fp32).
// Packed fp32 pairs (sm_100 and later): one instruction computes two FMAs, subtractions, additions or
// products. A pair lives in one 64-bit register (x in the low half).
__device__ __forceinline__ uint64_t f2(float x, float y) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
  return r;
}
__device__ __forceinline__ float2 uf2(uint64_t r) {
  float2 v;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(v.x), "=f"(v.y) : "l"(r));
  return v;
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t sub2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
// The two bf16 of a packed word as an fp32 pair (exact: bf16 is the top half of an fp32).
__device__ __forceinline__ uint64_t bf2_to_f2(uint32_t w) {
  return f2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
// Element-wise maximum of two bf16 pairs.
__device__ __forceinline__ uint32_t bf2_max(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Derivative of the tanh-form GELU g(u) = 0.5 u (1 + tanh(k (u + c u^3))), k = sqrt(2 / pi), c = 0.044715:
// g'(u) = 0.5 (1 + t) + 0.5 u (1 - t^2) k (1 + 3 c u^2) with t = tanh(k (u + c u^3)). approx: the SFU's
// tanh.approx (relative error about 2^-11; for bf16 activations), else tanhf.
__device__ __forceinline__ float gelu_tanh_grad(float u, bool approx) {
  const float k = 0.7978845608028654f, c = 0.044715f;
  const float a = k * (u + c * u * u * u);
  float t;
  if (approx) asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(a));
  else t = tanhf(a);
  return 0.5f * (1.f + t) + 0.5f * u * (1.f - t * t) * k * (1.f + 3.f * c * u * u);
}

template <typename T> struct Vec8;
template <> struct Vec8<bf16> {
  __device__ __forceinline__ static void load(const bf16* p, float* f) {
    uint4 u = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) { float2 t = __bfloat1622float2(h[i]); f[2 * i] = t.x; f[2 * i + 1] = t.y; }
  }
  __device__ __forceinline__ static void store(bf16* p, const float* f) {
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
    *reinterpret_cast<uint4*>(p) = u;
  }
};
template <> struct Vec8<float> {
  __device__ __forceinline__ static void load(const float* p, float* f) {
    float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w; f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
  }
  __device__ __forceinline__ static void store(float* p, const float* f) {
    reinterpret_cast<float4*>(p)[0] = make_float4(f[0], f[1], f[2], f[3]);
    reinterpret_cast<float4*>(p)[1] = make_float4(f[4], f[5], f[6], f[7]);
  }
};

// Programmatic dependent launch. A kernel launched with launch_pdl may start while the previous kernel
// of its stream is still running: it calls pdl_wait() before its first access to global memory (which
// waits for that kernel to finish and its writes to be visible), then pdl_trigger() so that the next
// kernel of the stream may begin launching in turn.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// The decoupled AdamW step of one parameter (Eq. 6, as AdamW): m <- b1 m + (1 - b1) g;
// v <- b2 v + (1 - b2) g^2; theta <- theta (1 - lr wd) - (lr / bc1) m / (sqrt(v / bc2) + eps), with
// bc1 = 1 - b1^t, bc2 = 1 - b2^t. Every operation is an explicitly rounded intrinsic or a hardware
// approximation instruction (square root and reciprocal, a few ulp, far inside the fp32 parameter
// tolerance), so every kernel that applies the step (the slab and range updates, the weight-gradient
// GEMM's fused epilogue, the split-K reduction) computes the same bits from the same gradient, in about
// a dozen instructions.
// Rotate-half RoPE of one pair (x1 at column i, x2 at column i + hd/2 of a head) by the angle with
// (cos, sin) = (c, sn): every product and sum explicitly rounded, so that every kernel that rotates
// (the RoPE kernels and the QKV product's epilogue) gives the same bits.
__device__ __forceinline__ void rope_rot(float x1, float x2, float c, float sn, float& y1, float& y2) {
  y1 = __fsub_rn(__fmul_rn(x1, c), __fmul_rn(x2, sn));
  y2 = __fadd_rn(__fmul_rn(x2, c), __fmul_rn(x1, sn));
}
struct AdamHP {
  float step, decay, inv_bc2, b1, omb1, b2, omb2, eps;   // step = lr / bc1, inv_bc2 = 1 / bc2
};
// hp = {lr_t, 1 - b1^t, 1 - b2^t} as written by the step-count kernel.
__device__ __forceinline__ AdamHP adam_hp(const float* hp, float b1, float b2, float eps, float wd) {
  AdamHP h;
  const float lr = hp[0];
  h.step = __fdiv_rn(lr, hp[1]);
  h.inv_bc2 = __fdiv_rn(1.f, hp[2]);
  h.decay = __fsub_rn(1.f, __fmul_rn(lr, wd));
  h.b1 = b1;
  h.omb1 = __fsub_rn(1.f, b1);
  h.b2 = b2;
  h.omb2 = __fsub_rn(1.f, b2);
  h.eps = eps;
  return h;
}
__device__ __forceinline__ float sqrt_approx(float x) {
  float r;
  asm("sqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
// Blocked layout of the fp32 master and AdamW moments of a matrix [M, N] (M % 16 == 0, N % 32 == 0)
// whose optimizer step runs in its weight-gradient product: 16 x 32 pieces of 512 contiguous floats
// (row-major inside a piece), the pieces in row-major order over the [M / 16, N / 32] grid. A piece is
// what one epilogue warp updates at a time, so the update streams whole 2 KB runs instead of 128-byte
// segments of rows far apart (the access pattern alone streams about 10% faster on the 7B-shaped
// matrices; the fused kernels, bound by their bytes in flight, gain about 2%). The compute copy and every
// gradient stay row-major.
__host__ __device__ __forceinline__ size_t blk_index(size_t r, size_t c, size_t N) {
  return ((r >> 4) * (N >> 5) + (c >> 5)) * 512 + (r & 15) * 32 + (c & 31);
}
__device__ __forceinline__ void adamw_elem(float& th, float& m, float& v, float g, const AdamHP& h) {
  m = __fmaf_rn(h.b1, m, __fmul_rn(h.omb1, g));
  v = __fmaf_rn(h.b2, v, __fmul_rn(__fmul_rn(h.omb2, g), g));
  const float den = __fadd_rn(sqrt_approx(__fmul_rn(v, h.inv_bc2)), h.eps);
  th = __fmaf_rn(th, h.decay, -__fmul_rn(__fmul_rn(h.step, m), rcp_approx(den)));
}
