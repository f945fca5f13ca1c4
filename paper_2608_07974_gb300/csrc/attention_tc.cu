// Causal attention with grouped KV heads on tensor cores (bf16 mma.sync m16n8k16, fp32
// accumulate), forward and backward. 64-row query / key blocks, four warps of 16 rows each,
// operands staged in XOR-swizzled shared memory by cp.async (double buffered) and read with
// ldmatrix. The forward keeps an online softmax and stores the row log-sum-exp; the backward
// recomputes the probabilities and is split into a dQ kernel (one CTA per query block) and a
// dK/dV kernel (one CTA per key block, looping over the query heads of its KV group), so every
// gradient is a fixed-order sum: no atomics, bit-reproducible under any schedule.
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "ops.h"

namespace zl {
namespace fa {

constexpr int BR = 64;      // rows per block (queries or keys)
constexpr int NT = 128;     // threads per CTA

template <int HDP>
struct Tile {
  static constexpr int CH = HDP / 8;   // 16-byte chunks per row
  __device__ __forceinline__ static int off(int r, int c) {
    const int pc = HDP >= 64 ? (c ^ (r & 7)) : (c ^ ((r >> 1) & 3));
    return r * HDP + pc * 8;
  }
};

__device__ __forceinline__ uint32_t s32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp8(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(s32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldsm4(uint32_t* r, const bf16* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(s32(p)));
}
__device__ __forceinline__ void ldsm4t(uint32_t* r, const bf16* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(s32(p)));
}
__device__ __forceinline__ void mma(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// A fragment (16 rows x 16 k) from a [row][k] tile.
template <int HDP>
__device__ __forceinline__ void frag_a(uint32_t* a, const bf16* t, int r0, int k0, int lane) {
  ldsm4(a, t + Tile<HDP>::off(r0 + (lane & 15), (k0 >> 3) + (lane >> 4)));
}
// B fragments of two 8-wide n tiles (n0..n0+15) x 16 k from an [n][k] tile.
template <int HDP>
__device__ __forceinline__ void frag_b_nk(uint32_t* b, const bf16* t, int n0, int k0, int lane) {
  ldsm4(b, t + Tile<HDP>::off(n0 + (lane & 7) + ((lane >> 4) << 3), (k0 >> 3) + ((lane >> 3) & 1)));
}
// B fragments of two 8-wide n tiles x 16 k from a [k][n] tile (transposing load).
template <int HDP>
__device__ __forceinline__ void frag_b_kn(uint32_t* b, const bf16* t, int k0, int n0, int lane) {
  ldsm4t(b, t + Tile<HDP>::off(k0 + (lane & 7) + (((lane >> 3) & 1) << 3), (n0 >> 3) + (lane >> 4)));
}

// rows [r0, r0 + 64) of a head slice (row stride ld elements) into a swizzled tile; rows >= nrows
// and columns >= hd read as zero. vec: 16-byte copies (hd % 8 == 0); otherwise 8-byte copies of
// 4-element halves when hd % 4 == 0 (e.g. hd = 100, whose head slices are 8-byte aligned).
template <int HDP>
__device__ __forceinline__ void load_tile(bf16* t, const bf16* g, long ld, int nrows, int hd, bool vec) {
  const bool vec8 = (hd & 3) == 0;
  for (int i = threadIdx.x; i < BR * Tile<HDP>::CH; i += NT) {
    const int r = i / Tile<HDP>::CH, c = i % Tile<HDP>::CH;
    bf16* dst = t + Tile<HDP>::off(r, c);
    const bf16* src = g + (size_t)r * ld + c * 8;
    if (r >= nrows || c * 8 >= hd) {
      *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
    } else if (vec) {
      cp16(dst, src);
    } else if (vec8) {
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        if (c * 8 + hf * 4 < hd) cp8(dst + hf * 4, src + hf * 4);
        else *reinterpret_cast<uint2*>(dst + hf * 4) = make_uint2(0u, 0u);
      }
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) dst[e] = c * 8 + e < hd ? src[e] : __float2bfloat16_rn(0.f);
    }
  }
}

constexpr float kLog2e = 1.4426950408889634f;

// 2^x on the SFU (ex2.approx, relative error about 2^-22; subnormal results flush to zero).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ----------------------------------------------------------------------------------------------
// forward
// ----------------------------------------------------------------------------------------------
template <int HDP>
__global__ void __launch_bounds__(NT) fwd_k(const bf16* __restrict__ qkv, bf16* __restrict__ out,
                                            float* __restrict__ lse, int S, int H, int Hkv, int hd, float scale) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(128) uint8_t smem[];
  bf16* Qs = reinterpret_cast<bf16*>(smem);
  bf16* Ks = Qs + BR * HDP;            // [2]
  bf16* Vs = Ks + 2 * BR * HDP;        // [2]
  const int qb = gridDim.z - 1 - blockIdx.z, h = blockIdx.x, b = blockIdx.y;   // longest blocks launch first
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kvh = h / (H / Hkv), ld = (H + 2 * Hkv) * hd;
  const bool vec = (hd & 7) == 0;
  const bf16* base = qkv + (size_t)b * S * ld;
  const int q0 = qb * BR;
  load_tile<HDP>(Qs, base + (size_t)q0 * ld + h * hd, ld, S - q0, hd, vec);
  load_tile<HDP>(Ks, base + (H + kvh) * hd, ld, S, hd, vec);
  load_tile<HDP>(Vs, base + (H + Hkv + kvh) * hd, ld, S, hd, vec);
  cp_commit();
  float o[HDP / 8][4];
#pragma unroll
  for (int i = 0; i < HDP / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
  const float sl2 = scale * kLog2e;
  const int row0 = q0 + warp * 16 + (lane >> 2);
  for (int kb = 0; kb <= qb; ++kb) {
    const int cur = kb & 1;
    if (kb < qb) {
      const int k1 = (kb + 1) * BR;
      load_tile<HDP>(Ks + (cur ^ 1) * BR * HDP, base + (size_t)k1 * ld + (H + kvh) * hd, ld, S - k1, hd, vec);
      load_tile<HDP>(Vs + (cur ^ 1) * BR * HDP, base + (size_t)k1 * ld + (H + Hkv + kvh) * hd, ld, S - k1, hd, vec);
    }
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    const bf16* Kt = Ks + cur * BR * HDP;
    const bf16* Vt = Vs + cur * BR * HDP;
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < HDP / 16; ++ks) {
      uint32_t a[4];
      frag_a<HDP>(a, Qs, warp * 16, ks * 16, lane);
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bb[4];
        frag_b_nk<HDP>(bb, Kt, np * 16, ks * 16, lane);
        mma(s[2 * np], a, bb[0], bb[1]);
        mma(s[2 * np + 1], a, bb[2], bb[3]);
      }
    }
    float mx[2] = {m[0], m[1]};
    if (kb < qb && (kb + 1) * BR <= S) {   // strictly below the diagonal and inside the sequence: no mask
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float v = s[nt][e] * sl2;
          s[nt][e] = v;
          mx[e >> 1] = fmaxf(mx[e >> 1], v);
        }
    } else {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int col = kb * BR + nt * 8 + 2 * (lane & 3) + (e & 1);
          const int row = row0 + ((e >> 1) << 3);
          const float v = (col <= row && col < S) ? s[nt][e] * sl2 : -INFINITY;
          s[nt][e] = v;
          mx[e >> 1] = fmaxf(mx[e >> 1], v);
        }
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 1));
      mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 2));
    }
    float corr[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      corr[i] = mx[i] == -INFINITY ? 1.f : ex2(m[i] - mx[i]);
      m[i] = mx[i];
      l[i] *= corr[i];
    }
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float mm = m[e >> 1];
        const float p = mm == -INFINITY ? 0.f : ex2(s[nt][e] - mm);
        s[nt][e] = p;
        l[e >> 1] += p;
      }
#pragma unroll
    for (int i = 0; i < HDP / 8; ++i) {
      o[i][0] *= corr[0]; o[i][1] *= corr[0];
      o[i][2] *= corr[1]; o[i][3] *= corr[1];
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t pa[4] = {pack(s[2 * kk][0], s[2 * kk][1]), pack(s[2 * kk][2], s[2 * kk][3]),
                        pack(s[2 * kk + 1][0], s[2 * kk + 1][1]), pack(s[2 * kk + 1][2], s[2 * kk + 1][3])};
#pragma unroll
      for (int np = 0; np < HDP / 16; ++np) {
        uint32_t bv[4];
        frag_b_kn<HDP>(bv, Vt, kk * 16, np * 16, lane);
        mma(o[2 * np], pa, bv[0], bv[1]);
        mma(o[2 * np + 1], pa, bv[2], bv[3]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    l[i] += __shfl_xor_sync(0xffffffffu, l[i], 1);
    l[i] += __shfl_xor_sync(0xffffffffu, l[i], 2);
  }
  const int HD = H * hd;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int row = row0 + 8 * i;
    if (row >= S) continue;
    const float inv = 1.f / l[i];
    bf16* orow = out + ((size_t)b * S + row) * HD + h * hd;
#pragma unroll
    for (int nt = 0; nt < HDP / 8; ++nt) {
      const int col = nt * 8 + 2 * (lane & 3);
      if (col < hd) *reinterpret_cast<uint32_t*>(orow + col) = pack(o[nt][2 * i] * inv, o[nt][2 * i + 1] * inv);
    }
    if ((lane & 3) == 0) lse[((size_t)b * H + h) * S + row] = (m[i] + log2f(l[i])) * 0.6931471805599453f;
  }
}

// ----------------------------------------------------------------------------------------------
// backward: dQ (one CTA per query block of one head)
// ----------------------------------------------------------------------------------------------
template <int HDP>
__global__ void __launch_bounds__(NT) bwd_dq_k(const bf16* __restrict__ qkv, const bf16* __restrict__ outp,
                                               const bf16* __restrict__ dout, const float* __restrict__ lse,
                                               float* __restrict__ Dv, bf16* __restrict__ dqkv, int S, int H,
                                               int Hkv, int hd, float scale) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(128) uint8_t smem[];
  bf16* Qs = reinterpret_cast<bf16*>(smem);
  bf16* dOs = Qs + BR * HDP;
  bf16* Ks = dOs + BR * HDP;           // [2]
  bf16* Vs = Ks + 2 * BR * HDP;        // [2]
  float* Ls = reinterpret_cast<float*>(Vs + 2 * BR * HDP);
  float* Ds = Ls + BR;
  const int qb = gridDim.z - 1 - blockIdx.z, h = blockIdx.x, b = blockIdx.y;   // longest blocks launch first
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kvh = h / (H / Hkv), ld = (H + 2 * Hkv) * hd, HD = H * hd;
  const bool vec = (hd & 7) == 0;
  const bf16* base = qkv + (size_t)b * S * ld;
  const int q0 = qb * BR;
  load_tile<HDP>(Qs, base + (size_t)q0 * ld + h * hd, ld, S - q0, hd, vec);
  load_tile<HDP>(dOs, dout + ((size_t)b * S + q0) * HD + h * hd, HD, S - q0, hd, vec);
  load_tile<HDP>(Ks, base + (H + kvh) * hd, ld, S, hd, vec);
  load_tile<HDP>(Vs, base + (H + Hkv + kvh) * hd, ld, S, hd, vec);
  cp_commit();
  // D_i = sum_d dO_i[d] O_i[d] for this block's rows (written for the dK/dV kernel that follows)
  for (int i = threadIdx.x >> 1; i < BR; i += NT / 2) {
    const int r = q0 + i;
    float acc = 0.f;
    if (r < S) {
      const bf16* orow = outp + ((size_t)b * S + r) * HD + h * hd;
      const bf16* drow = dout + ((size_t)b * S + r) * HD + h * hd;
      for (int dd = (threadIdx.x & 1) * 2; dd < hd; dd += 4) {
        const float2 o2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(orow + dd));
        const float2 g2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(drow + dd));
        acc = fmaf(o2.x, g2.x, fmaf(o2.y, g2.y, acc));
      }
    }
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);
    if ((threadIdx.x & 1) == 0) {
      const size_t si = ((size_t)b * H + h) * S + r;
      Ls[i] = r < S ? lse[si] * kLog2e : 0.f;
      Ds[i] = r < S ? acc : 0.f;
      if (r < S) Dv[si] = acc;
    }
  }
  float dq[HDP / 8][4];
#pragma unroll
  for (int i = 0; i < HDP / 8; ++i) dq[i][0] = dq[i][1] = dq[i][2] = dq[i][3] = 0.f;
  const float sl2 = scale * kLog2e;
  const int lr0 = warp * 16 + (lane >> 2);   // local rows lr0, lr0 + 8
  for (int kb = 0; kb <= qb; ++kb) {
    const int cur = kb & 1;
    if (kb < qb) {
      const int k1 = (kb + 1) * BR;
      load_tile<HDP>(Ks + (cur ^ 1) * BR * HDP, base + (size_t)k1 * ld + (H + kvh) * hd, ld, S - k1, hd, vec);
      load_tile<HDP>(Vs + (cur ^ 1) * BR * HDP, base + (size_t)k1 * ld + (H + Hkv + kvh) * hd, ld, S - k1, hd, vec);
    }
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    const bf16* Kt = Ks + cur * BR * HDP;
    const bf16* Vt = Vs + cur * BR * HDP;
    float s[8][4], dp[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int e = 0; e < 4; ++e) s[i][e] = dp[i][e] = 0.f;
#pragma unroll
    for (int ks = 0; ks < HDP / 16; ++ks) {
      uint32_t a[4], ad[4];
      frag_a<HDP>(a, Qs, warp * 16, ks * 16, lane);
      frag_a<HDP>(ad, dOs, warp * 16, ks * 16, lane);
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bk[4], bvv[4];
        frag_b_nk<HDP>(bk, Kt, np * 16, ks * 16, lane);
        frag_b_nk<HDP>(bvv, Vt, np * 16, ks * 16, lane);
        mma(s[2 * np], a, bk[0], bk[1]);
        mma(s[2 * np + 1], a, bk[2], bk[3]);
        mma(dp[2 * np], ad, bvv[0], bvv[1]);
        mma(dp[2 * np + 1], ad, bvv[2], bvv[3]);
      }
    }
    const float L0 = Ls[lr0], L1 = Ls[lr0 + 8], D0 = Ds[lr0], D1 = Ds[lr0 + 8];
    if (kb < qb && (qb + 1) * BR <= S) {   // no causal or length mask in this block
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float p = ex2(s[nt][e] * sl2 - (e < 2 ? L0 : L1));
          s[nt][e] = p * (dp[nt][e] - (e < 2 ? D0 : D1));   // dS
        }
    } else {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int col = kb * BR + nt * 8 + 2 * (lane & 3) + (e & 1);
          const int row = q0 + lr0 + ((e >> 1) << 3);
          const bool ok = col <= row && col < S && row < S;
          const float p = ok ? ex2(s[nt][e] * sl2 - (e < 2 ? L0 : L1)) : 0.f;
          s[nt][e] = p * (dp[nt][e] - (e < 2 ? D0 : D1));
        }
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t pa[4] = {pack(s[2 * kk][0], s[2 * kk][1]), pack(s[2 * kk][2], s[2 * kk][3]),
                        pack(s[2 * kk + 1][0], s[2 * kk + 1][1]), pack(s[2 * kk + 1][2], s[2 * kk + 1][3])};
#pragma unroll
      for (int np = 0; np < HDP / 16; ++np) {
        uint32_t bk[4];
        frag_b_kn<HDP>(bk, Kt, kk * 16, np * 16, lane);
        mma(dq[2 * np], pa, bk[0], bk[1]);
        mma(dq[2 * np + 1], pa, bk[2], bk[3]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int row = q0 + lr0 + 8 * i;
    if (row >= S) continue;
    bf16* drow = dqkv + ((size_t)b * S + row) * ld + h * hd;
#pragma unroll
    for (int nt = 0; nt < HDP / 8; ++nt) {
      const int col = nt * 8 + 2 * (lane & 3);
      if (col < hd) *reinterpret_cast<uint32_t*>(drow + col) = pack(dq[nt][2 * i] * scale, dq[nt][2 * i + 1] * scale);
    }
  }
}

// ----------------------------------------------------------------------------------------------
// backward: dK, dV (one CTA per key block of one KV head; loops over its query heads)
// ----------------------------------------------------------------------------------------------
// part == NULL: one CTA per (key block, KV head) looping over the group's query heads, writing dK, dV.
// part != NULL: one CTA per (key block, query head); fp32 partials part[2][H][B*S][hd] (dK unscaled,
// dV), reduced over each group by reduce_dkv_k.
template <int HDP>
__global__ void __launch_bounds__(NT) bwd_dkv_k(const bf16* __restrict__ qkv, const bf16* __restrict__ dout,
                                                const float* __restrict__ lse, const float* __restrict__ Dv,
                                                bf16* __restrict__ dqkv, int S, int H, int Hkv, int hd, float scale,
                                                float* __restrict__ part) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(128) uint8_t smem[];
  bf16* Ks = reinterpret_cast<bf16*>(smem);
  bf16* Vs = Ks + BR * HDP;
  bf16* Qs = Vs + BR * HDP;            // [2]
  bf16* dOs = Qs + 2 * BR * HDP;       // [2]
  float* Ls = reinterpret_cast<float*>(dOs + 2 * BR * HDP);   // [2][BR]
  float* Ds = Ls + 2 * BR;                                     // [2][BR]
  const int kb = blockIdx.z, b = blockIdx.y;   // key block 0 (the longest) launches first
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ld = (H + 2 * Hkv) * hd, HD = H * hd;
  const int kvh = part ? blockIdx.x / (H / Hkv) : blockIdx.x;
  const int rep = part ? 1 : H / Hkv;                  // query heads this CTA loops over
  const int h_first = part ? blockIdx.x : kvh * (H / Hkv);
  const bool vec = (hd & 7) == 0;
  const bf16* base = qkv + (size_t)b * S * ld;
  const int k0 = kb * BR;
  const int nqb = (S + BR - 1) / BR;
  const int per_head = nqb - kb;
  const int iters = rep * per_head;
  load_tile<HDP>(Ks, base + (size_t)k0 * ld + (H + kvh) * hd, ld, S - k0, hd, vec);
  load_tile<HDP>(Vs, base + (size_t)k0 * ld + (H + Hkv + kvh) * hd, ld, S - k0, hd, vec);
  auto stage = [&](int it, int buf) {
    const int h = h_first + it / per_head, qb = kb + it % per_head, q0 = qb * BR;
    load_tile<HDP>(Qs + buf * BR * HDP, base + (size_t)q0 * ld + h * hd, ld, S - q0, hd, vec);
    load_tile<HDP>(dOs + buf * BR * HDP, dout + ((size_t)b * S + q0) * HD + h * hd, HD, S - q0, hd, vec);
    for (int i = threadIdx.x; i < BR; i += NT) {
      const int r = q0 + i;
      const size_t si = ((size_t)b * H + h) * S + r;
      Ls[buf * BR + i] = r < S ? lse[si] * kLog2e : 0.f;
      Ds[buf * BR + i] = r < S ? Dv[si] : 0.f;
    }
  };
  stage(0, 0);
  cp_commit();
  float dk[HDP / 8][4], dv[HDP / 8][4];
#pragma unroll
  for (int i = 0; i < HDP / 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) dk[i][e] = dv[i][e] = 0.f;
  const float sl2 = scale * kLog2e;
  const int lr0 = warp * 16 + (lane >> 2);   // local key rows lr0, lr0 + 8
  for (int it = 0; it < iters; ++it) {
    const int cur = it & 1;
    if (it + 1 < iters) stage(it + 1, cur ^ 1);
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    const int q0 = (kb + it % per_head) * BR;
    const bf16* Qt = Qs + cur * BR * HDP;
    const bf16* dOt = dOs + cur * BR * HDP;
    const float* Lt = Ls + cur * BR;
    const float* Dt = Ds + cur * BR;
    // phase 1: S^T = K Q^T, then P^T, kept only as the packed bf16 A fragments of the dV product
    uint32_t pa[4][4];
    const bool inner = q0 > k0 && q0 + BR <= S;   // every query after every key, all in range: no mask
    {
      float st[8][4];
#pragma unroll
      for (int i = 0; i < 8; ++i) st[i][0] = st[i][1] = st[i][2] = st[i][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < HDP / 16; ++ks) {
        uint32_t ak[4];
        frag_a<HDP>(ak, Ks, warp * 16, ks * 16, lane);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          uint32_t bq[4];
          frag_b_nk<HDP>(bq, Qt, np * 16, ks * 16, lane);
          mma(st[2 * np], ak, bq[0], bq[1]);
          mma(st[2 * np + 1], ak, bq[2], bq[3]);
        }
      }
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        const int lq = nt * 8 + 2 * (lane & 3);
        const float2 L2 = *reinterpret_cast<const float2*>(Lt + lq);
        float p[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          bool ok = true;
          if (!inner) {
            const int q = q0 + lq + (e & 1);
            const int key = k0 + lr0 + ((e >> 1) << 3);
            ok = q >= key && q < S && key < S;
          }
          p[e] = ok ? ex2(st[nt][e] * sl2 - ((e & 1) ? L2.y : L2.x)) : 0.f;
        }
        pa[nt >> 1][(nt & 1) * 2] = pack(p[0], p[1]);
        pa[nt >> 1][(nt & 1) * 2 + 1] = pack(p[2], p[3]);
      }
    }
    // phase 2: dP^T = V dO^T, dS^T = P^T (dP^T - D) with P^T from the bf16 fragments
    uint32_t da[4][4];
    {
      float dpt[8][4];
#pragma unroll
      for (int i = 0; i < 8; ++i) dpt[i][0] = dpt[i][1] = dpt[i][2] = dpt[i][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < HDP / 16; ++ks) {
        uint32_t av[4];
        frag_a<HDP>(av, Vs, warp * 16, ks * 16, lane);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          uint32_t bd[4];
          frag_b_nk<HDP>(bd, dOt, np * 16, ks * 16, lane);
          mma(dpt[2 * np], av, bd[0], bd[1]);
          mma(dpt[2 * np + 1], av, bd[2], bd[3]);
        }
      }
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        const int lq = nt * 8 + 2 * (lane & 3);
        const float2 D2 = *reinterpret_cast<const float2*>(Dt + lq);
        const uint32_t u01 = pa[nt >> 1][(nt & 1) * 2], u23 = pa[nt >> 1][(nt & 1) * 2 + 1];
        const float2 p01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u01));
        const float2 p23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u23));
        da[nt >> 1][(nt & 1) * 2] = pack(p01.x * (dpt[nt][0] - D2.x), p01.y * (dpt[nt][1] - D2.y));
        da[nt >> 1][(nt & 1) * 2 + 1] = pack(p23.x * (dpt[nt][2] - D2.x), p23.y * (dpt[nt][3] - D2.y));
      }
    }
    // dV += P^T dO, dK += dS^T Q
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int np = 0; np < HDP / 16; ++np) {
        uint32_t bdo[4], bq[4];
        frag_b_kn<HDP>(bdo, dOt, kk * 16, np * 16, lane);
        frag_b_kn<HDP>(bq, Qt, kk * 16, np * 16, lane);
        mma(dv[2 * np], pa[kk], bdo[0], bdo[1]);
        mma(dv[2 * np + 1], pa[kk], bdo[2], bdo[3]);
        mma(dk[2 * np], da[kk], bq[0], bq[1]);
        mma(dk[2 * np + 1], da[kk], bq[2], bq[3]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int key = k0 + lr0 + 8 * i;
    if (key >= S) continue;
    if (part) {
      const size_t NS = (size_t)gridDim.y * S;
      float* pk = part + ((size_t)h_first * NS + (size_t)b * S + key) * hd;
      float* pv = pk + (size_t)H * NS * hd;
#pragma unroll
      for (int nt = 0; nt < HDP / 8; ++nt) {
        const int col = nt * 8 + 2 * (lane & 3);
        if (col < hd) {
          *reinterpret_cast<float2*>(pk + col) = make_float2(dk[nt][2 * i], dk[nt][2 * i + 1]);
          *reinterpret_cast<float2*>(pv + col) = make_float2(dv[nt][2 * i], dv[nt][2 * i + 1]);
        }
      }
      continue;
    }
    bf16* dkr = dqkv + ((size_t)b * S + key) * ld + (H + kvh) * hd;
    bf16* dvr = dqkv + ((size_t)b * S + key) * ld + (H + Hkv + kvh) * hd;
#pragma unroll
    for (int nt = 0; nt < HDP / 8; ++nt) {
      const int col = nt * 8 + 2 * (lane & 3);
      if (col < hd) {
        *reinterpret_cast<uint32_t*>(dkr + col) = pack(dk[nt][2 * i] * scale, dk[nt][2 * i + 1] * scale);
        *reinterpret_cast<uint32_t*>(dvr + col) = pack(dv[nt][2 * i], dv[nt][2 * i + 1]);
      }
    }
  }
}

template <int HDP>
void fwd_t(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s) {
  const int smem = 5 * BR * HDP * 2;
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(fwd_k<HDP>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(fwd_k<HDP>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    attr = true;
  }
  dim3 grid(H, B, (S + BR - 1) / BR);
  launch_pdl(fwd_k<HDP>, grid, NT, smem, s, (const bf16*)qkv, (bf16*)out, lse, S, H, Hkv, hd, 1.f / sqrtf((float)hd));
}

// dK, dV of each KV head = fixed-order sums of its query heads' partials.
__global__ void reduce_dkv_k(const float* __restrict__ part, bf16* __restrict__ dqkv, int NS, int H, int Hkv, int hd,
                             float scale) {
  pdl_wait();
  pdl_trigger();
  const int rep = H / Hkv, ld = (H + 2 * Hkv) * hd;
  const size_t total = (size_t)NS * Hkv * (hd / 2);
  const size_t HNS = (size_t)H * NS * hd;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
    const int dd = (int)(i % (hd / 2)) * 2;
    const int kvh = (int)((i / (hd / 2)) % Hkv);
    const size_t n = i / ((size_t)(hd / 2) * Hkv);
    float k0 = 0.f, k1 = 0.f, v0 = 0.f, v1 = 0.f;
    for (int hh = 0; hh < rep; ++hh) {
      const size_t o = ((size_t)(kvh * rep + hh) * NS + n) * hd + dd;
      const float2 a = *reinterpret_cast<const float2*>(part + o);
      const float2 c = *reinterpret_cast<const float2*>(part + HNS + o);
      k0 += a.x; k1 += a.y; v0 += c.x; v1 += c.y;
    }
    bf16* row = dqkv + n * ld;
    *reinterpret_cast<uint32_t*>(row + (H + kvh) * hd + dd) = pack(k0 * scale, k1 * scale);
    *reinterpret_cast<uint32_t*>(row + (H + Hkv + kvh) * hd + dd) = pack(v0, v1);
  }
}

template <int HDP>
void bwd_t(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv, int B, int S,
           int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool) {
  const float scale = 1.f / sqrtf((float)hd);
  const int smem = 6 * BR * HDP * 2 + 4 * BR * 4;
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(bwd_dq_k<HDP>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(bwd_dkv_k<HDP>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(bwd_dq_k<HDP>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    cudaFuncSetAttribute(bwd_dkv_k<HDP>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    attr = true;
  }
  dim3 gq(H, B, (S + BR - 1) / BR);
  launch_pdl(bwd_dq_k<HDP>, gq, NT, smem, s, (const bf16*)qkv, (const bf16*)out, (const bf16*)dout, lse, D, (bf16*)dqkv, S, H,
                                     Hkv, hd, scale);
  float* part = nullptr;
  if (H > Hkv) {   // grouped heads: one CTA per query head, then a fixed-order group reduction
    const size_t bytes = 2ull * H * B * S * hd * sizeof(float);
    cudaError_t e = pool ? cudaMallocFromPoolAsync((void**)&part, bytes, pool, s) : cudaMallocAsync((void**)&part, bytes, s);
    if (e != cudaSuccess) { cudaGetLastError(); part = nullptr; }
  }
  dim3 gk(part ? H : Hkv, B, (S + BR - 1) / BR);
  launch_pdl(bwd_dkv_k<HDP>, gk, NT, smem, s, (const bf16*)qkv, (const bf16*)dout, lse, D, (bf16*)dqkv, S, H, Hkv, hd, scale,
                                      part);
  if (part) {
    const size_t total = (size_t)B * S * Hkv * (hd / 2);
    const int blocks = (int)std::min<size_t>((total + 255) / 256, 152 * 16);
    launch_pdl(reduce_dkv_k, blocks, 256, 0, s, part, (bf16*)dqkv, B * S, H, Hkv, hd, scale);
    cudaFreeAsync(part, s);
  }
}

}  // namespace fa

bool attn_fwd_tc(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s) {
  if (hd > 128 || hd % 2) return false;
  if (hd <= 32) fa::fwd_t<32>(qkv, out, lse, B, S, H, Hkv, hd, s);
  else if (hd <= 64) fa::fwd_t<64>(qkv, out, lse, B, S, H, Hkv, hd, s);
  else fa::fwd_t<128>(qkv, out, lse, B, S, H, Hkv, hd, s);
  return true;
}

void launch_reduce_dkv(const float* part, void* dqkv, int NS, int H, int Hkv, int hd, float scale, cudaStream_t s) {
  const size_t total = (size_t)NS * Hkv * (hd / 2);
  const int blocks = (int)std::min<size_t>((total + 255) / 256, 152 * 16);
  launch_pdl(fa::reduce_dkv_k, blocks, 256, 0, s, part, (bf16*)dqkv, NS, H, Hkv, hd, scale);
}

bool attn_bwd_tc(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv, int B, int S,
                 int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool) {
  if (hd > 128 || hd % 2) return false;
  if (hd <= 32) fa::bwd_t<32>(qkv, out, dout, lse, D, dqkv, B, S, H, Hkv, hd, s, pool);
  else if (hd <= 64) fa::bwd_t<64>(qkv, out, dout, lse, D, dqkv, B, S, H, Hkv, hd, s, pool);
  else fa::bwd_t<128>(qkv, out, dout, lse, D, dqkv, B, S, H, Hkv, hd, s, pool);
  return true;
}

}  // namespace zl
