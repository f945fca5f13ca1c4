// Causal attention forward on the 5th-generation tensor cores (sm_103a), head dim 128 (the kernel is
// written for 64 and 128).
//
// One CTA per 128 query rows of one (batch, head). TMA brings Q once and K / V tiles of 128 keys
// through a stage ring (128-byte swizzle; a 3-D tensor map over [batch, token, feature] reads rows past
// the sequence end as zeros); one thread issues tcgen05.mma with fp32 accumulators in TMEM; eight
// softmax warps, two per TMEM lane quadrant (32 query rows, one row per thread), each take one 64-key
// half of every block. Two passes over
// the key blocks avoid rescaling the output in TMEM: pass 1 forms S = Q K^T and the exact row
// log-sum-exp; pass 2 forms S again, writes P = exp(S - lse) as bf16 into shared memory (the A operand
// of the next product) and accumulates O += P V. S is double-buffered in TMEM, so the product of the
// next key block runs while the softmax warps work on the current one. Every mbarrier wait is bounded
// (2 s); on expiry the kernel raises ZL_DEVERR_TIMEOUT and unwinds.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "ops.h"
#include "tcgen05.cuh"

namespace zl {
namespace tg {
using namespace tc;

constexpr int QB = 128;     // query rows per CTA
constexpr int KB = 128;     // keys per block
constexpr int NSM = 8;      // softmax warps: two per TMEM lane quadrant, one 64-key half of a block each
constexpr int NTHR = 64 + 32 * NSM;   // warp 0: TMA; warp 1: MMA and TMEM; warps 2-9: softmax and output
constexpr float kL2e = 1.4426950408889634f, kLn2 = 0.6931471805599453f;

template <int HD>
struct FCfg {
  static constexpr int QBYTES = QB * HD * 2;   // HD / 64 column blocks of [128 rows x 64] (16 KB each)
  static constexpr int KBYTES = KB * HD * 2;   // same layout
  static constexpr int VBYTES = KB * HD * 2;   // 2 key halves x HD / 64 column blocks of [64 keys x 64]
  static constexpr int STAGES = HD == 64 ? 3 : 2;
  static constexpr int STAGE = KBYTES + VBYTES;
  static constexpr int PBYTES = QB * KB * 2;   // P: 2 key halves of [128 rows x 64 keys]
  static constexpr int SMEM = QBYTES + STAGES * STAGE + PBYTES + 1024 + 256 + 2 * QB * 2 * 4;
  static constexpr int TMEM_COLS = 512;        // S double buffer (2 x 128 columns) + O (HD columns)
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int HD>
__global__ void __launch_bounds__(NTHR, 1)
    attn_fwd_tg_k(const __grid_constant__ CUtensorMap tqk, const __grid_constant__ CUtensorMap tvv,
                  bf16* __restrict__ out, float* __restrict__ lse, int S, int H, int Hkv, float scale,
                  unsigned* err) {
  using C_ = FCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sq = smem;
  uint8_t* sst = sq + C_::QBYTES;                      // stages: K tile, then V tile
  uint8_t* sp = sst + C_::STAGES * C_::STAGE;          // P
  uint64_t* full = (uint64_t*)(sp + C_::PBYTES);
  uint64_t* empty = full + C_::STAGES;
  uint64_t* qfull = empty + C_::STAGES;
  uint64_t* sfull = qfull + 1;                         // [2]
  uint64_t* sempty = sfull + 2;                        // [2]
  uint64_t* pfull = sempty + 2;
  uint64_t* pempty = pfull + 1;
  uint64_t* ofull = pempty + 1;
  uint64_t* fin = ofull + 1;
  uint64_t* statb = fin + 1;                            // the two halves' row statistics are in smem
  float* stat = (float*)(statb + 1);                    // [2 halves][128 rows][m, l]
  uint32_t* tbase = (uint32_t*)(stat + 2 * QB * 2);
  volatile int* abort_flag = (volatile int*)(tbase + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, b = blockIdx.y, qb = gridDim.z - 1 - blockIdx.z;   // longest blocks first
  const int kvh = h / (H / Hkv);
  const int q0 = qb * QB, nkb = qb + 1;                // causal: key blocks 0 .. qb
  const int xq = h * HD, xk = (H + kvh) * HD, xv = (H + Hkv + kvh) * HD;
  const int total = 2 * nkb;                           // pass 1 (S only), then pass 2 (S and P V)

  if (threadIdx.x == 0) {
    for (int s = 0; s < C_::STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(qfull, 1);
    for (int i = 0; i < 2; ++i) { mbar_init(&sfull[i], 1); mbar_init(&sempty[i], NSM); }
    mbar_init(pfull, NSM);
    mbar_init(statb, NSM);
    mbar_init(pempty, 1);
    mbar_init(ofull, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tbase)),
                 "r"((uint32_t)C_::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tbase;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      bool ok = true;
      int issued[C_::STAGES];
#pragma unroll
      for (int s = 0; s < C_::STAGES; ++s) issued[s] = -1;
      mbar_expect_tx(qfull, C_::QBYTES);
#pragma unroll
      for (int c = 0; c < HD / 64; ++c) tma3d(sq + c * 16384, &tqk, qfull, xq + 64 * c, q0, b);
      int stage = 0;
      uint32_t phase = 0;
      for (int it = 0; ok && it < total; ++it) {
        const bool withv = it >= nkb;
        const int j = withv ? it - nkb : it;
        if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err)) { ok = false; break; }
        mbar_expect_tx(&full[stage], C_::KBYTES + (withv ? C_::VBYTES : 0));
        issued[stage] = (int)phase;
        uint8_t* sk = sst + stage * C_::STAGE;
#pragma unroll
        for (int c = 0; c < HD / 64; ++c) tma3d(sk + c * 16384, &tqk, &full[stage], xk + 64 * c, j * KB, b);
        if (withv) {
          uint8_t* sv = sk + C_::KBYTES;
#pragma unroll
          for (int kh = 0; kh < 2; ++kh)
#pragma unroll
            for (int nb = 0; nb < HD / 64; ++nb)
              tma3d(sv + (kh * (HD / 64) + nb) * 8192, &tvv, &full[stage], xv + 64 * nb, j * KB + 64 * kh, b);
        }
        if (++stage == C_::STAGES) { stage = 0; phase ^= 1u; }
      }
      if (!ok) {   // unwinding: let the copies in flight land before the CTA exits
        for (int s = 0; s < C_::STAGES; ++s) {
          if (issued[s] < 0) continue;
          const unsigned long long t0 = gtimer();
          while (!mbar_test(&full[s], (uint32_t)issued[s]) && gtimer() - t0 < 100000000ull) {
          }
        }
        const unsigned long long t0 = gtimer();
        while (!mbar_test(qfull, 0) && gtimer() - t0 < 100000000ull) {
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (one thread) ----------------
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_f16(QB, KB, false, false);
      constexpr uint32_t id_o = idesc_f16(QB, HD, false, true);
      const uint32_t tso = tmem + 256;   // O
      bool ok = mbar_wait(qfull, 0, abort_flag, err);
      fence_after();
      int stage = 0, pstage = 0;
      uint32_t phase = 0;
      const uint32_t q_addr = su32(sq), p_addr = su32(sp);
      // P V of pass-2 block jb, reading the V tile of the stage that held it; frees that stage and P
      auto pv = [&](int jb, int st) -> bool {
        if (!mbar_wait(pfull, (uint32_t)(jb & 1), abort_flag, err)) return false;
        fence_after();
        const uint32_t v_addr = su32(sst + st * C_::STAGE + C_::KBYTES);
#pragma unroll
        for (int ks = 0; ks < KB / 16; ++ks) {
          const int kh = ks / 4, kr = ks % 4;
          const uint64_t ad = sdesc(p_addr + kh * 16384 + kr * 32, 16, 1024);
          const uint64_t bd = sdesc(v_addr + kh * (HD / 64) * 8192 + kr * 2048, 8192, 1024);
          mma_bf16(tso, ad, bd, id_o, (jb > 0 || ks > 0) ? 1u : 0u);
        }
        mma_commit(&empty[st]);
        mma_commit(pempty);
        return true;
      };
      for (int it = 0; ok && it < total; ++it) {
        const int sb = it & 1;
        if (!mbar_wait(&sempty[sb], ((uint32_t)(it >> 1) & 1u) ^ 1u, abort_flag, err)) { ok = false; break; }
        if (!mbar_wait(&full[stage], phase, abort_flag, err)) { ok = false; break; }
        fence_after();
        const uint32_t k_addr = su32(sst + stage * C_::STAGE);
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          const int kq = ks / 4, kr = ks % 4;
          const uint64_t ad = sdesc(q_addr + kq * 16384 + kr * 32, 16, 1024);
          const uint64_t bd = sdesc(k_addr + kq * 16384 + kr * 32, 16, 1024);
          mma_bf16(tmem + sb * 128, ad, bd, id_s, ks > 0 ? 1u : 0u);
        }
        mma_commit(&sfull[sb]);
        if (it < nkb) {
          mma_commit(&empty[stage]);   // pass 1: the K tile is done
        } else if (it > nkb) {
          if (!pv(it - nkb - 1, pstage)) { ok = false; break; }   // the previous block's P V
        }
        if (it >= nkb) pstage = stage;   // the stage this pass-2 block's V sits in
        if (++stage == C_::STAGES) { stage = 0; phase ^= 1u; }
      }
      if (ok && !pv(nkb - 1, pstage)) ok = false;
      if (ok) mma_commit(ofull);
      mma_commit(fin);   // every MMA of this thread completes before TMEM is released
    }
  } else {
    // ---------------- softmax and output: warps 2..9, one query row per thread ----------------
    const int quad = warp & 3, half = (warp - 2) / 4;    // TMEM lane quadrant; key half of every block
    const int r = quad * 32 + lane;                       // row within the block = TMEM lane
    const int q = q0 + r;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const float sl2 = scale * kL2e;
    float m = -INFINITY, l = 0.f, lse2 = 0.f;
    bool ok = true;
    for (int it = 0; it < total; ++it) {
      const int sb = it & 1;
      const bool pass2 = it >= nkb;
      const int j = pass2 ? it - nkb : it;
      int w = 1;
      if (lane == 0) w = mbar_wait(&sfull[sb], (uint32_t)(it >> 1) & 1u, abort_flag, err) ? 1 : 0;
      w = __shfl_sync(0xffffffffu, w, 0);
      if (!w) { ok = false; break; }
      fence_after();
      // keys of this half a row may see: k <= q (causal) and k < S
      const int kmax = min(q, S - 1) - j * KB - half * 64;   // last visible key offset in the half
      const uint32_t tcol = trow + (uint32_t)(sb * 128 + half * 64);
      if (!pass2) {
#pragma unroll 1
        for (int c = 0; c < 64; c += 32) {
          float v[32];
          tmem_ld32(tcol + (uint32_t)c, v);
          float mc = -INFINITY;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            v[e] = c + e <= kmax ? v[e] * sl2 : -INFINITY;
            mc = fmaxf(mc, v[e]);
          }
          const float mn = fmaxf(m, mc);
          if (mn > -INFINITY) {
            float sum = 0.f;
#pragma unroll
            for (int e = 0; e < 32; ++e) sum += ex2(v[e] - mn);
            l = l * ex2(m - mn) + sum;
            m = mn;
          }
        }
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sempty[sb]);
        if (j == nkb - 1) {   // merge the two halves' statistics of the row (bounded wait)
          stat[(half * QB + r) * 2] = m;
          stat[(half * QB + r) * 2 + 1] = l;
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(statb);
            w = mbar_wait(statb, 0, abort_flag, err) ? 1 : 0;
          }
          w = __shfl_sync(0xffffffffu, w, 0);
          __syncwarp();   // lane 0's acquire orders the partner warp's statistics for the whole warp
          if (!w) { ok = false; break; }
          const float mo = stat[((1 - half) * QB + r) * 2], lo = stat[((1 - half) * QB + r) * 2 + 1];
          const float mt = fmaxf(m, mo);
          const float lt = mt > -INFINITY ? l * ex2(m - mt) + lo * ex2(mo - mt) : 0.f;
          lse2 = lt > 0.f ? mt + log2f(lt) : INFINITY;   // rows with no key: P = 0
        }
      } else {
        // P may be written once the previous block's P V has read it
        if (lane == 0) w = mbar_wait(pempty, ((uint32_t)j & 1u) ^ 1u, abort_flag, err) ? 1 : 0;
        w = __shfl_sync(0xffffffffu, w, 0);
        if (!w) { ok = false; break; }
        uint8_t* prow = sp + half * 16384 + r * 128;   // this half's P block, row r (128-byte swizzle)
#pragma unroll 1
        for (int c = 0; c < 64; c += 32) {
          float v[32];
          tmem_ld32(tcol + (uint32_t)c, v);
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const float p0 = c + e <= kmax ? ex2(fmaf(v[e], sl2, -lse2)) : 0.f;
            const float p1 = c + e + 1 <= kmax ? ex2(fmaf(v[e + 1], sl2, -lse2)) : 0.f;
            __nv_bfloat162 hv = __floats2bfloat162_rn(p0, p1);
            pk[e / 2] = *reinterpret_cast<uint32_t*>(&hv);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int piece = c / 8 + u;
            *reinterpret_cast<uint4*>(prow + ((piece ^ (r & 7)) << 4)) =
                make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
          }
        }
        fence_before();
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&sempty[sb]);
          mbar_arrive(pfull);
        }
      }
    }
    // output: O = sum_j P_j V_j is already normalised; each warp of a quadrant stores half of the columns
    if (ok) {
      int w = 1;
      if (lane == 0) w = mbar_wait(ofull, 0, abort_flag, err) ? 1 : 0;
      w = __shfl_sync(0xffffffffu, w, 0);
      if (w) {
        fence_after();
        bf16* orow = out + ((size_t)b * S + min(q, S - 1)) * ((size_t)H * HD) + (size_t)h * HD;
#pragma unroll 1
        for (int c = half * (HD / 2); c < (half + 1) * (HD / 2); c += 32) {   // every lane loads (tcgen05.ld is
          float v[32];                                                        // warp-wide); rows >= S store nothing
          tmem_ld32(tmem + 256 + ((uint32_t)(quad * 32) << 16) + (uint32_t)c, v);
          if (q < S) {
#pragma unroll
            for (int u = 0; u < 4; ++u) Vec8<bf16>::store(orow + c + 8 * u, v + 8 * u);
          }
        }
        if (q < S && half == 0) lse[((size_t)b * H + h) * S + q] = lse2 * kLn2;
      }
    }
  }

  fence_before();
  __syncthreads();
  if (warp == 1) {
    if (lane == 0) {
      const unsigned long long t0 = gtimer();
      while (!mbar_test(fin, 0) && gtimer() - t0 < 100000000ull) {
      }
    }
    __syncwarp();
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)C_::TMEM_COLS)
                 : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;

bool enc_init() {
  static int avail = -1;
  if (avail >= 0) return avail == 1;
  avail = 0;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3) return false;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult qr;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &qr) != cudaSuccess ||
      qr != cudaDriverEntryPointSuccess || !fn)
    return false;
  g_enc = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  avail = 1;
  return true;
}

// 3-D map over qkv viewed as [B][S][W] bf16 (W = (H + 2 Hkv) hd), box [1][rows][64], 128-byte swizzle.
bool qkv_map(CUtensorMap* m, const void* qkv, int B, int S, int W, int rows) {
  cuuint64_t dims[3] = {(cuuint64_t)W, (cuuint64_t)S, (cuuint64_t)B};
  cuuint64_t strides[2] = {(cuuint64_t)W * 2, (cuuint64_t)S * W * 2};
  cuuint32_t box[3] = {64u, (cuuint32_t)rows, 1u};
  cuuint32_t es[3] = {1, 1, 1};
  return g_enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(qkv), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int HD>
bool fwd_launch(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, cudaStream_t s, unsigned* err) {
  using C_ = FCfg<HD>;
  static bool attr = false;
  auto kern = attn_fwd_tg_k<HD>;
  if (!attr) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C_::SMEM) != cudaSuccess) return false;
    attr = true;
  }
  const int W = (H + 2 * Hkv) * HD;
  CUtensorMap tqk, tvv;
  if (!qkv_map(&tqk, qkv, B, S, W, 128) || !qkv_map(&tvv, qkv, B, S, W, 64)) return false;
  const dim3 grid(H, B, (S + QB - 1) / QB);
  return launch_pdl(kern, grid, NTHR, C_::SMEM, s, tqk, tvv, (bf16*)out, lse, S, H, Hkv, 1.f / sqrtf((float)HD),
                    err) == cudaSuccess;
}

}  // namespace tg

// Returns false when the shape is outside this kernel: head dim 128 only (at 64 the mma.sync kernel is
// faster: a 128-row block has too little matrix work to cover this kernel's per-block latency, see the
// design notes), alignment, no sm_103a. The caller uses the mma.sync kernel then.
bool attn_fwd_tcgen05(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s,
                      unsigned* err) {
  if (hd != 128) return false;
  if (((uintptr_t)qkv & 15u) || ((uintptr_t)out & 15u) || B > 65535 || (S + tg::QB - 1) / tg::QB > 65535) return false;
  if (!tg::enc_init()) return false;
  note_launch(1);
  return tg::fwd_launch<128>(qkv, out, lse, B, S, H, Hkv, s, err);
}

}  // namespace zl
