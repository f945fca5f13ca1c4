// Causal attention on the 5th-generation tensor cores (sm_103a), head dims 64 and 128: a persistent
// one-pass forward with lazy rescaling and a two-kernel backward (dQ; dK and dV) with 64-row (head dim
// 128) or 128-row (head dim 64) inner blocks.
//
// A tile is 128 rows of one (batch, head): the forward runs at most one CTA per SM over a deal of the
// tiles, the backward kernels one CTA per tile. TMA brings a tile's fixed operands once and the streamed
// tiles through a stage ring (128-byte swizzle; a 3-D tensor map over [batch, token, feature] reads rows past
// the sequence end as zeros); one elected lane of the MMA warp issues tcgen05.mma with fp32
// accumulators in TMEM; the elementwise warps own TMEM lane quadrants (one row per thread). Every
// mbarrier wait is bounded (about 2 s); on expiry the kernel raises ZL_DEVERR_TIMEOUT and unwinds.
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

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ==============================================================================================
// Forward, one pass with lazy rescaling, persistent. Each CTA takes its share of the tiles (128 query
// rows of one batch and head; snake_tile's deal of a longest-first order), so the next tile's Q and K/V
// loads and first S product overlap the current tile's last softmax block and its output; the output
// accumulator O is double-buffered in TMEM by tile parity. Per 128-key block j: S_j = Q K_j^T (TMEM,
// double-buffered), then O += P_{j-1} V_{j-1} (across a tile boundary: the previous tile's last block).
// The softmax warps (two per lane quadrant, one 64-key half each) exchange the half-row maxima of S_j
// through shared memory, so both take the same decisions, and keep a running maximum m that moves only
// when the block maximum exceeds it by more than 8 (log2 units): P = 2^(s - m) then stays at most 256
// (exact in fp32 sums, the usual bf16 rounding), and O and the row sum l are rescaled (in TMEM /
// registers) only on such a move. The rescale happens after the wait that P's buffer is free, which is
// also the completion of the previous P V product, so no product touches O meanwhile. At the end O / l
// is the softmax-weighted sum and m + log2 l the row's log-sum-exp. Barrier phases follow global block
// and tile counters, so they run on across tiles.
// ==============================================================================================
template <int HD>
struct F1Cfg {
  static constexpr int QBYTES = QB * HD * 2;
  static constexpr int KBYTES = KB * HD * 2;
  static constexpr int VBYTES = KB * HD * 2;
  static constexpr int STAGES = HD == 64 ? 4 : 2;
  static constexpr int STAGE = KBYTES + VBYTES;
  static constexpr int PBYTES = QB * KB * 2;
  static constexpr int XBYTES = (2 * 2 * QB + 2 * QB) * 4;   // maxima [2 buffers][2 halves][rows], sums [2][rows]
  static constexpr int SMEM = QBYTES + STAGES * STAGE + PBYTES + XBYTES + 256 + 1024;
  static constexpr uint32_t OCOL = 256;                        // O of even tiles; odd tiles at OCOL + HD
  static_assert(SMEM <= 232448, "shared memory per CTA");
  static_assert(OCOL + 2 * HD <= 512, "TMEM columns");
};

// The it-th tile of CTA c among G: the tiles are sorted longest first and dealt out G at a time, the
// direction alternating between deals (deal 0: c, deal 1: 2G - 1 - c, ...), so every CTA's long and short
// tiles even out; past the last tile it returns a value >= every tile count (every later deal is past it
// too).
__device__ __forceinline__ int snake_tile(int it, int c, int G) {
  return (it & 1) ? (it + 1) * G - 1 - c : it * G + c;
}

// Tile t of the longest-first order: query block (longest first), then batch, then head (heads that share
// a K/V head are adjacent, so their K/V tiles come from L2).
__device__ __forceinline__ void fwd_tile(int t, int H, int B, int nqb, int& h, int& b, int& qb) {
  const int hb = H * B;
  qb = nqb - 1 - t / hb;
  const int r = t % hb;
  h = r % H;
  b = r / H;
}

template <int HD>
__global__ void __launch_bounds__(NTHR, 1)
    attn_fwd1_tg_k(const __grid_constant__ CUtensorMap tqk, const __grid_constant__ CUtensorMap tvv,
                   bf16* __restrict__ out, float* __restrict__ lse, int S, int B, int H, int Hkv, float scale,
                   unsigned* err) {
  using C_ = F1Cfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sq = smem;
  uint8_t* sst = sq + C_::QBYTES;                      // stages: K tile, then V tile
  uint8_t* sp = sst + C_::STAGES * C_::STAGE;          // P
  float* xmax = (float*)(sp + C_::PBYTES);             // [2][2][QB]
  float* xsum = xmax + 4 * QB;                         // [2][QB]
  uint64_t* full = (uint64_t*)(xsum + 2 * QB);
  uint64_t* empty = full + C_::STAGES;
  uint64_t* qfull = empty + C_::STAGES;
  uint64_t* qempty = qfull + 1;
  uint64_t* sfull = qempty + 1;                        // [2]
  uint64_t* sempty = sfull + 2;                        // [2]
  uint64_t* pfull = sempty + 2;
  uint64_t* pempty = pfull + 1;
  uint64_t* ofull = pempty + 1;                        // [2]
  uint64_t* oempty = ofull + 2;                        // [2]
  uint64_t* fin = oempty + 2;
  uint32_t* tbase = (uint32_t*)(fin + 1);
  volatile int* abort_flag = (volatile int*)(tbase + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqb = (S + QB - 1) / QB, ntiles = nqb * B * H;
  const int group = H / Hkv;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C_::STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(qfull, 1);
    mbar_init(qempty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sfull[i], 1);
      mbar_init(&sempty[i], NSM);
      mbar_init(&ofull[i], 1);
      mbar_init(&oempty[i], NSM);
    }
    mbar_init(pfull, NSM);
    mbar_init(pempty, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tbase)), "r"(512u)
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
    // ---------------- TMA producer (whole warp, one elected lane issues) ----------------
    const bool leader = elect_one();
    bool ok = true;
    int qlast = -1;   // tile count of the last Q load issued
    int issued[C_::STAGES];
#pragma unroll
    for (int s = 0; s < C_::STAGES; ++s) issued[s] = -1;
    int stage = 0, it = 0;
    uint32_t phase = 0;
    for (; ok; ++it) {
      const int t = snake_tile(it, blockIdx.x, gridDim.x);
      if (t >= ntiles) break;
      int h, b, qb;
      fwd_tile(t, H, B, nqb, h, b, qb);
      const int kvh = h / group, nkb = qb + 1;
      const int xq = h * HD, xk = (H + kvh) * HD, xv = (H + Hkv + kvh) * HD;
      // Q's buffer is free once the previous tile's S products have completed
      if (!uwait(qempty, ((uint32_t)it & 1u) ^ 1u, abort_flag, err)) { ok = false; break; }
      qlast = it;
      if (leader) {
        mbar_expect_tx(qfull, C_::QBYTES);
#pragma unroll
        for (int c = 0; c < HD / 64; ++c) tma3d(sq + c * 16384, &tqk, qfull, xq + 64 * c, qb * QB, b);
      }
      __syncwarp();
      for (int j = 0; j < nkb; ++j) {
        if (!uwait(&empty[stage], phase ^ 1u, abort_flag, err)) { ok = false; break; }
        issued[stage] = (int)phase;
        if (leader) {
          mbar_expect_tx(&full[stage], C_::STAGE);
          uint8_t* sk = sst + stage * C_::STAGE;
          uint8_t* sv = sk + C_::KBYTES;
#pragma unroll
          for (int c = 0; c < HD / 64; ++c) tma3d(sk + c * 16384, &tqk, &full[stage], xk + 64 * c, j * KB, b);
#pragma unroll
          for (int kh = 0; kh < 2; ++kh)
#pragma unroll
            for (int nb = 0; nb < HD / 64; ++nb)
              tma3d(sv + (kh * (HD / 64) + nb) * 8192, &tvv, &full[stage], xv + 64 * nb, j * KB + 64 * kh, b);
        }
        __syncwarp();
        if (++stage == C_::STAGES) { stage = 0; phase ^= 1u; }
      }
    }
    if (!ok && lane == 0) {   // unwinding: let the copies in flight land before the CTA exits
      for (int s = 0; s < C_::STAGES; ++s) {
        if (issued[s] < 0) continue;
        const unsigned long long t0 = gtimer();
        while (!mbar_test(&full[s], (uint32_t)issued[s]) && gtimer() - t0 < 100000000ull) {
        }
      }
      if (qlast >= 0) {   // the last Q load (phase parity = its tile count)
        const unsigned long long t0 = gtimer();
        while (!mbar_test(qfull, (uint32_t)qlast & 1u) && gtimer() - t0 < 100000000ull) {
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (whole warp, one elected lane issues and commits) ----------------
    constexpr uint32_t id_s = idesc_f16(QB, KB, false, false);
    constexpr uint32_t id_o = idesc_f16(QB, HD, false, true);
    const bool leader = elect_one();
    bool ok = true;
    int stage = 0, jg = 0, it = 0;
    uint32_t phase = 0;
    const uint32_t q_addr = su32(sq), p_addr = su32(sp);
    // the P V product still to issue: block jl (of its tile) with global index pg, in stage pst, of tile pit
    struct Pending { bool on; int jl, pg, pst, pit; bool last; } pend{false, 0, 0, 0, 0, false};
    // O[tile parity] += P V: waits for P (and, on a tile's first block, for O's buffer to be read out);
    // then the stage and P are free, and after a tile's last block O is complete
    auto pv = [&](const Pending& p) -> bool {
      if (!uwait(pfull, (uint32_t)p.pg & 1u, abort_flag, err)) return false;
      const int ob = p.pit & 1;
      if (p.jl == 0 && !uwait(&oempty[ob], ((uint32_t)(p.pit >> 1) & 1u) ^ 1u, abort_flag, err)) return false;
      fence_after();
      if (leader) {
        const uint32_t tso = tmem + C_::OCOL + (uint32_t)(ob * HD);
        const uint32_t v_addr = su32(sst + p.pst * C_::STAGE + C_::KBYTES);
#pragma unroll
        for (int ks = 0; ks < KB / 16; ++ks) {
          const int kh = ks / 4, kr = ks % 4;
          const uint64_t ad = sdesc(p_addr + kh * 16384 + kr * 32, 16, 1024);
          const uint64_t bd = sdesc(v_addr + kh * (HD / 64) * 8192 + kr * 2048, 8192, 1024);
          mma_bf16(tso, ad, bd, id_o, (p.jl > 0 || ks > 0) ? 1u : 0u);
        }
        mma_commit(&empty[p.pst]);
        mma_commit(pempty);
        if (p.last) mma_commit(&ofull[ob]);
      }
      __syncwarp();
      return true;
    };
    for (; ok; ++it) {
      const int t = snake_tile(it, blockIdx.x, gridDim.x);
      if (t >= ntiles) break;
      int h, b, qb;
      fwd_tile(t, H, B, nqb, h, b, qb);
      const int nkb = qb + 1;
      if (!uwait(qfull, (uint32_t)it & 1u, abort_flag, err)) { ok = false; break; }
      for (int j = 0; j < nkb; ++j, ++jg) {
        const int sb = jg & 1;
        if (!uwait(&sempty[sb], ((uint32_t)(jg >> 1) & 1u) ^ 1u, abort_flag, err) ||
            !uwait(&full[stage], phase, abort_flag, err)) {
          ok = false;
          break;
        }
        fence_after();
        if (leader) {
          const uint32_t k_addr = su32(sst + stage * C_::STAGE);
#pragma unroll
          for (int ks = 0; ks < HD / 16; ++ks) {
            const int kq = ks / 4, kr = ks % 4;
            mma_bf16(tmem + sb * 128, sdesc(q_addr + kq * 16384 + kr * 32, 16, 1024),
                     sdesc(k_addr + kq * 16384 + kr * 32, 16, 1024), id_s, ks > 0 ? 1u : 0u);
          }
          mma_commit(&sfull[sb]);
          if (j == nkb - 1) mma_commit(qempty);   // Q is free once the tile's last S product completes
        }
        __syncwarp();
        if (pend.on && !pv(pend)) { ok = false; break; }
        pend = Pending{true, j, jg, stage, it, j == nkb - 1};
        if (++stage == C_::STAGES) { stage = 0; phase ^= 1u; }
      }
    }
    if (ok && pend.on && !pv(pend)) ok = false;
    if (leader) mma_commit(fin);   // every MMA of the leader completes before TMEM is released
    __syncwarp();
  } else {
    // ---------------- softmax and output: warps 2..9, one query row per thread ----------------
    const int quad = warp & 3, half = (warp - 2) / 4;    // TMEM lane quadrant; key half of every block
    const int r = quad * 32 + lane;                       // row within the block = TMEM lane
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const float sl2 = scale * kL2e;
    // A failed wait only skips work: both warps of a quadrant still pass every named barrier (the same
    // tiles and blocks on both).
    bool ok = true;
    int jg = 0, it = 0;
    for (;; ++it) {
      const int t = snake_tile(it, blockIdx.x, gridDim.x);
      if (t >= ntiles) break;
      int h, b, qb;
      fwd_tile(t, H, B, nqb, h, b, qb);
      const int nkb = qb + 1, q = qb * QB + r;
      const uint32_t ocol = C_::OCOL + (uint32_t)((it & 1) * HD);
      float m = -INFINITY, l = 0.f;                       // running maximum (log2 units), this half's sum
      for (int j = 0; j < nkb; ++j, ++jg) {
        const int sb = jg & 1;
        if (ok && !uwait(&sfull[sb], (uint32_t)(jg >> 1) & 1u, abort_flag, err)) ok = false;
        float v[64];
        float mh = -INFINITY;
        if (ok) {
          fence_after();
          const int kmax = min(q, S - 1) - j * KB - half * 64;   // last visible key offset in the half
          const uint32_t tcol = trow + (uint32_t)(sb * 128 + half * 64);
          tmem_ld32(tcol, v);
          tmem_ld32(tcol + 32u, v + 32);
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sempty[sb]);
#pragma unroll
          for (int e = 0; e < 64; ++e) {
            v[e] = e <= kmax ? v[e] * sl2 : -INFINITY;
            mh = fmaxf(mh, v[e]);
          }
        }
        // the partner half's maximum (double-buffered by block parity; one barrier per block)
        float* xm = xmax + (jg & 1) * 2 * QB;
        xm[half * QB + r] = mh;
        asm volatile("bar.sync %0, 64;" ::"r"(1 + quad) : "memory");
        if (!ok) continue;
        const float mblk = fmaxf(mh, xm[(1 - half) * QB + r]);
        const float mnew = fmaxf(m, mblk);
        const bool move = mnew > m + 8.f;   // also true on the first block (m = -inf)
        // P's buffer is free once the previous P V product has completed; O then holds blocks < j
        if (!uwait(pempty, ((uint32_t)jg & 1u) ^ 1u, abort_flag, err)) { ok = false; continue; }
        if (j > 0 && __any_sync(0xffffffffu, move)) {   // rescale this half of the O row (warp-wide TMEM access)
          const float a = move ? ex2(m - mnew) : 1.f;
          l *= a;
          fence_after();
#pragma unroll 1
          for (int c = half * (HD / 2); c < (half + 1) * (HD / 2); c += 32) {
            float o[32];
            tmem_ld32(trow + ocol + (uint32_t)c, o);
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= a;
            tmem_st32(trow + ocol + (uint32_t)c, o);
          }
        }
        if (move) m = mnew;
        uint8_t* prow = sp + half * 16384 + r * 128;   // this half's P block, row r (128-byte swizzle)
        float sum = 0.f;
#pragma unroll
        for (int c = 0; c < 64; c += 32) {
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const float p0 = ex2(v[c + e] - m), p1 = ex2(v[c + e + 1] - m);   // masked scores are -inf: 0
            sum += p0 + p1;
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
        l += sum;
        fence_before();
        fence_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(pfull);
      }
      // output: both halves use the same m; O / (l_0 + l_1), log-sum-exp m + log2(l_0 + l_1)
      xsum[half * QB + r] = l;
      asm volatile("bar.sync %0, 64;" ::"r"(1 + quad) : "memory");
      if (!ok) continue;
      const float lt = l + xsum[(1 - half) * QB + r];
      const float inv = lt > 0.f ? 1.f / lt : 0.f;
      if (!uwait(&ofull[it & 1], (uint32_t)(it >> 1) & 1u, abort_flag, err)) { ok = false; continue; }
      fence_after();
      bf16* orow = out + ((size_t)b * S + min(q, S - 1)) * ((size_t)H * HD) + (size_t)h * HD;
#pragma unroll 1
      for (int c = half * (HD / 2); c < (half + 1) * (HD / 2); c += 32) {   // every lane loads (tcgen05.ld is
        float o[32];                                                        // warp-wide); rows >= S store nothing
        tmem_ld32(trow + ocol + (uint32_t)c, o);
        if (q < S) {
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] *= inv;
#pragma unroll
          for (int u = 0; u < 4; ++u) Vec8<bf16>::store(orow + c + 8 * u, o + 8 * u);
        }
      }
      // this warp's half of O has been read: the buffer may take the tile after next
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&oempty[it & 1]);
      if (q < S && half == 0) lse[((size_t)b * H + h) * S + q] = (lt > 0.f ? m + log2f(lt) : INFINITY) * kLn2;
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
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512u) : "memory");
  }
}

// ==============================================================================================
// Backward: two kernels, each a fixed-order sum per output row (no atomics). Head dim 128 runs the
// kernels of this section (64-row inner blocks); head dim 64 the 128-row variant that follows them.
//   dQ kernel: one CTA per 128 queries; 64-key inner blocks j: S = Q K_j^T, dP = dO V_j^T (TMEM),
//              dS = P * (dP - D) (shared memory, bf16), dQ += dS K_j (TMEM); also writes D = rowsum(dO * O).
//   dK/dV kernel: one CTA per 128 keys; 64-query inner blocks i: S^T = K Q_i^T, dP^T = V dO_i^T,
//              P^T and dS^T (shared memory), dV += P^T dO_i, dK += dS^T Q_i.
// The 128 x 64 S / dP blocks are double-buffered in TMEM (columns 0 and 128, dP 64 columns after S); the
// accumulators start at column 256. A 64-row tile of Q / dO / K / V is one K-major [64 x 64] block per 64
// head-dim columns (8 KB each); the same bytes are the MN-major B operand of the accumulating product
// (16-row steps 2 KB apart, head-dim blocks 8 KB apart).
// ==============================================================================================
constexpr int IB = 64;   // inner block rows
constexpr int NEW = 16;  // elementwise warps: two groups of eight (two per TMEM lane quadrant, one
                         // 32-column half each); group g takes the inner blocks of parity g
constexpr int NTHR_B = 64 + 32 * NEW;

template <int HD>
struct BCfg {
  static constexpr int T128 = 128 * HD * 2;
  static constexpr int T64 = IB * HD * 2;
  static constexpr int NST = HD == 64 ? 4 : 3;   // pipeline stages of (Q_i, dO_i) or (K_j, V_j)
  static constexpr int OPB = 128 * IB * 2;       // one bf16 [128 x 64] operand (P^T, dS^T or dS)
  // K, V | stages | P^T, dS^T double-buffered | stats (-lse2, D) per stage | barriers | alignment
  static constexpr int SMEM_DKV = 2 * T128 + NST * 2 * T64 + 4 * OPB + NST * 2 * IB * 4 + 256 + 1024;
  // Q, dO | stages | dS double-buffered | D quarters | barriers | alignment
  static constexpr int SMEM_DQ = 2 * T128 + NST * 2 * T64 + 2 * OPB + 4 * 128 * 4 + 256 + 1024;
  static_assert(SMEM_DKV <= 232448 && SMEM_DQ <= 232448, "shared memory per CTA");
};

// Stores 16 bf16 values (32 bytes: 16-byte chunks 2 qu and 2 qu + 1) into row r of a swizzled
// [128 x 64] K-major operand.
__device__ __forceinline__ void put_row16(uint8_t* g, int qu, int r, const uint32_t* pk) {
  uint8_t* row = g + r * 128;
#pragma unroll
  for (int u = 0; u < 2; ++u)
    *reinterpret_cast<uint4*>(row + (((2 * qu + u) ^ (r & 7)) << 4)) =
        make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Lane 0 of the producer, after a failed wait: lets the copies it issued land (bounded) before exit.
template <int N>
__device__ __forceinline__ void drain(uint64_t* full, const int* issued, uint64_t* first) {
  for (int s = 0; s < N; ++s) {
    if (issued[s] < 0) continue;
    const unsigned long long t0 = gtimer();
    while (!mbar_test(&full[s], (uint32_t)issued[s]) && gtimer() - t0 < 100000000ull) {
    }
  }
  const unsigned long long t0 = gtimer();
  while (!mbar_test(first, 0) && gtimer() - t0 < 100000000ull) {
  }
}

__device__ __forceinline__ void tmem_alloc512(uint32_t* dst) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(dst)), "r"(512u)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

// Warp 1 after the final __syncthreads: waits (bounded) for the last MMAs, frees the TMEM.
__device__ __forceinline__ void tmem_release(uint64_t* fin, uint32_t tmem) {
  if ((threadIdx.x & 31) == 0) {
    const unsigned long long t0 = gtimer();
    while (!mbar_test(fin, 0) && gtimer() - t0 < 100000000ull) {
    }
  }
  __syncwarp();
  fence_after();
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512u) : "memory");
}

// The TMA and MMA warps run their loops with the whole warp (uniform control flow, so addresses and
// descriptors stay in uniform registers); one elected lane issues each group of copies or products.

// dQ (and D) kernel. Maps: tq = qkv in 128-row boxes, tdo = dO in 128-row boxes, tkv = qkv in 64-row boxes.
template <int HD>
__global__ void __launch_bounds__(NTHR_B, 1)
    attn_bwd_dq_tg_k(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tdo,
                     const __grid_constant__ CUtensorMap tkv, const bf16* __restrict__ outp,
                     const bf16* __restrict__ dout, const float* __restrict__ lse, float* __restrict__ Dv,
                     bf16* __restrict__ dqkv, int S, int H, int Hkv, float scale, unsigned* err) {
  using C_ = BCfg<HD>;
  constexpr int NST = C_::NST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sq = smem;
  uint8_t* sdo = sq + C_::T128;
  uint8_t* sst = sdo + C_::T128;                  // stage s: K_j at s * 2 T64, V_j after it
  uint8_t* sds = sst + NST * 2 * C_::T64;         // dS, two buffers
  float* dpart = (float*)(sds + 2 * C_::OPB);     // [4][128] quarters of D
  uint64_t* full = (uint64_t*)(dpart + 512);
  uint64_t* empty = full + NST;
  uint64_t* qfull = empty + NST;
  uint64_t* sfull = qfull + 1;                    // [2]
  uint64_t* sempty = sfull + 2;                   // [2]
  uint64_t* dsfull = sempty + 2;                  // [2]
  uint64_t* dsempty = dsfull + 2;                 // [2]
  uint64_t* ofull = dsempty + 2;
  uint64_t* fin = ofull + 1;
  uint32_t* tbase = (uint32_t*)(fin + 1);
  volatile int* abort_flag = (volatile int*)(tbase + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, b = blockIdx.y, qb = gridDim.z - 1 - blockIdx.z;   // longest first
  const int kvh = h / (H / Hkv);
  const int q0 = qb * 128;
  const int nkb = min(2 * qb + 2, (S + IB - 1) / IB);
  const int ld = (H + 2 * Hkv) * HD, HDall = H * HD;
  const int xq = h * HD, xk = (H + kvh) * HD, xv = (H + Hkv + kvh) * HD;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(qfull, 1);
    for (int u = 0; u < 2; ++u) {   // buffer u is used by elementwise group u only
      mbar_init(&sfull[u], 1);
      mbar_init(&sempty[u], NEW / 2);
      mbar_init(&dsfull[u], NEW / 2);
      mbar_init(&dsempty[u], 1);
    }
    mbar_init(ofull, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc512(tbase);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tbase;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    int issued[NST];
#pragma unroll
    for (int s = 0; s < NST; ++s) issued[s] = -1;
    const bool leader = elect_one();
    if (leader) {
      mbar_expect_tx(qfull, 2 * C_::T128);
#pragma unroll
      for (int c = 0; c < HD / 64; ++c) {
        tma3d(sq + c * 16384, &tq, qfull, xq + 64 * c, q0, b);
        tma3d(sdo + c * 16384, &tdo, qfull, h * HD + 64 * c, q0, b);
      }
    }
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      if (!uwait(&empty[stage], phase ^ 1u, abort_flag, err)) { ok = false; break; }
      issued[stage] = (int)phase;
      if (leader) {
        mbar_expect_tx(&full[stage], 2 * C_::T64);
        uint8_t* st = sst + stage * 2 * C_::T64;
#pragma unroll
        for (int c = 0; c < HD / 64; ++c) {
          tma3d(st + c * 8192, &tkv, &full[stage], xk + 64 * c, j * IB, b);
          tma3d(st + C_::T64 + c * 8192, &tkv, &full[stage], xv + 64 * c, j * IB, b);
        }
      }
      __syncwarp();
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (!ok && lane == 0) drain<NST>(full, issued, qfull);
  } else if (warp == 1) {
    constexpr uint32_t id_s = idesc_f16(128, IB, false, false);
    constexpr uint32_t id_q = idesc_f16(128, HD, false, true);
    const uint32_t q_addr = su32(sq), do_addr = su32(sdo), ds_addr = su32(sds);
    const bool leader = elect_one();   // issues every product and every commit that tracks them
    bool ok = uwait(qfull, 0, abort_flag, err);
    fence_after();
    int stage = 0, pstage = 0;
    uint32_t phase = 0;
    auto dq = [&](int jb, int st) -> bool {   // dQ += dS_jb K_jb
      const int db = jb & 1;
      if (!uwait(&dsfull[db], (uint32_t)(jb >> 1) & 1u, abort_flag, err)) return false;
      fence_after();
      if (leader) {
        const uint32_t k_addr = su32(sst + st * 2 * C_::T64), a_addr = ds_addr + db * C_::OPB;
#pragma unroll
        for (int ks = 0; ks < IB / 16; ++ks)
          mma_bf16(tmem + 256, sdesc(a_addr + ks * 32, 16, 1024), sdesc(k_addr + ks * 2048, 8192, 1024), id_q,
                   (jb > 0 || ks > 0) ? 1u : 0u);
        mma_commit(&empty[st]);
        mma_commit(&dsempty[db]);
      }
      __syncwarp();
      return true;
    };
    for (int j = 0; ok && j < nkb; ++j) {
      const int buf = j & 1;
      if (!uwait(&sempty[buf], ((uint32_t)(j >> 1) & 1u) ^ 1u, abort_flag, err) ||
          !uwait(&full[stage], phase, abort_flag, err)) {
        ok = false;
        break;
      }
      fence_after();
      if (leader) {
        const uint32_t k_addr = su32(sst + stage * 2 * C_::T64), v_addr = k_addr + C_::T64;
        const uint32_t ts = tmem + (uint32_t)(buf * 128);
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          const int kq = ks / 4, kr = ks % 4;
          mma_bf16(ts, sdesc(q_addr + kq * 16384 + kr * 32, 16, 1024), sdesc(k_addr + kq * 8192 + kr * 32, 16, 1024),
                   id_s, ks > 0 ? 1u : 0u);
          mma_bf16(ts + IB, sdesc(do_addr + kq * 16384 + kr * 32, 16, 1024),
                   sdesc(v_addr + kq * 8192 + kr * 32, 16, 1024), id_s, ks > 0 ? 1u : 0u);
        }
        mma_commit(&sfull[buf]);
      }
      __syncwarp();
      if (j > 0 && !dq(j - 1, pstage)) { ok = false; break; }
      pstage = stage;
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (ok && !dq(nkb - 1, pstage)) ok = false;
    if (leader) {
      if (ok) mma_commit(ofull);
      mma_commit(fin);
    }
    __syncwarp();
  } else {
    const int quad = warp & 3, qu = (warp - 2) / 4;   // TMEM lane quadrant, 16-column quarter
    const int r = quad * 32 + lane;
    const int q = q0 + r, qc = min(q, S - 1);
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const size_t si = ((size_t)b * H + h) * S + qc;
    const float nlse2 = q < S ? -lse[si] * kL2e : -INFINITY;
    {   // D = rowsum(dO * O): each quarter sums a quarter of the row, fixed-order combination
      const bf16* orow = outp + ((size_t)b * S + qc) * HDall + (size_t)h * HD + qu * (HD / 4);
      const bf16* grow = dout + ((size_t)b * S + qc) * HDall + (size_t)h * HD + qu * (HD / 4);
      float acc = 0.f;
#pragma unroll
      for (int c = 0; c < HD / 4; c += 8) {
        float o8[8], g8[8];
        Vec8<bf16>::load(orow + c, o8);
        Vec8<bf16>::load(grow + c, g8);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc = fmaf(o8[e], g8[e], acc);
      }
      dpart[qu * 128 + r] = acc;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(32 * NEW) : "memory");
    const float Dq = (dpart[r] + dpart[128 + r]) + (dpart[256 + r] + dpart[384 + r]);
    if (q < S && qu == 0) Dv[si] = Dq;
    const uint64_t SL2 = f2(scale * kL2e, scale * kL2e), NL = f2(nlse2, nlse2), DD = f2(Dq, Dq);
    const int qmin = q0 + quad * 32;   // smallest query row of this warp
    // inner blocks alternate between the two groups, so each group's chain of waits, TMEM loads,
    // arithmetic and stores has two blocks' time; a thread takes 32 columns in two 16-column passes
    const int grp = (warp - 2) >> 3, half = ((warp - 2) >> 2) & 1;
    bool ok = true;
    for (int j = grp; j < nkb; j += 2) {
      const int buf = j & 1;
      if (!uwait(&sfull[buf], (uint32_t)(j >> 1) & 1u, abort_flag, err)) { ok = false; break; }
      fence_after();
      for (int sub = 0; sub < 2; ++sub) {
        const int c0 = half * 32 + sub * 16;
        float sv[16], dp[16];
        tmem_ld16(trow + (uint32_t)(buf * 128 + c0), sv);
        tmem_ld16(trow + (uint32_t)(buf * 128 + IB + c0), dp);
        if (sub == 1) {
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sempty[buf]);
        }
        const int kbase = j * IB + c0;
        const bool diag = kbase + 15 > qmin;   // warp-uniform: some column may lie above the diagonal
        const int kmax = q - kbase;            // causal: columns e <= kmax
        uint32_t pk[8];
#pragma unroll
        for (int e = 0; e < 16; e += 2) {
          float2 x = uf2(fma2(f2(sv[e], sv[e + 1]), SL2, NL));
          if (diag) {
            if (e > kmax) x.x = -INFINITY;
            if (e + 1 > kmax) x.y = -INFINITY;
          }
          const float p0 = ex2(x.x), p1 = ex2(x.y);
          const float2 ds = uf2(mul2(f2(p0, p1), sub2(f2(dp[e], dp[e + 1]), DD)));
          pk[e / 2] = pack2(ds.x, ds.y);
        }
        if (sub == 0 && !uwait(&dsempty[buf], ((uint32_t)(j >> 1) & 1u) ^ 1u, abort_flag, err)) { ok = false; break; }
        put_row16(sds + buf * C_::OPB, c0 >> 4, r, pk);
      }
      if (!ok) break;
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&dsfull[buf]);
    }
    if (ok && uwait(ofull, 0, abort_flag, err)) {
      fence_after();
      bf16* drow = dqkv + ((size_t)b * S + qc) * ld + (size_t)h * HD;
#pragma unroll
      for (int c = qu * (HD / 4); c < (qu + 1) * (HD / 4); c += 16) {
        float v[16];
        tmem_ld16(trow + 256 + (uint32_t)c, v);
        if (q < S) {
#pragma unroll
          for (int e = 0; e < 16; ++e) v[e] *= scale;
          Vec8<bf16>::store(drow + c, v);
          Vec8<bf16>::store(drow + c + 8, v + 8);
        }
      }
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) tmem_release(fin, tmem);
}

// dK / dV kernel. One CTA per 128 keys of one query head (grouped heads: fp32 partials
// part[2][H][B*S][HD], dK unscaled, summed per group afterwards) or of one KV head (H == Hkv: bf16 straight
// into dqkv). Maps: tkv = qkv in 128-row boxes, tq = qkv in 64-row boxes, tdo = dO in 64-row boxes.
template <int HD>
__global__ void __launch_bounds__(NTHR_B, 1)
    attn_bwd_dkv_tg_k(const __grid_constant__ CUtensorMap tkv, const __grid_constant__ CUtensorMap tq,
                      const __grid_constant__ CUtensorMap tdo, const float* __restrict__ lse,
                      const float* __restrict__ Dv, bf16* __restrict__ dqkv, int S, int H, int Hkv, float scale,
                      float* __restrict__ part, unsigned* err) {
  using C_ = BCfg<HD>;
  constexpr int NST = C_::NST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sk = smem;
  uint8_t* sv = sk + C_::T128;
  uint8_t* sst = sv + C_::T128;                   // stage s: Q_i at s * 2 T64, dO_i after it
  uint8_t* sp = sst + NST * 2 * C_::T64;          // buffer u: P^T at sp + 2 u OPB, dS^T after it
  float* stats = (float*)(sp + 4 * C_::OPB);      // stage s: -lse2[64], D[64]
  uint64_t* full = (uint64_t*)(stats + NST * 2 * IB);
  uint64_t* empty = full + NST;
  uint64_t* kvfull = empty + NST;
  uint64_t* sfull = kvfull + 1;                   // [2]
  uint64_t* sempty = sfull + 2;                   // [2]
  uint64_t* pfull = sempty + 2;                   // [2]
  uint64_t* pempty = pfull + 2;                   // [2]
  uint64_t* ofull = pempty + 2;
  uint64_t* fin = ofull + 1;
  uint32_t* tbase = (uint32_t*)(fin + 1);
  volatile int* abort_flag = (volatile int*)(tbase + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, b = blockIdx.y, kb = blockIdx.z;   // key block 0 (the longest) first
  const int kvh = part ? h / (H / Hkv) : h;
  const int k0 = kb * 128, i0 = 2 * kb;
  const int nit = (S + IB - 1) / IB - i0;
  const int ld = (H + 2 * Hkv) * HD;
  const int xq = h * HD, xk = (H + kvh) * HD, xv = (H + Hkv + kvh) * HD;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) { mbar_init(&full[s], 2); mbar_init(&empty[s], 1); }
    mbar_init(kvfull, 1);
    for (int u = 0; u < 2; ++u) {   // buffer u is used by elementwise group u only
      mbar_init(&sfull[u], 1);
      mbar_init(&sempty[u], NEW / 2);
      mbar_init(&pfull[u], NEW / 2);
      mbar_init(&pempty[u], 1);
    }
    mbar_init(ofull, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc512(tbase);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tbase;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    // one elected lane: TMA of K, V once and of (Q_i, dO_i) per block; every lane: two of the block's
    // -lse2 and D
    int issued[NST];
#pragma unroll
    for (int s = 0; s < NST; ++s) issued[s] = -1;
    const bool leader = elect_one();
    if (leader) {
      mbar_expect_tx(kvfull, 2 * C_::T128);
#pragma unroll
      for (int c = 0; c < HD / 64; ++c) {
        tma3d(sk + c * 16384, &tkv, kvfull, xk + 64 * c, k0, b);
        tma3d(sv + c * 16384, &tkv, kvfull, xv + 64 * c, k0, b);
      }
    }
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    // this lane's two statistics of the next block, loaded one block ahead
    float nl[2], dd[2];
    auto fetch = [&](int it) {
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int qq = (i0 + it) * IB + lane * 2 + u;
        const size_t si = ((size_t)b * H + h) * S + (qq < S ? qq : 0);
        nl[u] = qq < S ? -lse[si] * kL2e : -INFINITY;
        dd[u] = qq < S ? Dv[si] : 0.f;
      }
    };
    fetch(0);
    for (int it = 0; it < nit; ++it) {
      const int qi0 = (i0 + it) * IB;
      if (!uwait(&empty[stage], phase ^ 1u, abort_flag, err)) { ok = false; break; }
      issued[stage] = (int)phase;
      if (leader) {
        mbar_expect_tx(&full[stage], 2 * C_::T64);
        uint8_t* st = sst + stage * 2 * C_::T64;
#pragma unroll
        for (int c = 0; c < HD / 64; ++c) {
          tma3d(st + c * 8192, &tq, &full[stage], xq + 64 * c, qi0, b);
          tma3d(st + C_::T64 + c * 8192, &tdo, &full[stage], h * HD + 64 * c, qi0, b);
        }
      }
      float* sl = stats + stage * 2 * IB;
      *reinterpret_cast<float2*>(sl + lane * 2) = make_float2(nl[0], nl[1]);
      *reinterpret_cast<float2*>(sl + IB + lane * 2) = make_float2(dd[0], dd[1]);
      __syncwarp();
      if (lane == 0) mbar_arrive(&full[stage]);
      if (it + 1 < nit) fetch(it + 1);
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (!ok && lane == 0) drain<NST>(full, issued, kvfull);
  } else if (warp == 1) {
    constexpr uint32_t id_s = idesc_f16(128, IB, false, false);
    constexpr uint32_t id_g = idesc_f16(128, HD, false, true);
    const uint32_t k_addr = su32(sk), v_addr = su32(sv), p_addr = su32(sp);
    const bool leader = elect_one();   // issues every product and every commit that tracks them
    bool ok = uwait(kvfull, 0, abort_flag, err);
    fence_after();
    int stage = 0, pstage = 0;
    uint32_t phase = 0;
    auto grads = [&](int ib, int st) -> bool {   // dV += P^T dO_ib, dK += dS^T Q_ib
      const int pb = ib & 1;
      if (!uwait(&pfull[pb], (uint32_t)(ib >> 1) & 1u, abort_flag, err)) return false;
      fence_after();
      if (leader) {
        const uint32_t qa = su32(sst + st * 2 * C_::T64), da = qa + C_::T64;
        const uint32_t pa = p_addr + pb * 2 * C_::OPB, dsa = pa + C_::OPB;
#pragma unroll
        for (int ks = 0; ks < IB / 16; ++ks) {
          const uint32_t acc = (ib > 0 || ks > 0) ? 1u : 0u;
          mma_bf16(tmem + 256, sdesc(pa + ks * 32, 16, 1024), sdesc(da + ks * 2048, 8192, 1024), id_g, acc);
          mma_bf16(tmem + 256 + HD, sdesc(dsa + ks * 32, 16, 1024), sdesc(qa + ks * 2048, 8192, 1024), id_g, acc);
        }
        mma_commit(&empty[st]);
        mma_commit(&pempty[pb]);
      }
      __syncwarp();
      return true;
    };
    for (int it = 0; ok && it < nit; ++it) {
      const int buf = it & 1;
      if (!uwait(&sempty[buf], ((uint32_t)(it >> 1) & 1u) ^ 1u, abort_flag, err) ||
          !uwait(&full[stage], phase, abort_flag, err)) {
        ok = false;
        break;
      }
      fence_after();
      if (leader) {
        const uint32_t qa = su32(sst + stage * 2 * C_::T64), da = qa + C_::T64;
        const uint32_t ts = tmem + (uint32_t)(buf * 128);
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          const int kq = ks / 4, kr = ks % 4;
          mma_bf16(ts, sdesc(k_addr + kq * 16384 + kr * 32, 16, 1024), sdesc(qa + kq * 8192 + kr * 32, 16, 1024),
                   id_s, ks > 0 ? 1u : 0u);
          mma_bf16(ts + IB, sdesc(v_addr + kq * 16384 + kr * 32, 16, 1024),
                   sdesc(da + kq * 8192 + kr * 32, 16, 1024), id_s, ks > 0 ? 1u : 0u);
        }
        mma_commit(&sfull[buf]);
      }
      __syncwarp();
      if (it > 0 && !grads(it - 1, pstage)) { ok = false; break; }
      pstage = stage;
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (ok && !grads(nit - 1, pstage)) ok = false;
    if (leader) {
      if (ok) mma_commit(ofull);
      mma_commit(fin);
    }
    __syncwarp();
  } else {
    const int quad = warp & 3, qu = (warp - 2) / 4;   // TMEM lane quadrant, 16-column quarter
    const int r = quad * 32 + lane;                    // key row = TMEM lane
    const int key = k0 + r;
    const int kmaxw = k0 + quad * 32 + 31;             // largest key of this warp
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const uint64_t SL2 = f2(scale * kL2e, scale * kL2e);
    // Only the causal mask is applied: queries >= S have -lse2 = -inf (P = 0) and D = 0, and rows of
    // keys >= S are never stored. Inner blocks alternate between the two groups (as in the dQ kernel).
    const int grp = (warp - 2) >> 3, half = ((warp - 2) >> 2) & 1;
    bool ok = true;
    for (int it = grp; it < nit; it += 2) {
      const int buf = it & 1, stage = it % NST;
      const uint32_t phase = (uint32_t)(it / NST) & 1u;
      if (!uwait(&sfull[buf], (uint32_t)(it >> 1) & 1u, abort_flag, err)) { ok = false; break; }
      fence_after();
      // this stage's statistics: its full phase has completed (the S MMA waited on it); the wait orders
      // the producer's stores before these loads
      if (!uwait(&full[stage], phase, abort_flag, err)) { ok = false; break; }
      for (int sub = 0; sub < 2; ++sub) {
        const int c0 = half * 32 + sub * 16;
        float sv[16], dp[16];
        tmem_ld16(trow + (uint32_t)(buf * 128 + c0), sv);
        tmem_ld16(trow + (uint32_t)(buf * 128 + IB + c0), dp);
        if (sub == 1) {
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sempty[buf]);
        }
        const float4* sl4 = reinterpret_cast<const float4*>(stats + stage * 2 * IB + c0);
        const float4* sd4 = reinterpret_cast<const float4*>(stats + stage * 2 * IB + IB + c0);
        float4 l[4], d[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) { l[u] = sl4[u]; d[u] = sd4[u]; }
        const int qbase = (i0 + it) * IB + c0;   // query of column 0 of these 16
        const bool diag = qbase < kmaxw;          // warp-uniform: some column may precede its key
        const int qlo = key - qbase;              // causal: columns e >= qlo
        uint32_t pk[8], dk[8];
#pragma unroll
        for (int e4 = 0; e4 < 4; ++e4) {
          const int e = 4 * e4;
          float2 xa = uf2(fma2(f2(sv[e], sv[e + 1]), SL2, f2(l[e4].x, l[e4].y)));
          float2 xb = uf2(fma2(f2(sv[e + 2], sv[e + 3]), SL2, f2(l[e4].z, l[e4].w)));
          if (diag) {
            if (e < qlo) xa.x = -INFINITY;
            if (e + 1 < qlo) xa.y = -INFINITY;
            if (e + 2 < qlo) xb.x = -INFINITY;
            if (e + 3 < qlo) xb.y = -INFINITY;
          }
          const float p0 = ex2(xa.x), p1 = ex2(xa.y), p2 = ex2(xb.x), p3 = ex2(xb.y);
          const float2 da = uf2(mul2(f2(p0, p1), sub2(f2(dp[e], dp[e + 1]), f2(d[e4].x, d[e4].y))));
          const float2 db = uf2(mul2(f2(p2, p3), sub2(f2(dp[e + 2], dp[e + 3]), f2(d[e4].z, d[e4].w))));
          pk[2 * e4] = pack2(p0, p1);
          pk[2 * e4 + 1] = pack2(p2, p3);
          dk[2 * e4] = pack2(da.x, da.y);
          dk[2 * e4 + 1] = pack2(db.x, db.y);
        }
        if (sub == 0 && !uwait(&pempty[buf], ((uint32_t)(it >> 1) & 1u) ^ 1u, abort_flag, err)) { ok = false; break; }
        put_row16(sp + buf * 2 * C_::OPB, c0 >> 4, r, pk);
        put_row16(sp + buf * 2 * C_::OPB + C_::OPB, c0 >> 4, r, dk);
      }
      if (!ok) break;
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pfull[buf]);
    }
    if (ok && uwait(ofull, 0, abort_flag, err)) {
      fence_after();
      const int kc = min(key, S - 1);
      const size_t NS = (size_t)gridDim.y * S;
#pragma unroll
      for (int c = qu * (HD / 4); c < (qu + 1) * (HD / 4); c += 16) {
        float gv[16], gk[16];
        tmem_ld16(trow + 256 + (uint32_t)c, gv);
        tmem_ld16(trow + 256 + HD + (uint32_t)c, gk);
        if (key < S) {
          if (part) {
            float* pk2 = part + ((size_t)h * NS + (size_t)b * S + kc) * HD + c;
            float* pv2 = pk2 + (size_t)H * NS * HD;
#pragma unroll
            for (int e = 0; e < 16; e += 4) {
              *reinterpret_cast<float4*>(pk2 + e) = make_float4(gk[e], gk[e + 1], gk[e + 2], gk[e + 3]);
              *reinterpret_cast<float4*>(pv2 + e) = make_float4(gv[e], gv[e + 1], gv[e + 2], gv[e + 3]);
            }
          } else {
            bf16* dkr = dqkv + ((size_t)b * S + kc) * ld + (size_t)xk + c;
            bf16* dvr = dqkv + ((size_t)b * S + kc) * ld + (size_t)xv + c;
#pragma unroll
            for (int e = 0; e < 16; ++e) gk[e] *= scale;
            Vec8<bf16>::store(dkr, gk);
            Vec8<bf16>::store(dkr + 8, gk + 8);
            Vec8<bf16>::store(dvr, gv);
            Vec8<bf16>::store(dvr + 8, gv + 8);
          }
        }
      }
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) tmem_release(fin, tmem);
}

// ----------------------------------------------------------------------------------------------
// Backward with 128-wide inner blocks (head dim 64): per 128 keys (dQ) or 128 queries (dK / dV), one
// round of hand-offs and 24 products instead of two rounds and 32. S / dP are single-buffered in TMEM
// (columns 0 and 128): the elementwise warps read them into registers in two 16-column passes and
// release them after the second, so the next block's products still overlap the arithmetic. Sixteen
// elementwise warps, four per lane quadrant, 32 columns each. A 128-row tile of Q / dO / K / V is one
// K-major [128 x 64] block per 64 head-dim columns (16 KB); as the MN-major B operand of the
// accumulating product its 16-row steps are 2 KB apart.
// ----------------------------------------------------------------------------------------------
constexpr int WB = 128;   // inner block rows

template <int HD>
struct WCfg {
  static constexpr int T128 = 128 * HD * 2;
  static constexpr int NST = 3;             // stages of (Q_i, dO_i) or (K_j, V_j), 128 rows each
  static constexpr int OPB = 128 * WB * 2;  // one bf16 [128 x 128] operand: two 64-column halves of 16 KB
  // K, V | stages | P^T, dS^T | statistics (-lse2, D) per stage | barriers | alignment
  static constexpr int SMEM_DKV = 2 * T128 + NST * 2 * T128 + 2 * OPB + NST * 2 * WB * 4 + 256 + 1024;
  // Q, dO | stages | dS | D quarters | barriers | alignment
  static constexpr int SMEM_DQ = 2 * T128 + NST * 2 * T128 + OPB + 4 * 128 * 4 + 256 + 1024;
  static_assert(SMEM_DKV <= 232448 && SMEM_DQ <= 232448, "shared memory per CTA");
};

// 16 bf16 values (columns 16 s .. 16 s + 15 of a thread's 32, qq the 32-column quarter) into row r of a
// swizzled [128 x 128] K-major operand (two 64-column halves of 16 KB).
__device__ __forceinline__ void put_row16w(uint8_t* g, int qq, int sub, int r, const uint32_t* pk) {
  uint8_t* row = g + (qq >> 1) * 16384 + r * 128;
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int chunk = ((qq & 1) * 4 + sub * 2 + u) ^ (r & 7);
    *reinterpret_cast<uint4*>(row + (chunk << 4)) = make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
  }
}

// dQ (and D) kernel, 128-key inner blocks. Maps: tq, tdo, tkv, all in 128-row boxes.
template <int HD>
__global__ void __launch_bounds__(NTHR_B, 1)
    attn_bwd_dq_w_k(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tdo,
                    const __grid_constant__ CUtensorMap tkv, const bf16* __restrict__ outp,
                    const bf16* __restrict__ dout, const float* __restrict__ lse, float* __restrict__ Dv,
                    bf16* __restrict__ dqkv, int S, int H, int Hkv, float scale, unsigned* err) {
  using C_ = WCfg<HD>;
  constexpr int NST = C_::NST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sq = smem;
  uint8_t* sdo = sq + C_::T128;
  uint8_t* sst = sdo + C_::T128;                  // stage s: K_j at s * 2 T128, V_j after it
  uint8_t* sds = sst + NST * 2 * C_::T128;        // dS
  float* dpart = (float*)(sds + C_::OPB);         // [4][128] quarters of D
  uint64_t* full = (uint64_t*)(dpart + 512);
  uint64_t* empty = full + NST;
  uint64_t* qfull = empty + NST;
  uint64_t* sfull = qfull + 1;
  uint64_t* sempty = sfull + 1;
  uint64_t* dsfull = sempty + 1;
  uint64_t* dsempty = dsfull + 1;
  uint64_t* ofull = dsempty + 1;
  uint64_t* fin = ofull + 1;
  uint32_t* tbase = (uint32_t*)(fin + 1);
  volatile int* abort_flag = (volatile int*)(tbase + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, b = blockIdx.y, qb = gridDim.z - 1 - blockIdx.z;   // longest first
  const int kvh = h / (H / Hkv);
  const int q0 = qb * 128;
  const int nkb = min(qb + 1, (S + WB - 1) / WB);
  const int ld = (H + 2 * Hkv) * HD, HDall = H * HD;
  const int xq = h * HD, xk = (H + kvh) * HD, xv = (H + Hkv + kvh) * HD;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    mbar_init(qfull, 1);
    mbar_init(sfull, 1);
    mbar_init(sempty, NEW);
    mbar_init(dsfull, NEW);
    mbar_init(dsempty, 1);
    mbar_init(ofull, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc512(tbase);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tbase;   // S: columns 0-127, dP: 128-255, dQ: 256 + HD
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    int issued[NST];
#pragma unroll
    for (int s = 0; s < NST; ++s) issued[s] = -1;
    const bool leader = elect_one();
    if (leader) {
      mbar_expect_tx(qfull, 2 * C_::T128);
#pragma unroll
      for (int c = 0; c < HD / 64; ++c) {
        tma3d(sq + c * 16384, &tq, qfull, xq + 64 * c, q0, b);
        tma3d(sdo + c * 16384, &tdo, qfull, h * HD + 64 * c, q0, b);
      }
    }
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      if (!uwait(&empty[stage], phase ^ 1u, abort_flag, err)) { ok = false; break; }
      issued[stage] = (int)phase;
      if (leader) {
        mbar_expect_tx(&full[stage], 2 * C_::T128);
        uint8_t* st = sst + stage * 2 * C_::T128;
#pragma unroll
        for (int c = 0; c < HD / 64; ++c) {
          tma3d(st + c * 16384, &tkv, &full[stage], xk + 64 * c, j * WB, b);
          tma3d(st + C_::T128 + c * 16384, &tkv, &full[stage], xv + 64 * c, j * WB, b);
        }
      }
      __syncwarp();
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (!ok && lane == 0) drain<NST>(full, issued, qfull);
  } else if (warp == 1) {
    constexpr uint32_t id_s = idesc_f16(128, WB, false, false);
    constexpr uint32_t id_q = idesc_f16(128, HD, false, true);
    const uint32_t q_addr = su32(sq), do_addr = su32(sdo), ds_addr = su32(sds);
    const bool leader = elect_one();   // issues every product and every commit that tracks them
    bool ok = uwait(qfull, 0, abort_flag, err);
    fence_after();
    int stage = 0, pstage = 0;
    uint32_t phase = 0;
    auto dq = [&](int jb, int st) -> bool {   // dQ += dS_jb K_jb
      if (!uwait(dsfull, (uint32_t)(jb & 1), abort_flag, err)) return false;
      fence_after();
      if (leader) {
        const uint32_t k_addr = su32(sst + st * 2 * C_::T128);
#pragma unroll
        for (int ks = 0; ks < WB / 16; ++ks)
          mma_bf16(tmem + 256, sdesc(ds_addr + (ks / 4) * 16384 + (ks % 4) * 32, 16, 1024),
                   sdesc(k_addr + ks * 2048, 16384, 1024), id_q, (jb > 0 || ks > 0) ? 1u : 0u);
        mma_commit(&empty[st]);
        mma_commit(dsempty);
      }
      __syncwarp();
      return true;
    };
    for (int j = 0; ok && j < nkb; ++j) {
      if (!uwait(sempty, ((uint32_t)j & 1u) ^ 1u, abort_flag, err) || !uwait(&full[stage], phase, abort_flag, err)) {
        ok = false;
        break;
      }
      fence_after();
      if (leader) {
        const uint32_t k_addr = su32(sst + stage * 2 * C_::T128), v_addr = k_addr + C_::T128;
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          const int kq = ks / 4, kr = ks % 4;
          mma_bf16(tmem, sdesc(q_addr + kq * 16384 + kr * 32, 16, 1024), sdesc(k_addr + kq * 16384 + kr * 32, 16, 1024),
                   id_s, ks > 0 ? 1u : 0u);
          mma_bf16(tmem + 128, sdesc(do_addr + kq * 16384 + kr * 32, 16, 1024),
                   sdesc(v_addr + kq * 16384 + kr * 32, 16, 1024), id_s, ks > 0 ? 1u : 0u);
        }
        mma_commit(sfull);
      }
      __syncwarp();
      if (j > 0 && !dq(j - 1, pstage)) { ok = false; break; }
      pstage = stage;
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (ok && !dq(nkb - 1, pstage)) ok = false;
    if (leader) {
      if (ok) mma_commit(ofull);
      mma_commit(fin);
    }
    __syncwarp();
  } else {
    const int quad = warp & 3, qq = (warp - 2) / 4;   // TMEM lane quadrant, 32-column quarter
    const int r = quad * 32 + lane;
    const int q = q0 + r, qc = min(q, S - 1);
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const size_t si = ((size_t)b * H + h) * S + qc;
    const float nlse2 = q < S ? -lse[si] * kL2e : -INFINITY;
    {   // D = rowsum(dO * O): each quarter sums a quarter of the row, fixed-order combination
      const bf16* orow = outp + ((size_t)b * S + qc) * HDall + (size_t)h * HD + qq * (HD / 4);
      const bf16* grow = dout + ((size_t)b * S + qc) * HDall + (size_t)h * HD + qq * (HD / 4);
      float acc = 0.f;
#pragma unroll
      for (int c = 0; c < HD / 4; c += 8) {
        float o8[8], g8[8];
        Vec8<bf16>::load(orow + c, o8);
        Vec8<bf16>::load(grow + c, g8);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc = fmaf(o8[e], g8[e], acc);
      }
      dpart[qq * 128 + r] = acc;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(32 * NEW) : "memory");
    const float Dq = (dpart[r] + dpart[128 + r]) + (dpart[256 + r] + dpart[384 + r]);
    if (q < S && qq == 0) Dv[si] = Dq;
    const uint64_t SL2 = f2(scale * kL2e, scale * kL2e), NL = f2(nlse2, nlse2), DD = f2(Dq, Dq);
    const int qmin = q0 + quad * 32;   // smallest query row of this warp
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      if (!uwait(sfull, (uint32_t)j & 1u, abort_flag, err)) { ok = false; break; }
      fence_after();
      for (int sub = 0; sub < 2; ++sub) {
        const int c0 = qq * 32 + sub * 16;
        float sv[16], dp[16];
        tmem_ld16(trow + (uint32_t)c0, sv);
        tmem_ld16(trow + 128u + (uint32_t)c0, dp);
        if (sub == 1) {
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(sempty);
        }
        const int kbase = j * WB + c0;
        const bool diag = kbase + 15 > qmin;   // warp-uniform: some column may lie above the diagonal
        const int kmax = q - kbase;            // causal: columns e <= kmax
        uint32_t pk[8];
#pragma unroll
        for (int e = 0; e < 16; e += 2) {
          float2 x = uf2(fma2(f2(sv[e], sv[e + 1]), SL2, NL));
          if (diag) {
            if (e > kmax) x.x = -INFINITY;
            if (e + 1 > kmax) x.y = -INFINITY;
          }
          const float p0 = ex2(x.x), p1 = ex2(x.y);
          const float2 ds = uf2(mul2(f2(p0, p1), sub2(f2(dp[e], dp[e + 1]), DD)));
          pk[e / 2] = pack2(ds.x, ds.y);
        }
        if (sub == 0 && !uwait(dsempty, ((uint32_t)j & 1u) ^ 1u, abort_flag, err)) { ok = false; break; }
        put_row16w(sds, qq, sub, r, pk);
      }
      if (!ok) break;
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(dsfull);
    }
    if (ok && uwait(ofull, 0, abort_flag, err)) {
      fence_after();
      bf16* drow = dqkv + ((size_t)b * S + qc) * ld + (size_t)h * HD;
#pragma unroll
      for (int c = qq * (HD / 4); c < (qq + 1) * (HD / 4); c += 16) {
        float v[16];
        tmem_ld16(trow + 256 + (uint32_t)c, v);
        if (q < S) {
#pragma unroll
          for (int e = 0; e < 16; ++e) v[e] *= scale;
          Vec8<bf16>::store(drow + c, v);
          Vec8<bf16>::store(drow + c + 8, v + 8);
        }
      }
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) tmem_release(fin, tmem);
}

// dK / dV kernel, 128-query inner blocks; grouped heads and outputs as attn_bwd_dkv_tg_k. Maps: tkv, tq,
// tdo, all in 128-row boxes.
template <int HD>
__global__ void __launch_bounds__(NTHR_B, 1)
    attn_bwd_dkv_w_k(const __grid_constant__ CUtensorMap tkv, const __grid_constant__ CUtensorMap tq,
                     const __grid_constant__ CUtensorMap tdo, const float* __restrict__ lse,
                     const float* __restrict__ Dv, bf16* __restrict__ dqkv, int S, int H, int Hkv, float scale,
                     float* __restrict__ part, unsigned* err) {
  using C_ = WCfg<HD>;
  constexpr int NST = C_::NST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sk = smem;
  uint8_t* sv = sk + C_::T128;
  uint8_t* sst = sv + C_::T128;                   // stage s: Q_i at s * 2 T128, dO_i after it
  uint8_t* sp = sst + NST * 2 * C_::T128;         // P^T
  uint8_t* sds = sp + C_::OPB;                    // dS^T
  float* stats = (float*)(sds + C_::OPB);         // stage s: -lse2[128], D[128]
  uint64_t* full = (uint64_t*)(stats + NST * 2 * WB);
  uint64_t* empty = full + NST;
  uint64_t* kvfull = empty + NST;
  uint64_t* sfull = kvfull + 1;
  uint64_t* sempty = sfull + 1;
  uint64_t* pfull = sempty + 1;
  uint64_t* pempty = pfull + 1;
  uint64_t* ofull = pempty + 1;
  uint64_t* fin = ofull + 1;
  uint32_t* tbase = (uint32_t*)(fin + 1);
  volatile int* abort_flag = (volatile int*)(tbase + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, b = blockIdx.y, kb = blockIdx.z;   // key block 0 (the longest) first
  const int kvh = part ? h / (H / Hkv) : h;
  const int k0 = kb * 128;
  const int nit = (S + WB - 1) / WB - kb;         // query blocks kb .. : the causal ones
  const int ld = (H + 2 * Hkv) * HD;
  const int xq = h * HD, xk = (H + kvh) * HD, xv = (H + Hkv + kvh) * HD;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) { mbar_init(&full[s], 2); mbar_init(&empty[s], 1); }
    mbar_init(kvfull, 1);
    mbar_init(sfull, 1);
    mbar_init(sempty, NEW);
    mbar_init(pfull, NEW);
    mbar_init(pempty, 1);
    mbar_init(ofull, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc512(tbase);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tbase;   // S^T 0-127, dP^T 128-255, dV 256 + HD, dK 256 + HD .. 256 + 2 HD
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    // one elected lane: TMA of K, V once and of (Q_i, dO_i) per block; every lane: four of the block's
    // -lse2 and D, loaded one block ahead
    int issued[NST];
#pragma unroll
    for (int s = 0; s < NST; ++s) issued[s] = -1;
    const bool leader = elect_one();
    if (leader) {
      mbar_expect_tx(kvfull, 2 * C_::T128);
#pragma unroll
      for (int c = 0; c < HD / 64; ++c) {
        tma3d(sk + c * 16384, &tkv, kvfull, xk + 64 * c, k0, b);
        tma3d(sv + c * 16384, &tkv, kvfull, xv + 64 * c, k0, b);
      }
    }
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    float nl[4], dd[4];
    auto fetch = [&](int it) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int qq2 = (kb + it) * WB + lane * 4 + u;
        const size_t si = ((size_t)b * H + h) * S + (qq2 < S ? qq2 : 0);
        nl[u] = qq2 < S ? -lse[si] * kL2e : -INFINITY;
        dd[u] = qq2 < S ? Dv[si] : 0.f;
      }
    };
    fetch(0);
    for (int it = 0; it < nit; ++it) {
      const int qi0 = (kb + it) * WB;
      if (!uwait(&empty[stage], phase ^ 1u, abort_flag, err)) { ok = false; break; }
      issued[stage] = (int)phase;
      if (leader) {
        mbar_expect_tx(&full[stage], 2 * C_::T128);
        uint8_t* st = sst + stage * 2 * C_::T128;
#pragma unroll
        for (int c = 0; c < HD / 64; ++c) {
          tma3d(st + c * 16384, &tq, &full[stage], xq + 64 * c, qi0, b);
          tma3d(st + C_::T128 + c * 16384, &tdo, &full[stage], h * HD + 64 * c, qi0, b);
        }
      }
      float* sl = stats + stage * 2 * WB;
      *reinterpret_cast<float4*>(sl + lane * 4) = make_float4(nl[0], nl[1], nl[2], nl[3]);
      *reinterpret_cast<float4*>(sl + WB + lane * 4) = make_float4(dd[0], dd[1], dd[2], dd[3]);
      __syncwarp();
      if (lane == 0) mbar_arrive(&full[stage]);
      if (it + 1 < nit) fetch(it + 1);
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (!ok && lane == 0) drain<NST>(full, issued, kvfull);
  } else if (warp == 1) {
    constexpr uint32_t id_s = idesc_f16(128, WB, false, false);
    constexpr uint32_t id_g = idesc_f16(128, HD, false, true);
    const uint32_t k_addr = su32(sk), v_addr = su32(sv), p_addr = su32(sp), ds_addr = su32(sds);
    const bool leader = elect_one();   // issues every product and every commit that tracks them
    bool ok = uwait(kvfull, 0, abort_flag, err);
    fence_after();
    int stage = 0, pstage = 0;
    uint32_t phase = 0;
    auto grads = [&](int ib, int st) -> bool {   // dV += P^T dO_ib, dK += dS^T Q_ib
      if (!uwait(pfull, (uint32_t)(ib & 1), abort_flag, err)) return false;
      fence_after();
      if (leader) {
        const uint32_t qa = su32(sst + st * 2 * C_::T128), da = qa + C_::T128;
#pragma unroll
        for (int ks = 0; ks < WB / 16; ++ks) {
          const uint32_t acc = (ib > 0 || ks > 0) ? 1u : 0u;
          const uint32_t ao = (ks / 4) * 16384 + (ks % 4) * 32;
          mma_bf16(tmem + 256, sdesc(p_addr + ao, 16, 1024), sdesc(da + ks * 2048, 16384, 1024), id_g, acc);
          mma_bf16(tmem + 256 + HD, sdesc(ds_addr + ao, 16, 1024), sdesc(qa + ks * 2048, 16384, 1024), id_g, acc);
        }
        mma_commit(&empty[st]);
        mma_commit(pempty);
      }
      __syncwarp();
      return true;
    };
    for (int it = 0; ok && it < nit; ++it) {
      if (!uwait(sempty, ((uint32_t)it & 1u) ^ 1u, abort_flag, err) || !uwait(&full[stage], phase, abort_flag, err)) {
        ok = false;
        break;
      }
      fence_after();
      if (leader) {
        const uint32_t qa = su32(sst + stage * 2 * C_::T128), da = qa + C_::T128;
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          const int kq = ks / 4, kr = ks % 4;
          mma_bf16(tmem, sdesc(k_addr + kq * 16384 + kr * 32, 16, 1024), sdesc(qa + kq * 16384 + kr * 32, 16, 1024),
                   id_s, ks > 0 ? 1u : 0u);
          mma_bf16(tmem + 128, sdesc(v_addr + kq * 16384 + kr * 32, 16, 1024),
                   sdesc(da + kq * 16384 + kr * 32, 16, 1024), id_s, ks > 0 ? 1u : 0u);
        }
        mma_commit(sfull);
      }
      __syncwarp();
      if (it > 0 && !grads(it - 1, pstage)) { ok = false; break; }
      pstage = stage;
      if (++stage == NST) { stage = 0; phase ^= 1u; }
    }
    if (ok && !grads(nit - 1, pstage)) ok = false;
    if (leader) {
      if (ok) mma_commit(ofull);
      mma_commit(fin);
    }
    __syncwarp();
  } else {
    const int quad = warp & 3, qq = (warp - 2) / 4;   // TMEM lane quadrant, 32-column quarter
    const int r = quad * 32 + lane;                    // key row = TMEM lane
    const int key = k0 + r;
    const int kmaxw = k0 + quad * 32 + 31;             // largest key of this warp
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const uint64_t SL2 = f2(scale * kL2e, scale * kL2e);
    // Only the causal mask is applied: queries >= S have -lse2 = -inf (P = 0) and D = 0, and rows of
    // keys >= S are never stored.
    bool ok = true;
    for (int it = 0; it < nit; ++it) {
      const int stage = it % NST;
      const uint32_t phase = (uint32_t)(it / NST) & 1u;
      if (!uwait(sfull, (uint32_t)it & 1u, abort_flag, err)) { ok = false; break; }
      fence_after();
      // this stage's statistics: its full phase has completed (the S MMA waited on it); the wait orders
      // the producer's stores before these loads
      if (!uwait(&full[stage], phase, abort_flag, err)) { ok = false; break; }
      for (int sub = 0; sub < 2; ++sub) {
        const int c0 = qq * 32 + sub * 16;
        float svv[16], dp[16];
        tmem_ld16(trow + (uint32_t)c0, svv);
        tmem_ld16(trow + 128u + (uint32_t)c0, dp);
        if (sub == 1) {
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(sempty);
        }
        const float4* sl4 = reinterpret_cast<const float4*>(stats + stage * 2 * WB + c0);
        const float4* sd4 = reinterpret_cast<const float4*>(stats + stage * 2 * WB + WB + c0);
        const int qbase = (kb + it) * WB + c0;   // query of column 0 of these 16
        const bool diag = qbase < kmaxw;          // warp-uniform: some column may precede its key
        const int qlo = key - qbase;              // causal: columns e >= qlo
        uint32_t pk[8], dk[8];
#pragma unroll
        for (int e4 = 0; e4 < 4; ++e4) {
          const float4 l = sl4[e4], d = sd4[e4];
          const int e = 4 * e4;
          float2 xa = uf2(fma2(f2(svv[e], svv[e + 1]), SL2, f2(l.x, l.y)));
          float2 xb = uf2(fma2(f2(svv[e + 2], svv[e + 3]), SL2, f2(l.z, l.w)));
          if (diag) {
            if (e < qlo) xa.x = -INFINITY;
            if (e + 1 < qlo) xa.y = -INFINITY;
            if (e + 2 < qlo) xb.x = -INFINITY;
            if (e + 3 < qlo) xb.y = -INFINITY;
          }
          const float p0 = ex2(xa.x), p1 = ex2(xa.y), p2 = ex2(xb.x), p3 = ex2(xb.y);
          const float2 da = uf2(mul2(f2(p0, p1), sub2(f2(dp[e], dp[e + 1]), f2(d.x, d.y))));
          const float2 db = uf2(mul2(f2(p2, p3), sub2(f2(dp[e + 2], dp[e + 3]), f2(d.z, d.w))));
          pk[2 * e4] = pack2(p0, p1);
          pk[2 * e4 + 1] = pack2(p2, p3);
          dk[2 * e4] = pack2(da.x, da.y);
          dk[2 * e4 + 1] = pack2(db.x, db.y);
        }
        if (sub == 0 && !uwait(pempty, ((uint32_t)it & 1u) ^ 1u, abort_flag, err)) { ok = false; break; }
        put_row16w(sp, qq, sub, r, pk);
        put_row16w(sds, qq, sub, r, dk);
      }
      if (!ok) break;
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(pfull);
    }
    if (ok && uwait(ofull, 0, abort_flag, err)) {
      fence_after();
      const int kc = min(key, S - 1);
      const size_t NS = (size_t)gridDim.y * S;
#pragma unroll
      for (int c = qq * (HD / 4); c < (qq + 1) * (HD / 4); c += 16) {
        float gv[16], gk[16];
        tmem_ld16(trow + 256 + (uint32_t)c, gv);
        tmem_ld16(trow + 256 + HD + (uint32_t)c, gk);
        if (key < S) {
          if (part) {
            float* pk2 = part + ((size_t)h * NS + (size_t)b * S + kc) * HD + c;
            float* pv2 = pk2 + (size_t)H * NS * HD;
#pragma unroll
            for (int e = 0; e < 16; e += 4) {
              *reinterpret_cast<float4*>(pk2 + e) = make_float4(gk[e], gk[e + 1], gk[e + 2], gk[e + 3]);
              *reinterpret_cast<float4*>(pv2 + e) = make_float4(gv[e], gv[e + 1], gv[e + 2], gv[e + 3]);
            }
          } else {
            bf16* dkr = dqkv + ((size_t)b * S + kc) * ld + (size_t)xk + c;
            bf16* dvr = dqkv + ((size_t)b * S + kc) * ld + (size_t)xv + c;
#pragma unroll
            for (int e = 0; e < 16; ++e) gk[e] *= scale;
            Vec8<bf16>::store(dkr, gk);
            Vec8<bf16>::store(dkr + 8, gk + 8);
            Vec8<bf16>::store(dvr, gv);
            Vec8<bf16>::store(dvr + 8, gv + 8);
          }
        }
      }
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) tmem_release(fin, tmem);
}

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;
int g_nsm = 0;

bool enc_init() {
  static int avail = -1;
  if (avail >= 0) return avail == 1;
  avail = 0;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  cudaDeviceGetAttribute(&g_nsm, cudaDevAttrMultiProcessorCount, dev);
  if (major != 10 || minor != 3 || g_nsm < 1) return false;
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
bool bwd_launch(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv, int B,
                int S, int H, int Hkv, cudaStream_t s, cudaMemPool_t pool, unsigned* err, float scale) {
  using C_ = BCfg<HD>;
  static bool attr = false;
  auto kq = attn_bwd_dq_tg_k<HD>;
  auto kkv = attn_bwd_dkv_tg_k<HD>;
  if (!attr) {
    if (cudaFuncSetAttribute(kq, cudaFuncAttributeMaxDynamicSharedMemorySize, C_::SMEM_DQ) != cudaSuccess ||
        cudaFuncSetAttribute(kkv, cudaFuncAttributeMaxDynamicSharedMemorySize, C_::SMEM_DKV) != cudaSuccess)
      return false;
    attr = true;
  }
  const int W = (H + 2 * Hkv) * HD, Wo = H * HD;
  CUtensorMap q128, q64, do128, do64;
  if (!qkv_map(&q128, qkv, B, S, W, 128) || !qkv_map(&q64, qkv, B, S, W, IB) || !qkv_map(&do128, dout, B, S, Wo, 128) ||
      !qkv_map(&do64, dout, B, S, Wo, IB))
    return false;
  float* part = nullptr;
  if (H > Hkv) {   // grouped heads: one CTA per query head, then a fixed-order group reduction
    const size_t bytes = 2ull * H * B * S * HD * sizeof(float);
    cudaError_t e = pool ? cudaMallocFromPoolAsync((void**)&part, bytes, pool, s) : cudaMallocAsync((void**)&part, bytes, s);
    if (e != cudaSuccess) { cudaGetLastError(); return false; }
  }
  const int nqb = (S + 127) / 128;
  cudaError_t e = launch_pdl(kq, dim3(H, B, nqb), NTHR_B, C_::SMEM_DQ, s, q128, do128, q64, (const bf16*)out,
                             (const bf16*)dout, lse, D, (bf16*)dqkv, S, H, Hkv, scale, err);
  if (e == cudaSuccess)
    e = launch_pdl(kkv, dim3(part ? H : Hkv, B, nqb), NTHR_B, C_::SMEM_DKV, s, q128, q64, do64, (const float*)lse,
                   (const float*)D, (bf16*)dqkv, S, H, Hkv, scale, part, err);
  if (part) {
    if (e == cudaSuccess) launch_reduce_dkv(part, dqkv, B * S, H, Hkv, HD, scale, s);
    cudaFreeAsync(part, s);
  }
  return e == cudaSuccess;
}

// The 128-wide backward (head dim 64).
template <int HD>
bool bwd_w_launch(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv, int B,
                  int S, int H, int Hkv, cudaStream_t s, cudaMemPool_t pool, unsigned* err, float scale) {
  using C_ = WCfg<HD>;
  static bool attr = false;
  auto kq = attn_bwd_dq_w_k<HD>;
  auto kkv = attn_bwd_dkv_w_k<HD>;
  if (!attr) {
    if (cudaFuncSetAttribute(kq, cudaFuncAttributeMaxDynamicSharedMemorySize, C_::SMEM_DQ) != cudaSuccess ||
        cudaFuncSetAttribute(kkv, cudaFuncAttributeMaxDynamicSharedMemorySize, C_::SMEM_DKV) != cudaSuccess)
      return false;
    attr = true;
  }
  const int W = (H + 2 * Hkv) * HD, Wo = H * HD;
  CUtensorMap q128, do128;
  if (!qkv_map(&q128, qkv, B, S, W, 128) || !qkv_map(&do128, dout, B, S, Wo, 128)) return false;
  float* part = nullptr;
  if (H > Hkv) {   // grouped heads: one CTA per query head, then a fixed-order group reduction
    const size_t bytes = 2ull * H * B * S * HD * sizeof(float);
    cudaError_t e = pool ? cudaMallocFromPoolAsync((void**)&part, bytes, pool, s) : cudaMallocAsync((void**)&part, bytes, s);
    if (e != cudaSuccess) { cudaGetLastError(); return false; }
  }
  const int nqb = (S + 127) / 128;
  cudaError_t e = launch_pdl(kq, dim3(H, B, nqb), NTHR_B, C_::SMEM_DQ, s, q128, do128, q128, (const bf16*)out,
                             (const bf16*)dout, lse, D, (bf16*)dqkv, S, H, Hkv, scale, err);
  if (e == cudaSuccess)
    e = launch_pdl(kkv, dim3(part ? H : Hkv, B, nqb), NTHR_B, C_::SMEM_DKV, s, q128, q128, do128, (const float*)lse,
                   (const float*)D, (bf16*)dqkv, S, H, Hkv, scale, part, err);
  if (part) {
    if (e == cudaSuccess) launch_reduce_dkv(part, dqkv, B * S, H, Hkv, HD, scale, s);
    cudaFreeAsync(part, s);
  }
  return e == cudaSuccess;
}

template <int HD>
bool fwd1_launch(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, cudaStream_t s, unsigned* err,
                 float scale) {
  using C_ = F1Cfg<HD>;
  static bool attr = false;
  auto kern = attn_fwd1_tg_k<HD>;
  if (!attr) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C_::SMEM) != cudaSuccess) return false;
    attr = true;
  }
  const int W = (H + 2 * Hkv) * HD;
  CUtensorMap tqk, tvv;
  if (!qkv_map(&tqk, qkv, B, S, W, 128) || !qkv_map(&tvv, qkv, B, S, W, 64)) return false;
  const long ntiles = (long)H * B * ((S + QB - 1) / QB);   // persistent: at most one CTA per SM
  const int grid = (int)std::min<long>(ntiles, g_nsm);
  return launch_pdl(kern, dim3(grid), NTHR, C_::SMEM, s, tqk, tvv, (bf16*)out, lse, S, B, H, Hkv, scale, err) ==
         cudaSuccess;
}

}  // namespace tg

// Returns false when the shape is outside this kernel (head dim 64 or 128, alignment, no sm_103a); the
// caller uses the mma.sync kernel then. scale: the softmax scale (1 / sqrt of the true head dim when the
// heads are zero-padded up to hd).
bool attn_fwd_tcgen05(const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd, cudaStream_t s,
                      unsigned* err, float scale) {
  if (hd != 64 && hd != 128) return false;
  if (((uintptr_t)qkv & 15u) || ((uintptr_t)out & 15u) || (long)B * H * ((S + tg::QB - 1) / tg::QB) > 0x7fffffffL)
    return false;
  if (!tg::enc_init()) return false;
  note_launch(1);
  return hd == 64 ? tg::fwd1_launch<64>(qkv, out, lse, B, S, H, Hkv, s, err, scale)
                  : tg::fwd1_launch<128>(qkv, out, lse, B, S, H, Hkv, s, err, scale);
}

// Returns false when the shape is outside these kernels (head dim 64 or 128, alignment, no sm_103a) or the
// grouped-head partials could not be allocated; the caller then uses the mma.sync kernels.
bool attn_bwd_tcgen05(const void* qkv, const void* out, const void* dout, const float* lse, float* D, void* dqkv,
                      int B, int S, int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool, unsigned* err,
                      float scale) {
  if (hd != 64 && hd != 128) return false;
  if ((((uintptr_t)qkv | (uintptr_t)out | (uintptr_t)dout | (uintptr_t)dqkv) & 15u) || B > 65535 ||
      (S + 127) / 128 > 65535)
    return false;
  if (!tg::enc_init()) return false;
  return hd == 64 ? tg::bwd_w_launch<64>(qkv, out, dout, lse, D, dqkv, B, S, H, Hkv, s, pool, err, scale)
                  : tg::bwd_launch<128>(qkv, out, dout, lse, D, dqkv, B, S, H, Hkv, s, pool, err, scale);
}

}  // namespace zl
