// Tensor-core GEMM for sm_103a: TMA tiles (128-byte swizzle) -> tcgen05.mma (bf16 operands,
// fp32 accumulator in TMEM, double buffered) -> tcgen05.ld epilogue (bias, residual, bf16 store,
// or fp32 accumulate into a gradient, or the fused AdamW step of the weight). Persistent,
// warp-specialised: warp 0 issues TMA loads, warp 1 owns TMEM and issues the MMAs (one thread),
// warps 2-5 (fused update: 4-11) drain the accumulator.
// Every mbarrier wait is bounded: on expiry the kernel raises ZL_DEVERR_TIMEOUT and unwinds.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>

#include "common.cuh"
#include "ops.h"
#include "tcgen05.cuh"

namespace zl {
namespace tc {

constexpr int BM = 128, BK = 64;
constexpr int kThreads = 192;      // TMA warp, MMA warp, four epilogue warps
// Fused-update kernels (mode 4): warpgroup 0 = TMA warp, MMA warp and two idle warps on kRegsLow
// registers each; then kUpdWarps epilogue warps (two per TMEM lane quadrant) on kRegsUpd, which hold the
// optimizer state of two chunks at once. The split uses exactly the registers of the launch (384 threads
// x 168, the most a 384-thread CTA gets); the host checks the kernel's register count before it runs.
// (40 for warpgroup 0 spills in the MMA loop; 56 + 224 spills nowhere.)
constexpr int kUpdWarps = 8;
constexpr int kThreadsUpd = 128 + 32 * kUpdWarps;
constexpr int kRegsLow = 56, kRegsUpd = 224;
static_assert(128 * kRegsLow + 32 * kUpdWarps * kRegsUpd <= kThreadsUpd * 168, "register split above the pool");

template <int BN, bool UPD = false>
struct Cfg {
  // BN = 64 stays under 114 KB of shared memory so two CTAs (and TMEM allocations) fit on an SM.
  static constexpr int STAGES = UPD ? (BN == 256 ? 4 : (kUpdWarps > 8 ? 5 : 6)) : (BN == 256 ? 4 : (BN == 128 ? 6 : 3));
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;
  // epilogue staging: per epilogue warp two buffers of 32 rows x 128 B (the TMA store box), or, in the
  // fused-update kernels, one 32 x 32 accumulator piece per epilogue warp
  static constexpr int OUT_BYTES = UPD ? kUpdWarps * 32 * 128 : 4 * 2 * 32 * 128;
  static constexpr int SMEM = STAGES * STAGE_BYTES + OUT_BYTES + 1024 + 256;
};

// Mode 4, one chunk: 16 rows x 32 columns of the tensor (rows row0 + 16 h .., columns col0 ..), whose
// accumulator piece is staged (fp32, 128-byte rows, 16-byte pieces XOR-swizzled by row) in `sp`. Lane l
// takes columns col0 + 4 (l % 8) .. + 3 of rows 16 h + l / 8 + 4 j, j = 0..3: every warp-wide load or
// store covers four whole 128-byte lines. upd_load issues the chunk's loads; upd_apply applies the AdamW
// step (adamw_elem) with G = gscale * acc to the loaded state and writes the fp32 master, both moments
// and the bf16 compute copy back. The state is streamed (evict-first): it is touched once, and L2 is
// kept for the operand tiles. With the blocked state layout (u.blk) the chunk is one 16 x 32 piece of
// it: lane l's row j sits at piece offset 4 l + 128 j, so each warp-wide access covers 512 contiguous
// bytes.
struct UpdRegs {
  float4 th[4], mm[4], vv[4];
  size_t at;     // state offset of row j = 0; row j sits 4 j rows further down (blocked: 128 j floats)
  size_t ct;     // row-major offset of row j = 0 (the compute copy)
  unsigned ok;   // bit j: row j is inside the tensor
};
__device__ __forceinline__ void upd_load(const GemmUpdate& u, UpdRegs& r, int row0, int h, int col0, int M, int N,
                                         bool valid, int lane) {
  r.ok = 0;
  const int col = col0 + 4 * (lane & 7);
  if (!valid || col >= N) return;
  const int row = row0 + 16 * h + (lane >> 3);
  r.ct = (size_t)row * N + col;
  r.at = u.blk ? blk_index((size_t)(row0 + 16 * h), (size_t)col0, (size_t)N) + 4 * lane : r.ct;
  const size_t sj = u.blk ? 128 : (size_t)4 * N;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (row + 4 * j < M) {
      const size_t a = r.at + j * sj;
      r.ok |= 1u << j;
      r.th[j] = __ldcs(reinterpret_cast<const float4*>(u.theta + a));
      r.mm[j] = __ldcs(reinterpret_cast<const float4*>(u.m + a));
      r.vv[j] = __ldcs(reinterpret_cast<const float4*>(u.v + a));
    }
  }
}
__device__ __forceinline__ void upd_apply(const GemmUpdate& u, const AdamHP& h, UpdRegs& r, const uint8_t* sp,
                                          int hh, int N, int lane) {
  const int piece = lane & 7;
  const size_t sj = u.blk ? 128 : (size_t)4 * N;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (!(r.ok >> j & 1u)) continue;
    const size_t a = r.at + j * sj;
    const int rr = 16 * hh + (lane >> 3) + 4 * j;
    const float4 a4 = *reinterpret_cast<const float4*>(sp + rr * 128 + ((piece ^ (rr & 7)) << 4));
    const float acc[4] = {a4.x, a4.y, a4.z, a4.w};
    float* tp = &r.th[j].x; float* mp = &r.mm[j].x; float* vp = &r.vv[j].x;
#pragma unroll
    for (int q = 0; q < 4; ++q) adamw_elem(tp[q], mp[q], vp[q], __fmul_rn(acc[q], u.gscale), h);
    __stcs(reinterpret_cast<float4*>(u.theta + a), r.th[j]);
    __stcs(reinterpret_cast<float4*>(u.m + a), r.mm[j]);
    __stcs(reinterpret_cast<float4*>(u.v + a), r.vv[j]);
    __nv_bfloat162 c2[2] = {__floats2bfloat162_rn(tp[0], tp[1]), __floats2bfloat162_rn(tp[2], tp[3])};
    __stcs(reinterpret_cast<uint2*>((bf16*)u.comp + r.ct + (size_t)(4 * j) * N), *reinterpret_cast<const uint2*>(c2));
  }
}

struct UpdMaps {   // (reserved: the fused update reads and writes its state directly)
  CUtensorMap unused;
};

struct Args {
  int M, N, K, mode;       // mode 0/1: bf16 C (+bias, +R); 2: fp32 C += acc; 3: fp32 store into split slice;
                           // 4: the AdamW step of the tensor in `u` with this tile as (the last part of) its gradient
  void* C;
  const float* bias;
  const bf16* R;
  unsigned* err;
  int tiles_m, tiles_n;
  int group_m;                // tile rows per raster group (tile_coords)
  int splits, kb_per_split;   // split-K: unit u -> split u / tiles, k blocks [s*kps, min(nk, (s+1)*kps))
  float alpha;                // scale of the product
  int rmode;                  // R in modes 0/1: 0 adds it (residual); 1 multiplies by GELU'(R) (R = the GELU input)
  GemmUpdate u;               // mode 4
  const float2* rope_cs;      // mode 0: rotate-half RoPE of columns < rope_cols (heads of rope_hd = 64 or 128),
  int rope_S, rope_hd, rope_cols;   // row n by position n % rope_S (NULL: none)
};

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, operand majors, N, M.
template <int BN, bool A_MN, bool B_MN>
__device__ __forceinline__ constexpr uint32_t idesc() {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((A_MN ? 1u : 0u) << 15) | ((B_MN ? 1u : 0u) << 16) |
         ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
}

// Tile order: groups of G tile rows sweep the tile columns, so the rows of A a group reads and the
// B tile a column of the group reads are each fetched from DRAM about once. The host picks G: all the
// tile rows when A fits well inside L2 or is the smaller operand (then every B tile is read once and A
// about once per wave), else 8.
__device__ __forceinline__ void tile_coords(int tile, int tiles_m, int tiles_n, int G, int& tm, int& tn) {
  const int per_group = G * tiles_n;
  const int gid = tile / per_group, first = gid * G;
  const int gm = min(tiles_m - first, G);
  const int r = tile % per_group;
  tm = first + r % gm;
  tn = r / gm;
}

// Tile (tm, tn) of work unit `unit`. PAIR: units are pairs of vertically adjacent tiles sharing their B
// tile; the CTA of cluster rank r takes the pair's tile row 2 tmp + r.
__device__ __forceinline__ void unit_tile(const Args& g, int unit, int num_tiles, bool pair, uint32_t crank, int& tm,
                                          int& tn) {
  tile_coords(unit % num_tiles, pair ? (g.tiles_m + 1) / 2 : g.tiles_m, g.tiles_n, g.group_m, tm, tn);
  if (pair) tm = 2 * tm + (int)crank;
}

// UPD: the fused optimizer epilogue (mode 4) is compiled in (a kernel of its own, so the other modes keep
// their register budget). PAIR: the CTA runs in a cluster of two that share each B tile: each loads half
// of it and multicasts it to both (TMA), each CTA's MMA commit frees the stage in both, so every SM copies
// half as much of B from L2 as alone.
template <int BN, bool A_MN, bool B_MN, bool UPD = false, bool PAIR = false>
__global__ void __launch_bounds__(UPD ? kThreadsUpd : kThreads, 1)
    gemm_tc_k(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
              const __grid_constant__ CUtensorMap tcm, const Args g, const __grid_constant__ UpdMaps um) {
  using C_ = Cfg<BN, UPD>;
  constexpr uint16_t kPairMask = 3;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* outbuf = smem + C_::STAGES * C_::STAGE_BYTES;   // 1024-byte aligned (stage sizes are)
  uint64_t* full = (uint64_t*)(outbuf + C_::OUT_BYTES);
  uint64_t* empty = full + C_::STAGES;
  uint64_t* tfull = empty + C_::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* fin = tempty + 2;
  uint32_t* tbase = (uint32_t*)(fin + 1);
  volatile int* abort_flag = (volatile int*)(tbase + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C_::STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], PAIR ? 2 : 1); }
    for (int a = 0; a < 2; ++a) { mbar_init(&tfull[a], 1); mbar_init(&tempty[a], UPD ? kUpdWarps : 4); }
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
  // a pair's copies land in both CTAs' shared memory: both sets of barriers exist before any is issued
  if (PAIR) cluster_sync();
  const uint32_t crank = PAIR ? cluster_rank() : 0u;
  const int unit0 = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int ustride = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  const uint32_t tmem = *tbase;
  // Programmatic dependent launch: the set-up above may overlap the previous kernel of the stream;
  // every thread waits for that kernel (and its memory) before touching global memory, and lets the
  // next GEMM of the stream begin its own set-up.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int nk = (g.K + BK - 1) / BK;
  const int num_tiles = (PAIR ? (g.tiles_m + 1) / 2 : g.tiles_m) * g.tiles_n;
  const int num_units = num_tiles * g.splits;

  if (warp < 2 || (UPD && warp < 4)) {
    // warpgroup 0 of a fused-update kernel hands most of its registers to the epilogue warpgroups
    if constexpr (UPD) regs_dec<kRegsLow>();
    if (warp == 0) {
      // ---------------- TMA producer ----------------
      // The whole warp runs the loop (uniform control flow keeps coordinates and addresses in uniform
      // registers); one elected lane issues the copies.
      const bool leader = elect_one();
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int issued[C_::STAGES];   // parity of the last fill of each stage, -1 if none
  #pragma unroll
      for (int s = 0; s < C_::STAGES; ++s) issued[s] = -1;
      for (int unit = unit0; ok && unit < num_units; unit += ustride) {
        int tm, tn;
        unit_tile(g, unit, num_tiles, PAIR, crank, tm, tn);
        const int kb0 = (unit / num_tiles) * g.kb_per_split, kb1 = min(nk, kb0 + g.kb_per_split);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!uwait(&empty[stage], phase ^ 1u, abort_flag, g.err)) { ok = false; break; }
          issued[stage] = (int)phase;
          if (leader) {
            mbar_expect_tx(&full[stage], C_::STAGE_BYTES);
            uint8_t* sa = smem + stage * C_::STAGE_BYTES;
            uint8_t* sb = sa + C_::A_BYTES;
            const int k0 = kb * BK;
            if (!A_MN) {
              tma2d(sa, &ta, &full[stage], k0, tm * BM);
            } else {
              tma2d(sa, &ta, &full[stage], tm * BM, k0);
              tma2d(sa + 8192, &ta, &full[stage], tm * BM + 64, k0);
            }
            if (PAIR) {   // this CTA's half of the B tile, into both CTAs
              constexpr int HB = BN / 2;
              if (!B_MN) {
                tma2d_mc(sb + crank * (HB * 128), &tb, &full[stage], k0, tn * BN + (int)crank * HB, kPairMask);
              } else {
  #pragma unroll
                for (int j = 0; j < HB / 64; ++j) {
                  const int jj = (int)crank * (HB / 64) + j;
                  tma2d_mc(sb + jj * 8192, &tb, &full[stage], tn * BN + 64 * jj, k0, kPairMask);
                }
              }
            } else if (!B_MN) {
              tma2d(sb, &tb, &full[stage], k0, tn * BN);
            } else {
  #pragma unroll
              for (int j = 0; j < BN / 64; ++j) tma2d(sb + j * 8192, &tb, &full[stage], tn * BN + 64 * j, k0);
            }
          }
          __syncwarp();
          if (++stage == C_::STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      if (PAIR && ok) {
        // both CTAs' commits for the last fill of every stage have arrived: no arrival from the peer (and no
        // copy of this CTA's into the peer) is still on its way when the CTAs exit
  #pragma unroll 1
        for (int s = 0; s < C_::STAGES; ++s)
          if (issued[s] >= 0 && !uwait(&empty[s], (uint32_t)issued[s], abort_flag, g.err)) break;
      }
      if (!ok && lane == 0) {   // unwinding: let the copies already in flight land before the CTA exits
        for (int s = 0; s < C_::STAGES; ++s) {
          if (issued[s] < 0) continue;
          const unsigned long long t0 = gtimer();
          while (!mbar_test(&full[s], (uint32_t)issued[s]) && gtimer() - t0 < 100000000ull) {
          }
        }
      }
    } else if (warp == 1) {
      // ---------------- MMA issuer ----------------
      // The whole warp runs the loop and the waits; one elected lane issues every product and every
      // commit that tracks them.
      constexpr uint32_t id = idesc<BN, A_MN, B_MN>();
      const bool leader = elect_one();
      int stage = 0, it = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int unit = unit0; ok && unit < num_units; unit += ustride, ++it) {
        const int acc = it & 1;
        const uint32_t aph = (uint32_t)(it >> 1) & 1u;
        if (!uwait(&tempty[acc], aph ^ 1u, abort_flag, g.err)) break;
        fence_after();
        const uint32_t d = tmem + (uint32_t)(acc * BN);
        const int kb0 = (unit / num_tiles) * g.kb_per_split, kb1 = min(nk, kb0 + g.kb_per_split);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!uwait(&full[stage], phase, abort_flag, g.err)) { ok = false; break; }
          fence_after();
          if (leader) {
            const uint32_t a0 = su32(smem + stage * C_::STAGE_BYTES), b0 = a0 + C_::A_BYTES;
  #pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              const uint64_t ad = A_MN ? sdesc(a0 + kk * 2048, 8192, 1024) : sdesc(a0 + kk * 32, 16, 1024);
              const uint64_t bd = B_MN ? sdesc(b0 + kk * 2048, 8192, 1024) : sdesc(b0 + kk * 32, 16, 1024);
              mma_bf16(d, ad, bd, id, (kb > kb0 || kk > 0) ? 1u : 0u);
            }
            if (PAIR) mma_commit_mc(&empty[stage], kPairMask);   // the stage is free in both CTAs' view
            else mma_commit(&empty[stage]);
          }
          __syncwarp();
          if (++stage == C_::STAGES) { stage = 0; phase ^= 1u; }
        }
        if (ok && leader) mma_commit(&tfull[acc]);
        __syncwarp();
      }
      // all MMAs issued by the leader complete before TMEM is released
      if (leader) mma_commit(fin);
      __syncwarp();
    }
  } else if constexpr (UPD) {
    // ---------------- fused optimizer epilogue (mode 4): warps 4 .. 4 + kUpdWarps - 1 ----------------
    regs_inc<kRegsUpd>();
    if (g.mode == 4) {
      // WQ warps per TMEM lane quadrant take interleaved 32-column pieces of the quadrant's 32 accumulator
      // rows (piece column 32 (part + WQ p)). Per piece a warp stages the accumulator in its shared-memory
      // buffer and works through the piece's two 16-row chunks (upd_load, then upd_apply).
      constexpr int WQ = kUpdWarps / 4;
      const int q = warp & 3, part = (warp - 4) >> 2;
      uint8_t* sbuf = outbuf + (warp - 4) * (32 * 128);
      const AdamHP hpv = adam_hp(g.u.hp, g.u.b1, g.u.b2, g.u.eps, g.u.wd);
      constexpr int NP = UPD ? BN / (32 * WQ) : 1;   // pieces per warp and tile
      static_assert(!UPD || NP >= 1, "at least one 32-column piece per epilogue warp");
      constexpr int NC = 2 * NP;    // 16-row chunks per warp and tile: chunk k = piece k / 2, half k % 2
      // L2 prefetch of chunk `k` of tile `unit` (lanes 0-15 one row each: its 128-byte line of the master
      // and of both moments), issued PD chunks ahead of the loads that read it
      auto prefetch_chunk = [&](int unit, int k) {
        if (unit >= num_units || lane >= 16) return;
        int tm, tn;
        unit_tile(g, unit, num_tiles, PAIR, crank, tm, tn);
        const int row = tm * BM + q * 32 + 16 * (k & 1) + lane, col = tn * BN + 32 * (part + WQ * (k >> 1));
        if (row >= g.M || col >= g.N) return;
        // blocked: line `lane` of the chunk's 2 KB piece; row-major: row `lane`'s 128-byte segment
        const size_t at = g.u.blk ? blk_index((size_t)(row - lane), (size_t)col, (size_t)g.N) + 32 * lane
                                  : (size_t)row * g.N + col;
        asm volatile("prefetch.global.L2 [%0];" ::"l"(g.u.theta + at));
        asm volatile("prefetch.global.L2 [%0];" ::"l"(g.u.m + at));
        asm volatile("prefetch.global.L2 [%0];" ::"l"(g.u.v + at));
      };
      constexpr int PD = 2;   // prefetch distance in chunks (2 and 3 measured alike, 4 slower)
  #pragma unroll
      for (int k = 0; k < PD; ++k) prefetch_chunk(unit0 + (k / NC) * ustride, k % NC);
      // chunk (p, h) of tile `unit`: rows 16 h .. of the quadrant, columns 32 (part + WQ p) ..
      auto load_chunk = [&](UpdRegs& r, int unit, int p, int h) {
        if (unit >= num_units) { r.ok = 0; return; }
        int tm, tn;
        unit_tile(g, unit, num_tiles, PAIR, crank, tm, tn);
        const int c = 32 * (part + WQ * p);
        upd_load(g.u, r, tm * BM + q * 32, h, tn * BN + c, g.M, g.N, c < BN, lane);
      };
      // The state loads of the next chunk are always in flight while a chunk is worked on (two register
      // sets), across pieces and into the CTA's next tile; each piece is read from TMEM when it is due and
      // TMEM goes back to the MMA warp after the tile's last piece is read.
      UpdRegs ra, rb;
      load_chunk(ra, unit0, 0, 0);
      int it = 0;
      for (int unit = unit0; unit < num_units; unit += ustride, ++it) {
        const int acc = it & 1;
        const uint32_t aph = (uint32_t)(it >> 1) & 1u;
        int ok = 1;
        if (lane == 0) ok = mbar_wait(&tfull[acc], aph, abort_flag, g.err) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        fence_after();
        const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
  #pragma unroll 1
        for (int p = 0; p < NP; ++p) {
          const int c = 32 * (part + WQ * p);
          float v[32];
          tmem_ld32(trow + (uint32_t)c, v);
          if (p == NP - 1) {
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
          }
          if (g.alpha != 1.f) {
  #pragma unroll
            for (int e = 0; e < 32; ++e) v[e] *= g.alpha;
          }
          __syncwarp();   // the previous piece's reads of the staging buffer are done
  #pragma unroll
          for (int k = 0; k < 8; ++k)
            *reinterpret_cast<float4*>(sbuf + lane * 128 + ((k ^ (lane & 7)) << 4)) =
                make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
          __syncwarp();
          prefetch_chunk(unit + ((2 * p + PD) / NC) * ustride, (2 * p + PD) % NC);
          load_chunk(rb, unit, p, 1);
          upd_apply(g.u, hpv, ra, sbuf, 0, g.N, lane);
          prefetch_chunk(unit + ((2 * p + 1 + PD) / NC) * ustride, (2 * p + 1 + PD) % NC);
          if (p + 1 < NP) load_chunk(ra, unit, p + 1, 0);
          else load_chunk(ra, unit + ustride, 0, 0);
          upd_apply(g.u, hpv, rb, sbuf, 1, g.N, lane);
        }
      }
    }
  } else {
    // ---------------- epilogue: warps 2..5, one accumulator row per thread ----------------
    // Per 128-byte column chunk (64 bf16 or 32 fp32 columns): TMEM -> registers (alpha, bias,
    // residual) -> this warp's staging buffer in the TMA 128-byte swizzle -> one TMA store (modes
    // 0, 1: bf16 C; 3: fp32 split slice) or TMA reduce-add (mode 2: fp32 C += tile) by lane 0.
    // The TMA clips rows >= M and columns >= N; two buffers per warp let a store drain while the
    // next chunk is formed.
    const int q = warp & 3;   // TMEM lanes 32q..32q+31 are the ones this warp may read
    uint8_t* stage_out = outbuf + q * (2 * 32 * 128);
    const bool f32out = g.mode >= 2;
    const int ccols = f32out ? 32 : 64;   // columns per chunk
    int it = 0, nchunk = 0, drain = 0;
    for (int unit = unit0; unit < num_units; unit += ustride, ++it) {
      int tm, tn;
      unit_tile(g, unit, num_tiles, PAIR, crank, tm, tn);
      const int split = unit / num_tiles;
      const int acc = it & 1;
      const uint32_t aph = (uint32_t)(it >> 1) & 1u;
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[acc], aph, abort_flag, g.err) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      fence_after();
      const int row0 = tm * BM + q * 32;
      const int m = row0 + lane;
      const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll 1
      for (int c = 0; c < BN; c += ccols, ++nchunk) {
        const int n0 = tn * BN + c;
        if constexpr (BN >= 128 && !A_MN && !B_MN) {   // mode 0 kernels of 128- or 256-column tiles
        if (g.rope_cs != nullptr && n0 < g.rope_cols) {
          // one query / key head (rope_hd columns: one or two 64-column chunks, both staging buffers):
          // pairs (i, i + hd/2) read from TMEM together, rounded to bf16, rotated, rounded again
          const int hd = g.rope_hd, half = hd >> 1, nch = hd >> 6;
          if (lane == 0) bulk_wait_read0();   // both buffers free
          __syncwarp();
          const float2* csr = g.rope_cs + (size_t)(m % g.rope_S) * half;
#pragma unroll 1
          for (int a = 0; a < half; a += 32) {
            float4 cs4[16];   // (cos, sin) of pairs a .. a + 31 (16-byte loads, issued before the TMEM reads)
#pragma unroll
            for (int e = 0; e < 16; ++e) cs4[e] = reinterpret_cast<const float4*>(csr + a)[e];
            float v1[32], v2[32];
            tmem_ld32(trow + (uint32_t)(c + a), v1);
            tmem_ld32(trow + (uint32_t)(c + a + half), v2);
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              float x1 = v1[e] * g.alpha, x2 = v2[e] * g.alpha;
              if (g.bias) {
                if (n0 + a + e < g.N) x1 += g.bias[n0 + a + e];
                if (n0 + a + half + e < g.N) x2 += g.bias[n0 + a + half + e];
              }
              x1 = __bfloat162float(__float2bfloat16_rn(x1));
              x2 = __bfloat162float(__float2bfloat16_rn(x2));
              const float4 c4 = cs4[e >> 1];
              rope_rot(x1, x2, (e & 1) ? c4.z : c4.x, (e & 1) ? c4.w : c4.y, v1[e], v2[e]);
            }
#pragma unroll
            for (int side = 0; side < 2; ++side) {
              const float* vv = side ? v2 : v1;
              const int col = a + side * half;   // column within the head
              uint8_t* srow = stage_out + (col >> 6) * (32 * 128) + lane * 128;
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                __nv_bfloat162 hv[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) hv[e] = __floats2bfloat162_rn(vv[8 * k + 2 * e], vv[8 * k + 2 * e + 1]);
                const int piece = ((col & 63) >> 3) + k;
                *reinterpret_cast<uint4*>(srow + ((piece ^ (lane & 7)) << 4)) = *reinterpret_cast<const uint4*>(hv);
              }
            }
          }
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
            for (int j = 0; j < nch; ++j) {
              if (row0 < g.M && n0 + 64 * j < g.N) tma_store2d(&tcm, stage_out + j * (32 * 128), n0 + 64 * j, row0);
              bulk_commit();
            }
          }
          drain = 1;
          c += hd - ccols;
          nchunk += nch - 1;
          continue;
        }
        }
        uint8_t* sbuf = stage_out + (nchunk & 1) * (32 * 128);
        if (lane == 0) {   // the store that last used this buffer has read it
          if (drain) bulk_wait_read0();
          else bulk_wait_read1();
        }
        drain = 0;
        __syncwarp();
        uint8_t* srow = sbuf + lane * 128;
        // 32 columns at a time: f32 chunks are one half, bf16 chunks two (16-byte pieces 4h .. 4h+3)
#pragma unroll 1
        for (int h = 0; h < ccols / 32; ++h) {
          const int nh = n0 + 32 * h;
          float v[32];
          tmem_ld32(trow + (uint32_t)(c + 32 * h), v);
          if (g.alpha != 1.f) {
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] *= g.alpha;
          }
          if (f32out) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const uint4 u = make_uint4(__float_as_uint(v[4 * k]), __float_as_uint(v[4 * k + 1]),
                                         __float_as_uint(v[4 * k + 2]), __float_as_uint(v[4 * k + 3]));
              *reinterpret_cast<uint4*>(srow + ((k ^ (lane & 7)) << 4)) = u;
            }
          } else {
            if (g.bias) {
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                if (nh + 4 * j < g.N) {
                  const float4 b4 = *reinterpret_cast<const float4*>(g.bias + nh + 4 * j);
                  v[4 * j] += b4.x; v[4 * j + 1] += b4.y; v[4 * j + 2] += b4.z; v[4 * j + 3] += b4.w;
                }
              }
            }
            if (g.R && m < g.M) {
              const bf16* rr = g.R + (size_t)m * g.N + nh;
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                if (nh + 8 * j < g.N) {
                  float r8[8];
                  Vec8<bf16>::load(rr + 8 * j, r8);
                  if (g.rmode) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) v[8 * j + e] *= gelu_tanh_grad(r8[e], true);
                  } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) v[8 * j + e] += r8[e];
                  }
                }
              }
            }
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              __nv_bfloat162 hv[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) hv[e] = __floats2bfloat162_rn(v[8 * k + 2 * e], v[8 * k + 2 * e + 1]);
              const int piece = 4 * h + k;
              *reinterpret_cast<uint4*>(srow + ((piece ^ (lane & 7)) << 4)) = *reinterpret_cast<const uint4*>(hv);
            }
          }
        }
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (row0 < g.M && n0 < g.N) {
            if (g.mode == 2) tma_reduce_add2d(&tcm, sbuf, n0, row0);
            else if (g.mode == 3) tma_store3d(&tcm, sbuf, n0, row0, split);
            else tma_store2d(&tcm, sbuf, n0, row0);
          }
          bulk_commit();
        }
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
    if (lane == 0) bulk_wait_all();   // every store of this warp has landed in global memory
  }

  __syncthreads();
  if (warp == 1) {
    // wait (bounded) for the final commit issued above, then release TMEM
    if (lane == 0) {
      const unsigned long long t0 = gtimer();
      while (!mbar_test(fin, 0) && gtimer() - t0 < 100000000ull) {
      }
    }
    __syncwarp();
  }
  if (PAIR) {   // neither CTA of a pair leaves while the other may still use its shared memory
    __syncthreads();
    cluster_sync();
  }
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)C_::TMEM_COLS)
                 : "memory");
  }
}

// Sums the split-K partials in split order (deterministic) and applies the epilogue (mode 4: the fused
// optimizer step of `u`, as update_row32 does it).
__global__ void splitk_reduce_k(const float* __restrict__ ws, int splits, int M, int N, int mode, void* C,
                                const float* __restrict__ bias, const bf16* R, float alpha, int rmode,
                                const GemmUpdate u) {
  pdl_wait();
  pdl_trigger();
  const size_t n8 = (size_t)M * N / 8, MN = (size_t)M * N;
  AdamHP hpv;
  if (mode == 4) hpv = adam_hp(u.hp, u.b1, u.b2, u.eps, u.wd);
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n8; i += (size_t)gridDim.x * blockDim.x) {
    const size_t e = i * 8;
    float acc[8];
    Vec8<float>::load(ws + e, acc);
    for (int s = 1; s < splits; ++s) {
      float t[8];
      Vec8<float>::load(ws + s * MN + e, t);
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] += t[q];
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] *= alpha;
    if (mode == 4) {
      float th[8], mm[8], vv[8], gg[8];
      const size_t se = u.blk ? blk_index(e / N, e % N, (size_t)N) : e;   // eight columns stay contiguous
      Vec8<float>::load(u.theta + se, th);
      Vec8<float>::load(u.m + se, mm);
      Vec8<float>::load(u.v + se, vv);
      if (u.g) Vec8<float>::load(u.g + e, gg);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float gsum = u.g ? __fadd_rn(gg[q], acc[q]) : acc[q];
        adamw_elem(th[q], mm[q], vv[q], __fmul_rn(gsum, u.gscale), hpv);
      }
      Vec8<float>::store(u.theta + se, th);
      Vec8<float>::store(u.m + se, mm);
      Vec8<float>::store(u.v + se, vv);
      if (u.comp) Vec8<bf16>::store((bf16*)u.comp + e, th);
      if (u.g) {
        const float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        Vec8<float>::store(u.g + e, z);
      }
    } else if (mode == 2) {
      float c[8];
      Vec8<float>::load((float*)C + e, c);
#pragma unroll
      for (int q = 0; q < 8; ++q) c[q] += acc[q];
      Vec8<float>::store((float*)C + e, c);
    } else {
      const int n = (int)(e % N);
      if (bias) {
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] += bias[n + q];
      }
      if (R) {
        float r[8];
        Vec8<bf16>::load(R + e, r);
        if (rmode) {
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[q] *= gelu_tanh_grad(r[q], true);
        } else {
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[q] += r[q];
        }
      }
      Vec8<bf16>::store((bf16*)C + e, acc);
    }
  }
}

// ------------------------------------------------------------------------------------------------
// host side
// ------------------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
int g_sms = 0;
int g_avail = -1;

bool init() {
  if (g_avail >= 0) return g_avail == 1;
  g_avail = 0;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
  if (major != 10 || minor != 3) return false;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || !fn)
    return false;
  g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  g_avail = 1;
  return true;
}

// 2-D bf16 tensor [outer, inner] (inner contiguous), box [box_outer, box_inner], 128-byte swizzle.
bool make_map(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer, uint32_t box_inner, uint32_t box_outer) {
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map of C for the epilogue's TMA stores: bf16 [M, N] in boxes of 32 rows x 64 columns (modes
// 0, 1), fp32 [M, N] in 32 x 32 (mode 2, reduce-add), fp32 [splits, M, N] in 1 x 32 x 32 (mode 3), all
// in the 128-byte swizzle the epilogue writes its staging buffers in.
bool make_map_c(CUtensorMap* m, const Args& a) {
  const bool f32 = a.mode >= 2;
  const uint64_t esz = f32 ? 4 : 2;
  cuuint64_t dims[3] = {(cuuint64_t)a.N, (cuuint64_t)a.M, (cuuint64_t)a.splits};
  cuuint64_t strides[2] = {(cuuint64_t)a.N * esz, (cuuint64_t)a.M * a.N * esz};
  cuuint32_t box[3] = {f32 ? 32u : 64u, 32u, 1u};
  cuuint32_t es[3] = {1, 1, 1};
  return g_encode(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.mode == 3 ? 3 : 2,
                  a.C, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, bool A_MN, bool B_MN, bool UPD = false, bool PAIR = false>
bool launch(const Args& a, const void* A, const void* B, cudaStream_t s, int ctas_per_sm) {
  using C_ = Cfg<BN, UPD>;
  static bool attr = false;
  static int max_pairs = 0;   // clusters of two that can be resident at once
  auto kern = gemm_tc_k<BN, A_MN, B_MN, UPD, PAIR>;
  if (!attr) {
    if (UPD) {   // the register split of the fused-update kernels must fit the pool the CTA is launched with
      cudaFuncAttributes fa;
      if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess ||
          128 * kRegsLow + 32 * kUpdWarps * kRegsUpd > kThreadsUpd * fa.numRegs) {
        cudaGetLastError();
        return false;
      }
    }
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C_::SMEM) != cudaSuccess) return false;
    if (PAIR) {
      cudaLaunchConfig_t oc = {};
      oc.gridDim = dim3(2u * (unsigned)g_sms);
      oc.blockDim = dim3((unsigned)(UPD ? kThreadsUpd : kThreads));
      oc.dynamicSmemBytes = C_::SMEM;
      cudaLaunchAttribute ca[1];
      ca[0].id = cudaLaunchAttributeClusterDimension;
      ca[0].val.clusterDim.x = 2;
      ca[0].val.clusterDim.y = 1;
      ca[0].val.clusterDim.z = 1;
      oc.attrs = ca;
      oc.numAttrs = 1;
      if (cudaOccupancyMaxActiveClusters(&max_pairs, kern, &oc) != cudaSuccess || max_pairs < 1) {
        cudaGetLastError();
        return false;
      }
    }
    attr = true;
  }
  CUtensorMap ta, tb;
  const bool okA = A_MN ? make_map(&ta, A, (uint64_t)a.M, (uint64_t)a.K, 64, 64)
                        : make_map(&ta, A, (uint64_t)a.K, (uint64_t)a.M, 64, BM);
  // a pair's CTA loads half of a K-major B tile (BN / 2 rows); MN-major B tiles are 64-column boxes
  const bool okB = B_MN ? make_map(&tb, B, (uint64_t)a.N, (uint64_t)a.K, 64, 64)
                        : make_map(&tb, B, (uint64_t)a.K, (uint64_t)a.N, 64, PAIR ? BN / 2 : BN);
  CUtensorMap tcm;
  if (!okA || !okB || !make_map_c(&tcm, a)) return false;
  UpdMaps um;
  std::memset(&um, 0, sizeof um);
  int grid;
  if (PAIR) {   // one cluster of two per pair of tile rows, as many as can be resident
    const int units = (a.tiles_m + 1) / 2 * a.tiles_n * a.splits;
    grid = 2 * std::min(units, max_pairs);
  } else {
    const int units = a.tiles_m * a.tiles_n * a.splits;
    const int slots = g_sms * ctas_per_sm;
    grid = units < slots ? units : slots;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3((unsigned)(UPD ? kThreadsUpd : kThreads));
  cfg.dynamicSmemBytes = C_::SMEM;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = 2;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = PAIR ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kern, ta, tb, tcm, a, um) == cudaSuccess;
}

template <bool A_MN, bool B_MN>
bool launch_bn(int bn, bool pair, const Args& a, const void* A, const void* B, cudaStream_t s) {
  if (bn == 256) return pair ? launch<256, A_MN, B_MN, false, true>(a, A, B, s, 1) : launch<256, A_MN, B_MN>(a, A, B, s, 1);
  if (bn == 128) return pair ? launch<128, A_MN, B_MN, false, true>(a, A, B, s, 1) : launch<128, A_MN, B_MN>(a, A, B, s, 1);
  return launch<64, A_MN, B_MN>(a, A, B, s, 2);
}

// The fused-update kernels (mode 4): 128 x 128 or 128 x 256 tiles, one CTA per SM.
bool launch_upd(int bn, bool pair, const Args& a, const void* A, const void* B, cudaStream_t s) {
  if (bn == 256)
    return pair ? launch<256, true, true, true, true>(a, A, B, s, 1) : launch<256, true, true, true>(a, A, B, s, 1);
  return pair ? launch<128, true, true, true, true>(a, A, B, s, 1) : launch<128, true, true, true>(a, A, B, s, 1);
}

// Tile width and split count from a wave model: units of 128 x BN x (K / splits) run on 152 (BN
// 256/128) or 304 (BN 64) slots, each k block (64 deep) of a unit taking the time measured for that
// tile on GB300 (4096^3 and transformer-shape sweeps; the operands of the mode-2 kernel are both
// MN-major and load in more boxes), plus, for splits, the fp32 partial traffic and the reduction.
void choose(int mode, int M, int N, int K, int& bn_out, int& splits_out, bool no64 = false) {
  const double hbm = 6.0e12;                  // bytes/s for the partials
  const int nk = (K + BK - 1) / BK;
  double best = 1e30;
  for (int bn : {256, 128, 64}) {
    if (no64 && bn == 64) continue;
    const double kb = mode == 2 ? (bn == 256 ? 0.40e-6 : bn == 128 ? 0.30e-6 : 0.36e-6)
                                : (bn == 256 ? 0.36e-6 : bn == 128 ? 0.29e-6 : 0.32e-6);
    const long tiles = (long)((M + BM - 1) / BM) * ((N + bn - 1) / bn);
    const int cps = bn == 64 ? 2 : 1;
    for (int sp : {1, 2, 3, 4, 6, 8}) {
      if (sp > 1 && nk / sp < 6) continue;
      const int kps = (nk + sp - 1) / sp;
      const long units = tiles * sp;
      const long slots = (long)g_sms * cps;
      const long waves = (units + slots - 1) / slots;
      double t = waves * kps * kb;
      if (sp > 1) t += (double)sp * M * N * 4.0 * 2.0 / hbm + 3e-6;
      if (t < best * 0.97) { best = t; bn_out = bn; splits_out = sp; }
    }
  }
}

}  // namespace tc

bool gemm_tc_available() { return tc::init(); }

namespace {

// Plans and launches one tensor-core GEMM (modes 0-2, or 4 with `u`); false if the shape or alignment
// is outside the kernel's rules.
bool run_tc(int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias, const void* R,
            unsigned* err, cudaStream_t s, cudaMemPool_t pool, float alpha, int rmode, const GemmUpdate* u,
            const GemmRope* rope = nullptr) {
  if (!tc::init()) return false;
  if (M < 16 || N < 16 || K < 16) return false;
  auto al16 = [](const void* p) { return ((uintptr_t)p & 15u) == 0; };
  if (!al16(A) || !al16(B) || !al16(C) || (R && !al16(R))) return false;
  // the fused update: 16-byte aligned state rows, a compute copy, no accumulated gradient
  if (u && (!al16(u->theta) || !al16(u->m) || !al16(u->v) || u->g || !u->comp || !al16(u->comp) || N % 8 != 0 ||
            (u->blk && (M % 16 != 0 || N % 32 != 0))))
    return false;
  if (N % 8 != 0) return false;
  // the rotation: bf16 C without residual, whole heads of 64 or 128 columns from column 0
  if (rope && (mode != 0 || R || !rope->cs || ((uintptr_t)rope->cs & 7u) || (rope->hd != 64 && rope->hd != 128) ||
               rope->S < 1 || rope->cols < 0 || rope->cols % rope->hd != 0 || rope->cols > N))
    return false;
  if ((mode == 0 || mode == 1) && K % 8 != 0) return false;
  if (mode >= 2 && M % 8 != 0) return false;
  int bn = 128, splits = 1;
  tc::choose(mode == 4 ? 2 : mode, M, N, K, bn, splits, mode == 4);
  // CTA pairs sharing B tiles wherever there are two tile rows to pair (BN 64 runs two CTAs per SM instead)
  int pair = bn >= 128 && M > tc::BM ? 1 : 0;
  if (const char* force = std::getenv("ZL_GEMM_TILE")) {   // test hook "BN:SPLITS[:PAIR]": forces the plan
    int fb = 0, fs = 0, fp = -1;
    const int nf = std::sscanf(force, "%d:%d:%d", &fb, &fs, &fp);
    if (nf >= 2 && (fb == 64 || fb == 128 || fb == 256) && fs >= 1 && fs <= 16) {
      bn = mode == 4 && fb == 64 ? 128 : fb;
      splits = std::max(1, std::min(fs, (K + tc::BK - 1) / tc::BK));
      pair = bn >= 128 && M > tc::BM ? 1 : 0;
      if (nf == 3 && (fp == 0 || fp == 1)) pair = fp && bn >= 128 ? 1 : 0;
    }
  }
  if (rope) {   // one split (the reduction does not rotate); tiles of 128 or 256 columns (heads never straddle)
    splits = 1;
    if (bn < 128) bn = 128;
    pair = bn >= 128 && M > tc::BM ? pair : 0;
  }
  tc::Args a;
  a.M = M; a.N = N; a.K = K; a.mode = mode;
  a.rope_cs = rope ? reinterpret_cast<const float2*>(rope->cs) : nullptr;
  a.rope_S = rope ? rope->S : 1;
  a.rope_hd = rope ? rope->hd : 0;
  a.rope_cols = rope ? rope->cols : 0;
  a.C = C; a.bias = bias; a.R = (const bf16*)R; a.err = err; a.alpha = alpha; a.rmode = rmode;
  a.u = u ? *u : GemmUpdate{};
  a.tiles_m = (M + tc::BM - 1) / tc::BM;
  a.tiles_n = (N + bn - 1) / bn;
  // one group of every tile row (each B tile fetched once, A once per wave of tile columns) when A fits
  // well inside L2 or is the smaller operand; else groups of 8 tile rows (A once, B once per group)
  const double a_bytes = (double)M * K * 2.0, b_bytes = (double)N * K * 2.0;
  a.group_m = (a_bytes <= 48e6 || a_bytes <= b_bytes) ? a.tiles_m : std::min(8, a.tiles_m);
  if (pair) a.group_m = (a.group_m + 1) / 2;   // in pairs of tile rows
  const int nk = (K + tc::BK - 1) / tc::BK;
  a.kb_per_split = (nk + splits - 1) / splits;
  a.splits = (nk + a.kb_per_split - 1) / a.kb_per_split;   // no empty split (its slice would never be formed)
  float* ws = nullptr;
  if (a.splits > 1) {
    const size_t bytes = (size_t)a.splits * M * N * 4;
    cudaError_t e = pool ? cudaMallocFromPoolAsync((void**)&ws, bytes, pool, s) : cudaMallocAsync((void**)&ws, bytes, s);
    if (e != cudaSuccess) {   // no room for the partials: one split
      cudaGetLastError();
      ws = nullptr;
      a.splits = 1;
      a.kb_per_split = nk;
    } else {
      a.mode = 3;
      a.C = ws;
      a.bias = nullptr;
      a.R = nullptr;
      a.alpha = 1.f;   // applied by the reduction
    }
  }
  note_launch(1);
  bool ok;
  if (mode == 0) ok = tc::launch_bn<false, false>(bn, pair, a, A, B, s);
  else if (mode == 1) ok = tc::launch_bn<false, true>(bn, pair, a, A, B, s);
  else if (a.mode == 4) ok = tc::launch_upd(bn, pair, a, A, B, s);
  else ok = tc::launch_bn<true, true>(bn, pair, a, A, B, s);
  if (ws) {
    if (ok) {
      note_launch(1);
      const size_t n8 = (size_t)M * N / 8;
      const int blocks = (int)std::min<size_t>((n8 + 255) / 256, (size_t)tc::g_sms * 8);
      launch_pdl(tc::splitk_reduce_k, blocks, 256, 0, s, ws, a.splits, M, N, mode, C, bias, (const bf16*)R, alpha,
                 rmode, a.u);
    }
    cudaFreeAsync(ws, s);
  }
  return ok;
}

}  // namespace

// Returns false when the shape / alignment is outside what the tensor-core path handles.
bool gemm_tc(int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias, const void* R,
             unsigned* err, cudaStream_t s, cudaMemPool_t pool, float alpha, int rmode) {
  return run_tc(mode, M, N, K, A, B, C, bias, R, err, s, pool, alpha, rmode, nullptr);
}

bool gemm_tc_update(int M, int N, int K, const void* A, const void* B, const GemmUpdate& u, unsigned* err,
                    cudaStream_t s, cudaMemPool_t pool, float alpha) {
  return run_tc(4, M, N, K, A, B, u.theta, nullptr, nullptr, err, s, pool, alpha, 0, &u);
}

bool gemm_tc_rope(int M, int N, int K, const void* A, const void* B, void* C, const float* bias, const GemmRope& r,
                  unsigned* err, cudaStream_t s, cudaMemPool_t pool) {
  return run_tc(0, M, N, K, A, B, C, bias, nullptr, err, s, pool, 1.f, 0, nullptr, &r);
}

}  // namespace zl
