// Host-side launchers of the engine's kernels (internal; the public ABI is include/zerolock.h).
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <string>

namespace zl {

enum Dt { F32 = 0, BF16 = 1 };
inline size_t dt_size(int dt) { return dt == BF16 ? 2 : 4; }

// Message returned by zl_last_error() on this thread.
void set_last_error(const char* msg);
inline void set_last_error(const std::string& msg) { set_last_error(msg.c_str()); }

// Count of kernels launched by the library (process-wide).
void note_launch(int n);
unsigned long long launches_so_far();

// h_0 = E[ids] (+ P[s]); bad ids set ZL_DEVERR_BAD_ID in *err and give a zero row.
void launch_embed(int dt, const int32_t* ids, const void* E, const void* P, void* h, int N, int S, int d,
                  int V, unsigned* err, cudaStream_t s);

// y = Norm(x) * g (+ b). RMSNorm (ln = false) or LayerNorm (ln = true). Saves rstd (and mean).
void launch_norm_fwd(int dt, bool ln, const void* x, const float* g, const float* b, void* y, float* rstd,
                     float* mean, int N, int d, float eps, cudaStream_t s);
// dx = Norm'(x)^T (g * dy) (+ dres). g may be NULL (gain 1).
void launch_norm_bwd_dx(int dt, bool ln, const void* x, const float* g, const float* rstd, const float* mean,
                        const void* dy, const void* dres, void* dx, int N, int d, cudaStream_t s);
// Column sums over rows, deterministic: per-row-block partials (part_*[b][c]), then the last block of
// each 256-column group adds sum_b part_*[b][c] into the outputs. Norm parameters: out_g += sum dy * xhat,
// out_b += sum dy (LN). counters: colsum_groups(d) device words, 0 before the launch and 0 again after
// it (one array per stream).
int colsum_blocks(int N);
int colsum_groups(int d);
void launch_norm_bwd_dparam(int dt, bool ln, const void* x, const float* rstd, const float* mean,
                            const void* dy, float* part_g, float* part_b, int N, int d, float* out_g, float* out_b,
                            unsigned* counters, cudaStream_t s);
// Bias gradients: out[c] += sum_r A[r][c].
void launch_colsum(int dt, const void* A, float* part, int N, int d, float* out, unsigned* counters, cudaStream_t s);
// out[c] += sum_b part[b][c], b in increasing order (deterministic).
void launch_partials_add(const float* part, int nb, int d, float* out, cudaStream_t s);

// Rotate q and k heads of qkv [N, (H + 2 Hkv) hd] in place by +angle (inverse = 0) or -angle.
// cs: [S, hd/2] (cos, sin) pairs.
void launch_rope(int dt, void* qkv, const float* cs, int N, int S, int H, int Hkv, int hd, int inverse,
                 cudaStream_t s);
// The same on the first nh heads of rows of ld elements.
void launch_rope_heads(int dt, void* qkv, const float* cs, int N, int S, int nh, int hd, int ld, int inverse,
                       cudaStream_t s);
void launch_swiglu_fwd(int dt, const void* gu, void* a, int N, int f, cudaStream_t s);
void launch_swiglu_bwd(int dt, const void* gu, const void* da, void* dgu, int N, int f, cudaStream_t s);
void launch_gelu_fwd(int dt, const void* x, void* y, size_t n, cudaStream_t s);
void launch_gelu_bwd(int dt, const void* x, const void* dy, void* dx, size_t n, cudaStream_t s);

// |Omega| = #(labels >= 0); labels outside [-1, V) set ZL_DEVERR_BAD_LABEL.
void launch_count_valid(const int32_t* labels, int N, int V, int* count, unsigned* err, cudaStream_t s);
// Fused local objective: dz and per-row loss (Eq. 3-5). t may be NULL iff alpha == 1. dz may be z.
void launch_local_loss(int dt, const void* z, const void* t, const int32_t* labels, int N, int V, int ldz,
                       float alpha, int kl_dir, const int* count, void* dz, float* row_loss, cudaStream_t s);
// *out = sum(row_loss) / count.
void launch_loss_reduce(const float* row_loss, int N, const int* count, float* out, cudaStream_t s);

// One AdamW step over a contiguous slab; zeroes g; refreshes the bf16 copy if comp != NULL. The step
// count t lives in device memory (advanced here by one); hp (3 floats) receives lr_t and the bias
// corrections; lr_t = lr0 or lr0 / sqrt(t - 1 + gamma) (schedule 1).
void launch_adamw(float* theta, float* g, float* m, float* v, void* comp, size_t n, long long* t, float* hp,
                  float lr0, int schedule, float gamma, float b1, float b2, float eps, float wd, float gscale,
                  cudaStream_t s);
// Advances the step count and writes hp = {lr_t, 1 - b1^t, 1 - b2^t} (the first kernel of launch_adamw).
void launch_adamw_tick(long long* t, float* hp, float lr0, int schedule, float gamma, float b1, float b2,
                       cudaStream_t s);
// AdamW over one contiguous span of n floats (a multiple of 4), hp already written for this step.
void launch_adamw_span(float* theta, float* g, float* m, float* v, void* comp, size_t n, const float* hp, float b1,
                       float b2, float eps, float wd, float gscale, cudaStream_t s);
// AdamW over `nranges` (offset, length) pairs of a slab (device array ranges[2 * nranges], lengths and
// offsets multiples of 4, the longest max_len), with hp already written for this step; zeroes g there.
void launch_adamw_ranges(float* theta, float* g, float* m, float* v, void* comp, const long long* ranges,
                         int nranges, size_t max_len, const float* hp, float b1, float b2, float eps, float wd,
                         float gscale, cudaStream_t s);
// AdamW over a matrix [M, N] (M % 16 == 0, N % 32 == 0) whose theta, m and v are in the blocked layout of
// blk_index while g (zeroed here) and comp are row-major; hp already written for this step.
void launch_adamw_span_blk(float* theta, float* g, float* m, float* v, void* comp, int M, int N, const float* hp,
                           float b1, float b2, float eps, float wd, float gscale, cudaStream_t s);
// Copies a matrix [M, N] (M % 16 == 0, N % 32 == 0) between row-major and the blocked layout of
// blk_index: to_blk = 1 reads src row-major and writes dst blocked, 0 the reverse.
void launch_blk_permute(const float* src, float* dst, int M, int N, int to_blk, cudaStream_t s);
void launch_f32_to_bf16(const float* src, void* dst, size_t n, cudaStream_t s);

// GEMM (row-major): mode 0: C = A[M,K] B[N,K]^T (+ bias[N]) (+ R[M,N]); mode 1: C = A[M,K] B[K,N] (+ R);
// mode 2: C[M,N] (fp32) += A[K,M]^T B[K,N]. bf16 runs on the tcgen05 kernel where its shape and
// alignment rules hold, everything else on the CUDA-core kernel. err: device word for timeouts;
// pool: stream-ordered pool for split-K partials (NULL: the device's default pool).
// alpha scales the product: C = alpha A op(B) (+ bias) (+ R), or C += alpha A^T B. R may alias C.
// rmode 1 (modes 0 and 1): C = alpha A op(B) * GELU'(R) instead of + R (R is the GELU input; bf16 uses
// the SFU tanh, as the GELU backward kernel does).
void gemm(int dt, int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias,
          const void* R, cudaStream_t s, unsigned* err = nullptr, cudaMemPool_t pool = nullptr, float alpha = 1.f,
          int rmode = 0);
// The optimizer step fused into a weight-gradient product (mode 2's C += alpha A^T B, here the last
// micro-batch of an update window): for the [M, N] tensor whose fp32 master, AdamW moments and bf16
// compute copy are theta, m, v and comp (comp may be NULL), the window's gradient is
// G = gscale * (g + alpha A^T B), g the accumulated gradient of the window's earlier micro-batches
// (NULL when there are none; zeroed here otherwise), and AdamW (hp as written by the step-count
// kernel) updates theta, m, v and comp in place; no gradient is stored. blk = 1: theta, m and v are in
// the blocked layout of blk_index (comp and g stay row-major).
struct GemmUpdate {
  float *theta, *m, *v, *g;
  void* comp;
  const float* hp;
  float b1, b2, eps, wd, gscale;
  int blk;
};
// bf16 operands on the tcgen05 kernel; false when the shape or alignment rules of mode 2 do not hold
// (the caller then forms the gradient with gemm() and applies the step with launch_adamw_ranges).
bool gemm_tc_update(int M, int N, int K, const void* A, const void* B, const GemmUpdate& u, unsigned* err,
                    cudaStream_t s, cudaMemPool_t pool, float alpha = 1.f);
// Rotate-half RoPE applied by the forward QKV product's epilogue: output columns < cols (the query and key
// heads, head dim hd = 64 or 128) of row n are rotated by the angles of position n % S, (cos, sin) pairs
// from cs [S][hd / 2][2] (fp32). The product is rounded to the output type before the rotation, as a
// separate RoPE pass over the stored product would see it.
struct GemmRope {
  const float* cs;
  int S, hd, cols;
};
// C = A B^T (+ bias) in bf16 with the rotation in the epilogue (mode 0, no residual); false when the
// tensor-core product or the rotation's rules do not hold (the caller then runs gemm() and launch_rope).
bool gemm_tc_rope(int M, int N, int K, const void* A, const void* B, void* C, const float* bias, const GemmRope& r,
                  unsigned* err, cudaStream_t s, cudaMemPool_t pool);
bool gemm_tc_available();
bool gemm_tc(int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias, const void* R,
             unsigned* err, cudaStream_t s, cudaMemPool_t pool, float alpha, int rmode = 0);
void gemm_simt(int dt, int mode, int M, int N, int K, const void* A, const void* B, void* C, const float* bias,
               const void* R, cudaStream_t s, float alpha = 1.f, int rmode = 0);

// Causal attention over qkv [N, (H + 2 Hkv) hd] (token-major, rows b*S + s): out [N, H hd], lse [B, H, S].
// bf16 with head dim 64 or 128: the one-pass tcgen05 kernel (err: device word for its bounded waits, may
// be NULL); other even bf16 head dims up to 128: the same kernel on copies zero-padded to 64 or 128 (pool:
// where the copies come from, NULL = the device's default pool), mma.sync if they cannot be had; fp32:
// CUDA cores.
void attn_fwd(int dt, const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd,
              cudaStream_t s, unsigned* err = nullptr, cudaMemPool_t pool = nullptr);
// Gradients into dqkv (same layout as qkv). Dbuf: [B, H, S] scratch. bf16 with head dim 64 or 128: the
// tcgen05 kernels (err as for attn_fwd); other even bf16 head dims up to 128: the tcgen05 kernels on
// zero-padded copies; else mma.sync; fp32: CUDA cores.
void attn_bwd(int dt, const void* qkv, const void* out, const void* dout, const float* lse, float* Dbuf,
              void* dqkv, int B, int S, int H, int Hkv, int hd, cudaStream_t s, cudaMemPool_t pool = nullptr,
              unsigned* err = nullptr);
// dK, dV of each KV head (bf16, into dqkv) = fixed-order sums over its query heads of the fp32 partials
// part[2][H][NS][hd] (dK unscaled; times scale here).
void launch_reduce_dkv(const float* part, void* dqkv, int NS, int H, int Hkv, int hd, float scale, cudaStream_t s);

}  // namespace zl
