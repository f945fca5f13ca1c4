/*
 * zerolock.h -- C ABI of the GB300 (sm_103a) engine for ZeroLock's decoupled per-chunk update.
 *
 * The method (paper Section II-A): a decoder-only transformer is cut into K
 * chunks of consecutive layers (Eq. 1: h_0 = E(x), h_k = f_k(h_{k-1})). Every
 * chunk reads its output through the model's frozen final norm and LM head
 * (Eq. 2: z_k = Norm(h_k) W_lm^T), builds the local objective
 *   L_k = alpha * CE(p_k, y) + (1 - alpha) * KL(p_k || sg(p_{k-1}))   (Eq. 3-5)
 * averaged over the loss set Omega (positions whose label is >= 0), back-
 * propagates inside the chunk only (Remark 1) and applies its own optimizer
 * step (Eq. 6, here AdamW as in Section III-C). Chunks exchange only hidden
 * states (Section III-A, technique III), so the K chunk updates run
 * concurrently: one CUDA stream per chunk, chunk k's output h_k handed to
 * chunk k+1 as soon as its forward ends (early forwarding, technique I).
 *
 * Conventions shared by every call:
 *   - Chunks are numbered k = 1..K as in the paper; h_0 is the embedding output.
 *   - Token-major activations: row n = b * S + s of a [N = B*S, d] row-major array.
 *   - Device arrays are in the context's compute dtype (ZL_DTYPE_F32: float,
 *     ZL_DTYPE_BF16: bfloat16) unless stated otherwise. ids and labels are
 *     int32 device arrays of B*S entries; a label of -1 marks a position
 *     outside Omega; ids must lie in [0, vocab), labels in [-1, vocab).
 *     A micro-batch holds 1 <= B*S <= 2^24 tokens, B <= 65535, S <= max_seq.
 *   - Pointers passed in are borrowed: the library never frees them, and
 *     device pointers given to a call must stay valid and unmodified until the
 *     next zl_synchronize() on that context returns (work is asynchronous).
 *   - Every call returns a zl_status. On failure zl_last_error() describes it;
 *     the context stays usable unless ZL_ERR_STATE is returned. No C++
 *     exception crosses this boundary.
 *   - A context is used by one host thread at a time.
 */
#ifndef ZEROLOCK_H
#define ZEROLOCK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct zl_ctx zl_ctx;

typedef enum {
  ZL_OK = 0,
  ZL_ERR_ARG = -1,          /* invalid argument (size, index, pointer, id or label range)      */
  ZL_ERR_CUDA = -2,         /* a CUDA runtime call failed                                      */
  ZL_ERR_OOM = -3,          /* device allocation failed                                        */
  ZL_ERR_STATE = -4,        /* the context is no longer usable (sticky CUDA error)              */
  ZL_ERR_TIMEOUT = -5,      /* zl_synchronize gave up waiting                                  */
  ZL_ERR_UNSUPPORTED = -6   /* valid but not implemented combination                           */
} zl_status;

/* Device-side error bits: kernels OR them into an error word, which zl_synchronize reports as
 * ZL_ERR_ARG (bad ids or labels) with a message naming each bit, and zl_wait_selftest returns. */
#define ZL_DEVERR_BAD_ID 1u      /* a token id outside [0, vocab)                   */
#define ZL_DEVERR_BAD_LABEL 2u   /* a label outside [-1, vocab)                     */
#define ZL_DEVERR_TIMEOUT 4u     /* a bounded wait inside a kernel gave up          */

enum { ZL_ARCH_LLAMA = 0, ZL_ARCH_GPT2 = 1 };
enum { ZL_DTYPE_F32 = 0, ZL_DTYPE_BF16 = 1 };

/* Model shape. arch ZL_ARCH_LLAMA: RMSNorm, rotate-half RoPE, grouped KV heads,
 * SwiGLU FFN (w1 = [W_gate; W_up]), untied LM head. ZL_ARCH_GPT2: LayerNorm with
 * bias, learned positions, GELU (tanh) MLP, biased linears, head tied to tok_emb.
 * d_model must equal n_heads * head_dim with head_dim even and <= 128. */
typedef struct {
  int arch;
  int dtype;                /* ZL_DTYPE_F32 or ZL_DTYPE_BF16 (fp32 master weights and AdamW state) */
  int n_layers, d_model, n_heads, n_kv_heads, d_ff, vocab, max_seq;
  float norm_eps, rope_theta;
} zl_model_dims;

/* Training settings of the local update (Eq. 3-6, step S3 of Section III-B). */
typedef struct {
  float alpha;              /* weight of the task term, 0 < alpha <= 1 (Eq. 3)                      */
  int kl_dir;               /* 0: KL(p_k || p_{k-1}) (Eq. 5);  1: KL(p_{k-1} || p_k)                  */
  int consis_first;         /* 1: chunk 1's consistency target is p_0 = readout(h_0); 0: alpha_1 = 1  */
  float lr, beta1, beta2, eps, weight_decay;     /* decoupled AdamW                                  */
  int accum_m;              /* micro-batches per update window (gradient = their mean), >= 1         */
  int max_live_chunks;      /* chunks whose activations may be alive at once; 0 means K              */
  int lr_schedule;          /* 0: constant lr;  1: lr / sqrt(t + lr_gamma), t = 0,1,.. (Theorem 1)    */
  float lr_gamma;
  int serialize;            /* 1: every chunk on one stream (no overlap; for measurement), 0: K streams */
  int lora_rank;            /* 0: full fine-tune; r > 0: LoRA (Section II-A) on the QKV, output and FFN  */
  float lora_scale;         /*   linears, w + lora_scale * B A, only A [r, in] and B [out, r] trainable  */
  int replay_depth;         /* D >= 0: zl_step keeps each chunk's last D inputs for zl_replay          */
  int adapter_dim;          /* 0: static readout head; r > 0 (a multiple of 16): chunk k's own readout  */
                            /*   goes through its adapter a_k(h) = h + GELU(h D_k^T) U_k^T (Section     */
                            /*   III-B, local update interface (b)), D_k [r, d], U_k [d, r] trainable   */
  int graph;                /* 1: zl_step / zl_bp_step are captured as a CUDA graph once per micro-batch */
                            /*   shape (after one eager call at that shape) and replayed; taken only    */
                            /*   with accum_m = 1, replay_depth = 0 and profiling off (else eager)      */
  int unfused_update;       /* 0: at a window's last micro-batch the weight-gradient products of the    */
                            /*   chunk's matrices apply AdamW in their epilogue (no gradient stored), the */
                            /*   other trainable tensors get AdamW after the backward; 1: one AdamW over */
                            /*   the whole slab after the backward. Same results either way.            */
  int loss_rows;            /* 0: each chunk's logits z_k (and the teacher's) exist for the whole       */
                            /*   micro-batch, z_{k-1} reused as chunk k's teacher; R > 0: the readout,   */
                            /*   local objective and head backward run over row slices of R rows (the    */
                            /*   head fused with the loss, Eq. 2-5): per slice z and the teacher's logits */
                            /*   (the frozen head on h_{k-1}, recomputed) are formed, the loss writes dz  */
                            /*   over z and dn = dz W_lm follows, so vocab-sized buffers hold R rows.    */
                            /*   Not with readout adapters (ZL_ERR_UNSUPPORTED).                         */
  int fuzz_delay_us;        /* scheduler fuzz (tests): > 0 sleeps the host a pseudo-random 0..this many  */
  unsigned fuzz_seed;       /*   microseconds (SplitMix64 stream of fuzz_seed) at every phase boundary of */
                            /*   an enqueue, so the GPU runs ahead in varying interleavings; 0 is off,   */
                            /*   at most 100000. Results do not depend on it.                           */
} zl_train_cfg;

/* Create a context: parameters, AdamW state, K streams and events, a stream-ordered
 * activation pool. bounds has K+1 entries, bounds[0] = 0 < bounds[1] < ... <
 * bounds[K] = n_layers; chunk k owns layers bounds[k-1] .. bounds[k]-1 (Eq. 1).
 * Parameters start at zero (norm gains at one); load them with zl_set_param.
 * *out is owned by the caller and released with zl_free. */
zl_status zl_create(const zl_model_dims* dims, int K, const int* bounds, const zl_train_cfg* cfg,
                    zl_ctx** out);

/* Release everything the context owns (waits for its queued work first). NULL-safe. */
void zl_free(zl_ctx* ctx);

/* Order the context's work after `stream` (a cudaStream_t; NULL = legacy default stream):
 * every call waits for the work queued on it so far. Results are joined back into it by
 * zl_join / zl_synchronize. */
zl_status zl_set_stream(zl_ctx* ctx, void* stream);

/* Tensor names: tok_emb [V,d], pos_emb [max_seq,d] (GPT-2), norm_f.weight [d],
 * norm_f.bias [d] (GPT-2), lm_head [V,d] (Llama), and per layer l
 * layers.{l}.{attn_norm.weight, attn_norm.bias, wqkv, bqkv, wo, bo, ffn_norm.weight,
 * ffn_norm.bias, w1, b1, w2, b2} (biases: GPT-2 only); weights are [out, in] row-major. With
 * lora_rank r > 0 also layers.{l}.{wqkv, wo, w1, w2}.{lora_a [r, in], lora_b [out, r]}. With
 * adapter_dim r > 0 also adapters.{k}.down [r, d] and adapters.{k}.up [d, r], k = 1..K (up starts
 * at zero: the adapter is the identity until it trains). The teacher p_{k-1} of chunk k stays the
 * frozen head on h_{k-1}; the backpropagation step and the global loss use no adapter.
 * zl_set_param copies `bytes` = numel * 4 of fp32 values from src (device memory if
 * on_device, else host) into the master copy (and the compute copy). */
zl_status zl_set_param(zl_ctx* ctx, const char* name, const void* src, size_t bytes, int on_device);

/* zl_load_weights: the same operation as zl_set_param under the name the problem statement's
 * interface uses (weights loaded once before training). Same arguments, ownership (src is only
 * read during the call) and errors (ZL_ERR_ARG for an unknown name or a byte count other than
 * numel * 4). */
zl_status zl_load_weights(zl_ctx* ctx, const char* name, const void* src, size_t bytes, int on_device);

/* Copy one tensor out as fp32 (waits for queued work). which: 0 value (master copy),
 * 1 accumulated gradient, 2 AdamW first moment, 3 AdamW second moment (1-3: trainable only). */
zl_status zl_get_param(zl_ctx* ctx, const char* name, int which, void* dst, size_t bytes, int on_device);

/* Number of elements of a named tensor (0 with ZL_ERR_ARG if unknown). */
zl_status zl_param_numel(zl_ctx* ctx, const char* name, size_t* numel);

/* h_0 = E(x) (Eq. 1): h0_out [B*S, d] (caller-owned device array, compute dtype). */
zl_status zl_embed(zl_ctx* ctx, const int32_t* ids, int B, int S, void* h0_out);

/* h_k = f_k(h_{k-1}) (Eq. 1) for one chunk, no gradient state touched. h_in: [B*S,d]
 * device array; may be NULL only for k = 1, in which case h_0 = E(ids) is formed
 * internally. h_out: caller-owned [B*S,d] device array. */
zl_status zl_forward_chunk(zl_ctx* ctx, int k, const void* h_in, const int32_t* ids, void* h_out,
                           int B, int S);

/* One local step of chunk k on one micro-batch (steps S1-S3 of Section III-B): forward,
 * readout, local objective with the teacher p_{k-1} = readout(h_in) (stop-gradient),
 * backward inside the chunk, gradient accumulation, AdamW at the end of the window.
 * h_in as in zl_forward_chunk. h_out (optional, may be NULL) receives h_k.
 * loss_out (optional host pointer): if non-NULL the call waits and stores L_k. */
zl_status zl_local_step(zl_ctx* ctx, int k, const void* h_in, const int32_t* ids,
                        const int32_t* labels, int B, int S, void* h_out, float* loss_out);

/* One micro-batch through all K chunks, concurrently (one stream per chunk, early
 * forwarding; chunk k's teacher is chunk k-1's logits). Same values as K calls of
 * zl_local_step in order k = 1..K. losses_out: NULL (losses stay on the device, see
 * zl_read_losses) or a host array of K floats, in which case the call waits. */
zl_status zl_step(zl_ctx* ctx, const int32_t* ids, const int32_t* labels, int B, int S,
                  float* losses_out);

/* Same-engine backpropagation baseline: the chunks chained, one readout on h_K,
 * CE over Omega, gradient through every chunk, AdamW on all (window rules as above). */
zl_status zl_bp_step(zl_ctx* ctx, const int32_t* ids, const int32_t* labels, int B, int S,
                     float* loss_out);

/* Failure recovery (Section III-B-3). Proactive checkpointing: zl_chunk_save writes chunk k's
 * state (fp32 master weights, gradient accumulator, AdamW moments, optimizer step, progress) into a
 * caller-owned host buffer of zl_chunk_state_bytes bytes; zl_chunk_load restores it (ZL_ERR_ARG if
 * the blob belongs to another chunk or shape). Reactive recovery: with replay_depth D > 0, zl_step
 * keeps each chunk's inputs h_{k-1} and labels of the last D micro-batches in a device ring (the
 * paper's hidden-state buffer); zl_replay re-runs chunk k's local steps for every buffered
 * micro-batch after its restored progress, catching it up to the pipeline frontier while the other
 * chunks keep their state. *replayed (optional) gets the count, *loss_out (optional) the last L_k.
 * ZL_ERR_ARG if a needed micro-batch has left the ring. */
zl_status zl_chunk_state_bytes(zl_ctx* ctx, int k, size_t* bytes);
zl_status zl_chunk_save(zl_ctx* ctx, int k, void* host_dst, size_t bytes);
zl_status zl_chunk_load(zl_ctx* ctx, int k, const void* host_src, size_t bytes);
zl_status zl_replay(zl_ctx* ctx, int k, int* replayed, float* loss_out);

/* Global objective L(p_K) = CE of the last chunk's readout over Omega (Section II-C). */
zl_status zl_eval_global_loss(zl_ctx* ctx, const int32_t* ids, const int32_t* labels, int B, int S,
                              float* loss_out);

/* Wait for the last zl_step / zl_bp_step and copy its K (or 1) losses to host. */
zl_status zl_read_losses(zl_ctx* ctx, float* losses_out, int n);

/* Make the stream given to zl_set_stream wait for all queued work (no host wait). */
zl_status zl_join(zl_ctx* ctx);

/* Wait for all queued work, polling; ZL_ERR_TIMEOUT after timeout_ms (< 0: no limit).
 * Also reports device-side argument errors (ids or labels out of range) of that work. */
zl_status zl_synchronize(zl_ctx* ctx, int timeout_ms);

/* Device bytes held by the context: peak since creation or the last reset, and now
 * (parameters and optimizer state plus the activation pool's high-water mark). */
zl_status zl_peak_bytes(zl_ctx* ctx, size_t* peak, size_t* current);
zl_status zl_reset_peak(zl_ctx* ctx);

/* Message of the last failed call on this thread (owned by the library). */
const char* zl_last_error(void);

/* Instrumentation. zl_profile(ctx, 1) brackets every kernel the context launches with CUDA
 * events on the launching stream; zl_profile_read waits for queued work and writes a JSON
 * object {class: {"launches", "ms", "flops", "bytes"}} (algorithmic FLOPs / HBM bytes of those
 * launches) into buf (NUL-terminated, truncated to cap), then clears the records.
 * zl_kernel_launches returns how many kernels the library has launched in this process. */
zl_status zl_profile(zl_ctx* ctx, int on);
zl_status zl_profile_read(zl_ctx* ctx, char* buf, size_t cap);
zl_status zl_kernel_launches(uint64_t* count);

/* ---------------------------------------------------------------------------------------
 * Single-kernel entry points (used by the tests and the roofline measurement). All
 * pointers are device pointers; `stream` is a cudaStream_t (NULL = legacy default).
 * ------------------------------------------------------------------------------------- */

/* Fused local objective (Eq. 3-5) over N rows of logits. z, t: [N, ldz] in `dtype`
 * (columns >= V are padding and ignored); t may be NULL when alpha == 1.
 * labels: [N] int32; 1 <= N <= 2^24 (|Omega| is counted exactly up to 2^24 rows, so larger N is
 * rejected with ZL_ERR_ARG). Writes dz = dL/dz [N, ldz] (dtype; padding columns 0) and
 * row_loss[N] (fp32, alpha*CE_i + (1-alpha)*KL_i, 0 outside Omega), and *loss
 * (one fp32 on the device) = sum(row_loss) / |Omega|. A label outside [-1, V) is treated as
 * -1 (the row leaves Omega); this call does not report it, since reporting would need a
 * synchronisation (the engine's step calls do report it, through zl_synchronize). */
zl_status zl_op_local_loss(int dtype, const void* z, const void* t, const int32_t* labels, int N,
                           int V, int ldz, float alpha, int kl_dir, void* dz, float* row_loss,
                           float* loss, void* stream);

/* The frozen head fused with the local objective (Eq. 2-5), over row slices: for rows i of n [N, d]
 * (the final norm of h_k) and tn [N, d] (of h_{k-1}; NULL when alpha == 1), z = n W^T and t = tn W^T
 * with W [ldw, d] the head (rows V.. ldw - 1 are padding and must be zero), the loss of
 * zl_op_local_loss, and dn = dL/dn = dz W [N, d] (dtype; may alias n). Logits exist for
 * rows_per_slice rows at a time only (1 <= rows_per_slice; the slice buffers and |Omega| come from the
 * stream-ordered default pool of the device). row_loss [N] and *loss (device, fp32) as for
 * zl_op_local_loss. ldw >= V, ldw % 8 == 0, d % 8 == 0; 1 <= N <= 2^24. */
zl_status zl_op_head_loss(int dtype, const void* n, const void* tn, const void* W, const int32_t* labels, int N,
                          int d, int V, int ldw, float alpha, int kl_dir, int rows_per_slice, void* dn,
                          float* row_loss, float* loss, void* stream);

/* Causal softmax attention with grouped KV heads (the attention of every transformer layer of
 * Eq. 1): qkv [B*S, (H + 2*Hkv)*hd] token-major (per row: H query heads, Hkv key heads, Hkv value
 * heads, each hd wide; query head h reads KV head h / (H/Hkv)), scale 1/sqrt(hd). Forward writes
 * out [B*S, H*hd] and lse [B, H, S] (fp32 natural-log row log-sum-exp). Backward takes dout
 * [B*S, H*hd] and writes dqkv (qkv layout). dtype of qkv/out/dout/dqkv; hd even and <= 128. */
zl_status zl_op_attention(int dtype, const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd,
                          void* stream);
zl_status zl_op_attention_bwd(int dtype, const void* qkv, const void* out, const void* dout, const float* lse,
                              void* dqkv, int B, int S, int H, int Hkv, int hd, void* stream);

/* Allocation-free variant of zl_op_local_loss (no counterpart in the paper). For callers that
 * cannot allocate device memory: a host framework whose own caching allocator has reserved the
 * device budget, so an outside cudaMalloc fails or breaks its accounting, or a latency-critical
 * loop that must not take the synchronisation cudaMalloc / cudaFree can imply. Same inputs and
 * outputs as zl_op_local_loss except that the per-row losses stay internal (out-of-range labels
 * leave Omega without being reported, as there); the scratch (per-row losses, |Omega|, a word the
 * label check writes) is a file-scope device array of
 * ZL_NOALLOC_MAX_ROWS + 128 floats (257 KB) that every GPU which loads the library holds until
 * process exit. N > ZL_NOALLOC_MAX_ROWS is rejected with ZL_ERR_ARG. The first call in each CUDA
 * context looks up the array's device address (cudaGetSymbolAddress, with that device current);
 * make that first call before any stream capture. All calls share the array: calls whose work
 * overlaps on the GPU race on it, so order them on one stream (or synchronise between them).
 * Calls no cudaMalloc, cudaFree or allocating library routine. */
#define ZL_NOALLOC_MAX_ROWS 65536
zl_status zl_op_local_loss_noalloc(int dtype, const void* z, const void* t, const int32_t* labels, int N, int V,
                                   int ldz, float alpha, int kl_dir, void* dz, float* loss, void* stream);

/* C[M,N] (+)= A[M,K] . B^T where B is [N,K] (mode 0, "forward"), or A[M,K] . B with B
 * [K,N] (mode 1, "dX"), or C[M,N] += A^T . B with A [K,M], B [K,N] (mode 2, "dW",
 * C fp32 and always accumulated). dtype of A, B and (modes 0/1) C. Row-major, dense. */
zl_status zl_op_gemm(int dtype, int mode, int M, int N, int K, const void* A, const void* B, void* C,
                     void* stream);

/* zl_op_gemm with the fused epilogues the chunk forward and backward use. Modes 0 and 1:
 * C = A op(B) (+ bias[N], fp32, read) (+ R[M,N]) when r_mode == 0, or C = A op(B) * GELU'(R) when
 * r_mode == 1 (R the input of the tanh-form GELU, so C is the gradient at that input). bias and R
 * may be NULL (R is required for r_mode 1); R has the dtype and layout of C and may alias it.
 * Mode 2 (dW): C += A^T B and, if bias is not NULL, bias[M] += the column sums of A[K,M] (the bias
 * gradient that goes with the weight gradient, by the engine's column-sum kernel); R must be NULL
 * and r_mode 0 (else ZL_ERR_ARG). */
zl_status zl_op_gemm_ex(int dtype, int mode, int M, int N, int K, const void* A, const void* B, void* C,
                        float* bias, const void* R, int r_mode, void* stream);

/* The query / key / value projection of a Llama-style layer with rotate-half RoPE (the first
 * product and rotation of the chunk function f_k, Eq. 1): C[M,N] = A[M,K] . B^T (+ bias[N], fp32), B [N,K], then in
 * every row n the columns < rot_cols, whole heads of hd columns, rotated pairwise (column i with
 * i + hd/2 of the head) by the angles of position n % S: cs is the device table [S][hd/2][2] of
 * (cos, sin), fp32, read only. dtype of A, B, C; row-major, dense; C must not overlap A or B.
 * bf16 products of head dim 64 or 128 on the tensor-core path rotate in the product's epilogue
 * (one kernel; the product is rounded to bf16 before its rotation, exactly as the two-pass
 * path sees it), other cases run the product and then a RoPE pass. Returns ZL_ERR_ARG for NULL
 * pointers or rot_cols that is not a multiple of hd within N, ZL_ERR_CUDA on a launch failure. */
zl_status zl_op_qkv_rope(int dtype, int M, int N, int K, const void* A, const void* B, void* C, const float* bias,
                         const float* cs, int S, int hd, int rot_cols, void* stream);

/* Self-test of the bounded waits (no counterpart in the paper; failure detection without a GPU
 * fault). Every wait of the tcgen05 kernels on an mbarrier (a TMA copy landing, a product completing,
 * a tile drained) gives up after about 2 s of SM clock (longer at lower clocks), ORs
 * ZL_DEVERR_TIMEOUT into the error word and unwinds the kernel, so a lost arrival ends as an error
 * status instead of a hung GPU. This call runs that same wait on an mbarrier that nothing ever
 * arrives at (one CTA, its own stream), waits for the kernel, and writes the kernel's error bits to
 * *bits_out (host): ZL_DEVERR_TIMEOUT when the wait gave up as designed. It takes the wait's full
 * limit (seconds). Returns ZL_OK with the bits written, or ZL_ERR_CUDA / ZL_ERR_STATE if the launch
 * or the synchronisation failed. The device and any context on it stay usable afterwards. */
zl_status zl_wait_selftest(unsigned* bits_out);

#ifdef __cplusplus
}
#endif
#endif /* ZEROLOCK_H */
