// ZeroLock engine behind the C ABI of include/zerolock.h: parameter slabs, the chunk forward /
// local backward (Section II-A, Remark 1), the readout and local objective (Eq. 2-5), AdamW
// (Eq. 6 as AdamW), and the K-stream scheduler with early forwarding, per-entry readiness
// events and a bound on live activation arenas (Section III-A/B).
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <atomic>
#include <cstdio>
#include <chrono>
#include <cmath>
#include <cstring>
#include <string>
#include <thread>
#include <vector>

#include "common.cuh"
#include "ops.h"
#include "zerolock.h"

namespace zl {
static std::atomic<unsigned long long> g_launches{0};
void note_launch(int n) { g_launches.fetch_add((unsigned long long)n, std::memory_order_relaxed); }
unsigned long long launches_so_far() { return g_launches.load(std::memory_order_relaxed); }
}  // namespace zl

namespace {

using namespace zl;

// Kernel classes of the per-launch profile (zl_profile).
enum { PC_GEMM, PC_GEMM_HEAD, PC_GEMM_UPD, PC_ATTN_F, PC_ATTN_B, PC_LOSS, PC_NORM, PC_ADAMW, PC_ELEM, PC_COUNT };
const char* kPCName[PC_COUNT] = {"gemm_layer", "gemm_head", "gemm_update", "attn_fwd", "attn_bwd", "local_loss",
                                 "norm", "adamw", "elementwise"};
struct ProfRec {
  int cls;
  cudaEvent_t a, b;
  double flops, bytes, launches;
};

thread_local std::string g_err;

struct ZlError {
  zl_status st;
  std::string msg;
};
[[noreturn]] void raise_err(zl_status st, const std::string& msg) { throw ZlError{st, msg}; }

bool sticky(cudaError_t e) {
  return e == cudaErrorIllegalAddress || e == cudaErrorLaunchFailure || e == cudaErrorIllegalInstruction ||
         e == cudaErrorMisalignedAddress || e == cudaErrorHardwareStackError || e == cudaErrorAssert ||
         e == cudaErrorInvalidPc || e == cudaErrorInvalidAddressSpace;
}

#define CK(call)                                                                                  \
  do {                                                                                            \
    cudaError_t e_ = (call);                                                                      \
    if (e_ != cudaSuccess) {                                                                      \
      raise_err(e_ == cudaErrorMemoryAllocation ? ZL_ERR_OOM : (sticky(e_) ? ZL_ERR_STATE : ZL_ERR_CUDA), \
                std::string(#call) + " failed: " + cudaGetErrorString(e_));                       \
    }                                                                                             \
  } while (0)

#define CHECK_LAUNCH() CK(cudaGetLastError())

// ----------------------------------------------------------------------------------------------
// Parameter layout: per layer a fixed list of tensors, stored in one contiguous slab per chunk
// (fp32 master, gradient, AdamW m and v; plus a bf16 compute copy in bf16 mode).
// ----------------------------------------------------------------------------------------------
enum PK { P_N1W, P_N1B, P_WQKV, P_BQKV, P_WO, P_BO, P_N2W, P_N2B, P_W1, P_B1, P_W2, P_B2, P_COUNT };
const char* kPName[P_COUNT] = {"attn_norm.weight", "attn_norm.bias", "wqkv", "bqkv", "wo", "bo",
                               "ffn_norm.weight", "ffn_norm.bias", "w1", "b1", "w2", "b2"};

// Where a tensor lives: the trainable slab (fp32 master, grad, AdamW m/v, compute copy), the frozen
// fp32 vector slab, or the frozen matrix slab (compute dtype only).
enum Slab { S_TRAIN = 0, S_FVEC = 1, S_FMAT = 2 };
constexpr int kLoraP[4] = {P_WQKV, P_WO, P_W1, P_W2};   // the linears that carry LoRA factors

struct Layer {
  size_t off[P_COUNT];
  size_t numel[P_COUNT];
  bool has[P_COUNT];
  int slab[P_COUNT];
  size_t la[4], lb[4];        // LoRA A [r16, in] and B^T [r16, out] offsets in the trainable slab
  int lin_in[4], lin_out[4];  // shapes of the four linears
  bool blk[P_COUNT];          // trainable matrix whose master and moments are in the blocked layout
  int rows[P_COUNT], cols[P_COUNT];   // [rows, cols] of each matrix (out, in)
};

struct Chunk {
  int k = 0, l0 = 0, l1 = 0;
  size_t n = 0;
  float *master = nullptr, *grad = nullptr, *m = nullptr, *v = nullptr;
  void* comp = nullptr;
  float* fvec = nullptr;   // frozen vectors (norm gains, biases) in LoRA mode
  void* fmat = nullptr;    // frozen base matrices in LoRA mode (compute dtype)
  size_t fvec_n = 0, fmat_n = 0;
  std::vector<Layer> layers;
  size_t ad_down = 0, ad_up = 0;   // readout adapter D [r, d] and U [d, r] in the trainable slab
  size_t ad_end = 0;               // end of the adapter (= ad_down without one): vectors before, matrices after
  size_t grad_n = 0;               // floats of the gradient accumulator (n, or ad_end with the fused update)
  int micro = 0;
  long t = 0;                // optimizer steps (host mirror of *d_t)
  long long* d_t = nullptr;  // optimizer steps on the device, advanced by the AdamW launch
  float* d_hp = nullptr;     // this step's lr and bias corrections (written on the device)
  long done = 0;             // micro-batches this chunk has processed (progress metadata)
  // Fused update: at a window's last micro-batch the weight-gradient products of the chunk's matrices
  // apply the optimizer step in their epilogue; the other trainable ranges (norm gains, biases, readout
  // adapter) get a range update after the backward.
  bool fuse = false;          // this micro-batch's backward updates the matrices in place
  long long* d_ranges = nullptr;   // device (offset, length) pairs of the non-matrix trainable ranges
  std::vector<long long> h_ranges; // the same on the host
  int n_ranges = 0, n_ranges_layers = 0;   // all of them / those before the readout adapter
  size_t max_range = 0;
  // hidden-state buffer (Section III-B-3): the last replay_depth inputs h_{k-1} with their labels
  struct Entry {
    long seq = -1;
    int B = 0, S = 0;
    size_t cap = 0;          // tokens the buffers hold
    void* h = nullptr;
    int32_t* labels = nullptr;
  };
  std::vector<Entry> ring;
  cudaStream_t s = nullptr;
  cudaEvent_t ev_h = nullptr, ev_z = nullptr, ev_loss = nullptr, ev_hb = nullptr, ev_done = nullptr;
  // side stream of the backward's column sums (the chunk stream itself when serialised) and its events
  cudaStream_t side = nullptr;
  cudaEvent_t ev_sin = nullptr, ev_ln2 = nullptr, ev_layer = nullptr, ev_ln1 = nullptr, ev_send = nullptr;
};

// Saved activations of one layer (pointers into the chunk's arena).
struct LayerSave {
  const void* x = nullptr;   // layer input
  void *xn1, *qkv, *att, *x2, *xn2, *hid, *act, *y;
  float *rstd1, *mean1, *rstd2, *mean2, *lse;
  void* u[4];                // LoRA: x A^T of each linear [N, r]
};

}  // namespace

struct zl_ctx {
  zl_model_dims dims;
  zl_train_cfg cfg;
  int K = 0;
  std::vector<int> bounds;
  int dt = 0;
  bool llama = true;
  int d = 0, hd = 0, H = 0, Hkv = 0, qkvw = 0, ad = 0, f = 0, f1 = 0, V = 0, Vp = 0;
  std::vector<Chunk> ch;   // ch[1..K]
  void *tok_emb = nullptr, *pos_emb = nullptr, *lm_head = nullptr;
  float *normf_w = nullptr, *normf_b = nullptr;
  float* rope_cs = nullptr;
  cudaMemPool_t pool = nullptr;
  size_t static_bytes = 0;
  cudaStream_t user = nullptr, aux = nullptr;
  cudaEvent_t ev_start = nullptr, ev_aux = nullptr, ev_sync = nullptr;
  std::vector<cudaEvent_t> live_ring;
  long live_seq = 0;
  unsigned* d_err = nullptr;
  int* d_count = nullptr;        // [K + 1] one |Omega| per stream
  float* d_losses = nullptr;     // [K + 1]
  float* h_losses = nullptr;     // pinned [K + 1]
  int last_nloss = 0;
  long seq = 0;              // micro-batches seen by zl_step (the pipeline frontier)
  bool broken = false;
  std::vector<void*> statics;
  bool prof = false;
  std::vector<ProfRec> recs;
  std::vector<cudaEvent_t> evpool;
  size_t evnext = 0;
  // CUDA-graph form of zl_step / zl_bp_step: one capture per micro-batch shape, then replays
  struct StepGraph {
    int B = 0, S = 0;
    int seen = 0;                 // calls at this shape so far (the first runs eagerly)
    cudaGraphExec_t exec = nullptr;
    int32_t *ids = nullptr, *labels = nullptr;   // staging copies of the inputs the graph reads
    size_t cap = 0;
    unsigned long long launches = 0;             // kernel launches the captured step contains
  } zg, bg;
  bool capturing = false;
  cudaStream_t cap = nullptr;   // capture origin (the user's stream may be the uncapturable legacy stream)
  uint64_t fuzz_state = 0;      // scheduler fuzz stream (cfg.fuzz_seed)
};

namespace {

// ----------------------------------------------------------------------------------------------
// small helpers
// ----------------------------------------------------------------------------------------------
size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

void* salloc(zl_ctx* c, size_t bytes) {
  void* p = nullptr;
  CK(cudaMalloc(&p, std::max<size_t>(bytes, 256)));
  c->statics.push_back(p);
  c->static_bytes += std::max<size_t>(bytes, 256);
  return p;
}

void* palloc(zl_ctx* c, size_t bytes, cudaStream_t s) {
  void* p = nullptr;
  CK(cudaMallocFromPoolAsync(&p, std::max<size_t>(bytes, 256), c->pool, s));
  return p;
}
void pfree(void* p, cudaStream_t s) {
  if (p) CK(cudaFreeAsync(p, s));
}

// A bump allocator over one pool allocation (256-byte aligned pieces).
struct Arena {
  char* base = nullptr;
  size_t used = 0, cap = 0;
  void* take(size_t bytes) {
    void* p = base + used;
    used += round_up(std::max<size_t>(bytes, 1), 256);
    if (used > cap) raise_err(ZL_ERR_STATE, "internal: arena overflow");
    return p;
  }
};

const void* Wc(zl_ctx* c, Chunk& k, int li, PK p) {   // compute-dtype pointer of a matrix
  const Layer& L = k.layers[li];
  const size_t off = L.off[p];
  if (L.slab[p] == S_FMAT)
    return c->dt == BF16 ? (const void*)((const bf16*)k.fmat + off) : (const void*)((const float*)k.fmat + off);
  return c->dt == BF16 ? (const void*)((const bf16*)k.comp + off) : (const void*)(k.master + off);
}
float* Wm(Chunk& k, int li, PK p) {   // fp32 pointer of a vector (gain or bias)
  const Layer& L = k.layers[li];
  if (!L.has[p]) return nullptr;
  return L.slab[p] == S_FVEC ? k.fvec + L.off[p] : k.master + L.off[p];
}
bool trainable(Chunk& k, int li, PK p) {
  const Layer& L = k.layers[li];
  return L.has[p] && L.slab[p] == S_TRAIN;
}
float* Gm(Chunk& k, int li, PK p) {   // gradient accumulator; NULL for frozen tensors and unstored gradients
  const Layer& L = k.layers[li];
  return (trainable(k, li, p) && L.off[p] < k.grad_n) ? k.grad + L.off[p] : nullptr;
}
int lora_r16(int r) { return r > 0 ? (r + 15) / 16 * 16 : 0; }

const void* TrainC(zl_ctx* c, Chunk& k, size_t off) {
  return c->dt == BF16 ? (const void*)((const bf16*)k.comp + off) : (const void*)(k.master + off);
}

size_t esz(zl_ctx* c) { return dt_size(c->dt); }

// Scheduler fuzz (cfg.fuzz_delay_us > 0): the host sleeps a pseudo-random 0..fuzz_delay_us microseconds,
// drawn from a SplitMix64 stream seeded by cfg.fuzz_seed, so the GPU runs ahead of the enqueues in
// varying interleavings. Only the timing changes; every dependency is an event or stream order.
void fuzz_pause(zl_ctx* c) {
  if (c->cfg.fuzz_delay_us <= 0) return;
  uint64_t z = (c->fuzz_state += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  z ^= z >> 31;
  std::this_thread::sleep_for(std::chrono::microseconds(z % (uint64_t)(c->cfg.fuzz_delay_us + 1)));
}

// Consecutive host-side NVTX ranges over the phases a call enqueues, named by chunk and phase, so a
// profiler can select one chunk's or one phase's kernels (ncu --nvtx --nvtx-include "zl chunk 2 loss/").
// Without an attached tool each range is a cheap no-op. Each phase boundary is also a fuzz point.
class NvtxPhases {
 public:
  explicit NvtxPhases(zl_ctx* c) : c_(c) {}
  ~NvtxPhases() { end(); }
  void next(const char* fmt, int k = 0) {
    end();
    fuzz_pause(c_);
    char name[64];
    std::snprintf(name, sizeof name, fmt, k);
    nvtxRangePushA(name);
    open_ = true;
  }
  void end() {
    if (open_) nvtxRangePop();
    open_ = false;
  }

 private:
  zl_ctx* c_;
  bool open_ = false;
};

void wait_ev(cudaStream_t s, cudaEvent_t e) { CK(cudaStreamWaitEvent(s, e, 0)); }
void rec(cudaEvent_t e, cudaStream_t s) { CK(cudaEventRecord(e, s)); }

cudaEvent_t take_ev(zl_ctx* c) {
  if (c->evnext == c->evpool.size()) {
    cudaEvent_t e;
    CK(cudaEventCreate(&e));
    c->evpool.push_back(e);
  }
  return c->evpool[c->evnext++];
}

// Brackets the launches of its scope with timing events when the context profiles.
struct ProfScope {
  zl_ctx* c;
  cudaStream_t s;
  int cls;
  double flops, bytes, launches;
  cudaEvent_t a = nullptr;
  bool keep = true;   // false: nothing of the scope ran, no record
  ProfScope(zl_ctx* c_, cudaStream_t s_, int cls_, double fl, double by, double nl = 1)
      : c(c_), s(s_), cls(cls_), flops(fl), bytes(by), launches(nl) {
    if (c && c->prof) {
      a = take_ev(c);
      CK(cudaEventRecord(a, s));
    }
  }
  ~ProfScope() {
    if (!a || !keep) return;
    if (c->evnext == c->evpool.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return;
      c->evpool.push_back(e);
    }
    cudaEvent_t b = c->evpool[c->evnext++];
    cudaEventRecord(b, s);
    c->recs.push_back(ProfRec{cls, a, b, flops, bytes, launches});
  }
};

// ----------------------------------------------------------------------------------------------
// Profiled launch wrappers (algorithmic FLOPs / bytes per launch)
// ----------------------------------------------------------------------------------------------
void G(zl_ctx* c, cudaStream_t s, int mode, int M, int N, int K, const void* A, const void* B, void* C,
       const float* bias, const void* R, float alpha = 1.f) {
  if (!C) return;   // frozen weight: no gradient to form
  const double e = (double)esz(c);
  const double out = mode == 2 ? 8.0 * M * N : (R ? 2.0 : 1.0) * e * M * N;
  const bool head = B == c->lm_head;
  ProfScope p(c, s, head ? PC_GEMM_HEAD : PC_GEMM, 2.0 * M * N * (double)K, e * ((double)M * K + (double)N * K) + out);
  gemm(c->dt, mode, M, N, K, A, B, C, bias, R, s, c->d_err, c->pool, alpha);
}
// Weight gradient of matrix p of layer li: C += A^T B into its gradient accumulator, or, with the fused
// update on (k.fuse: one micro-batch per window), the AdamW step of the matrix in the product's epilogue,
// with no gradient stored. Where the tensor-core product does not apply (fp32, or a shape outside its
// rules) the gradient is formed with gemm() in the accumulator and the step applied to the matrix's
// range right after it: the same arithmetic either way.
void GW(zl_ctx* c, cudaStream_t s, Chunk& k, int li, PK p, int M, int N, int K, const void* A, const void* B) {
  if (!trainable(k, li, p)) return;   // frozen
  float* g = Gm(k, li, p);
  if (!k.fuse) {
    if (!g) raise_err(ZL_ERR_STATE, "internal: unfused weight gradient without an accumulator");
    G(c, s, 2, M, N, K, A, B, g, nullptr, nullptr);
    return;
  }
  const zl_train_cfg& cf = c->cfg;
  const size_t off = k.layers[li].off[p];
  const bool blk = k.layers[li].blk[p];
  const GemmUpdate u{k.master + off, k.m + off, k.v + off, nullptr,
                     c->dt == BF16 ? (void*)((bf16*)k.comp + off) : nullptr, k.d_hp, cf.beta1, cf.beta2, cf.eps,
                     cf.weight_decay, 1.f, blk ? 1 : 0};
  const double e = (double)esz(c), mn = (double)M * N;
  // operands, then read theta, m, v and write them back, plus the compute copy
  const double upd = 24.0 * mn + (c->dt == BF16 ? 2.0 : 0.0) * mn;
  ProfScope ps(c, s, PC_GEMM_UPD, 2.0 * mn * (double)K, e * ((double)M * K + (double)N * K) + upd);
  if (c->dt == BF16 && gemm_tc_update(M, N, K, A, B, u, c->d_err, s, c->pool)) return;
  // the gradient in the accumulator (or, where the matrix has none, a zeroed pool buffer), then the step
  float* tmp = nullptr;
  if (!g) {
    tmp = (float*)palloc(c, (size_t)M * N * 4, s);
    CK(cudaMemsetAsync(tmp, 0, (size_t)M * N * 4, s));
  }
  float* gg = g ? g : tmp;
  gemm(c->dt, 2, M, N, K, A, B, gg, nullptr, nullptr, s, c->d_err, c->pool);
  if (blk)
    launch_adamw_span_blk(u.theta, gg, u.m, u.v, u.comp, M, N, k.d_hp, cf.beta1, cf.beta2, cf.eps, cf.weight_decay,
                          u.gscale, s);
  else
    launch_adamw_span(u.theta, gg, u.m, u.v, u.comp, (size_t)M * N, k.d_hp, cf.beta1, cf.beta2, cf.eps,
                      cf.weight_decay, u.gscale, s);
  pfree(tmp, s);
}

void AF(zl_ctx* c, cudaStream_t s, const void* qkv, void* out, float* lse, int B, int S) {
  const double e = (double)esz(c), N = (double)B * S;
  ProfScope p(c, s, PC_ATTN_F, 2.0 * B * c->H * (double)S * S * c->hd, e * N * (c->qkvw + c->ad));
  attn_fwd(c->dt, qkv, out, lse, B, S, c->H, c->Hkv, c->hd, s, c->d_err, c->pool);
}
void AB(zl_ctx* c, cudaStream_t s, const void* qkv, const void* out, const void* dout, const float* lse, float* D,
        void* dqkv, int B, int S) {
  const double e = (double)esz(c), N = (double)B * S;
  ProfScope p(c, s, PC_ATTN_B, 4.0 * B * c->H * (double)S * S * c->hd, e * N * (2.0 * c->qkvw + 2.0 * c->ad), 3);
  attn_bwd(c->dt, qkv, out, dout, lse, D, dqkv, B, S, c->H, c->Hkv, c->hd, s, c->pool, c->d_err);
}
void NF(zl_ctx* c, cudaStream_t s, const void* x, const float* g, const float* b, void* y, float* rstd, float* mean,
        int N) {
  ProfScope p(c, s, PC_NORM, 0, 2.0 * esz(c) * (double)N * c->d);
  launch_norm_fwd(c->dt, !c->llama, x, g, b, y, rstd, mean, N, c->d, c->dims.norm_eps, s);
}
void NBX(zl_ctx* c, cudaStream_t s, const void* x, const float* g, const float* rstd, const float* mean, const void* dy,
         const void* dres, void* dx, int N) {
  ProfScope p(c, s, PC_NORM, 0, (dres ? 4.0 : 3.0) * esz(c) * (double)N * c->d);
  launch_norm_bwd_dx(c->dt, !c->llama, x, g, rstd, mean, dy, dres, dx, N, c->d, s);
}
// ----------------------------------------------------------------------------------------------
// Layer forward / backward
// ----------------------------------------------------------------------------------------------
size_t layer_save_bytes(zl_ctx* c, int N, int B, int S, bool with_y) {
  const size_t e = esz(c);
  size_t b = 0;
  auto add = [&](size_t x) { b += round_up(std::max<size_t>(x, 1), 256); };
  add((size_t)N * c->d * e);        // xn1
  add((size_t)N * c->qkvw * e);     // qkv
  add((size_t)N * c->ad * e);       // att
  add((size_t)N * c->d * e);        // x2
  add((size_t)N * c->d * e);        // xn2
  add((size_t)N * c->f1 * e);       // hid
  add((size_t)N * c->f * e);        // act
  if (with_y) add((size_t)N * c->d * e);
  for (int i = 0; i < 4; ++i) add((size_t)N * 4);
  add((size_t)B * c->H * S * 4);    // lse
  const int r = lora_r16(c->cfg.lora_rank);
  if (r > 0)
    for (int i = 0; i < 4; ++i) add((size_t)N * r * e);
  return b;
}

void carve_layer(zl_ctx* c, Arena& a, LayerSave& sv, int N, int B, int S, bool with_y) {
  const size_t e = esz(c);
  sv.xn1 = a.take((size_t)N * c->d * e);
  sv.qkv = a.take((size_t)N * c->qkvw * e);
  sv.att = a.take((size_t)N * c->ad * e);
  sv.x2 = a.take((size_t)N * c->d * e);
  sv.xn2 = a.take((size_t)N * c->d * e);
  sv.hid = a.take((size_t)N * c->f1 * e);
  sv.act = a.take((size_t)N * c->f * e);
  sv.y = with_y ? a.take((size_t)N * c->d * e) : nullptr;
  sv.rstd1 = (float*)a.take((size_t)N * 4);
  sv.mean1 = (float*)a.take((size_t)N * 4);
  sv.rstd2 = (float*)a.take((size_t)N * 4);
  sv.mean2 = (float*)a.take((size_t)N * 4);
  sv.lse = (float*)a.take((size_t)B * c->H * S * 4);
  const int r = lora_r16(c->cfg.lora_rank);
  for (int i = 0; i < 4; ++i) sv.u[i] = r > 0 ? a.take((size_t)N * r * e) : nullptr;
}

// LoRA on linear i (Delta w = s B A, Section II-A): u = X A^T [N, r16], out += s u (B^T).
void lora_fwd(zl_ctx* c, Chunk& k, int li, int i, const void* X, void* out, void* u, int N, cudaStream_t s) {
  const int r = lora_r16(c->cfg.lora_rank);
  if (r <= 0) return;
  const Layer& L = k.layers[li];
  G(c, s, 0, N, r, L.lin_in[i], X, TrainC(c, k, L.la[i]), u, nullptr, nullptr);
  G(c, s, 1, N, L.lin_out[i], r, u, TrainC(c, k, L.lb[i]), out, nullptr, out, c->cfg.lora_scale);
}

// LoRA backward of linear i, after dX holds dY W: du = s dY B; d(B^T) += s u^T dY; dA += du^T X;
// dX += du A.
void lora_bwd(zl_ctx* c, Chunk& k, int li, int i, const void* X, const void* u, const void* dY, void* dX, void* du,
              int N, cudaStream_t s) {
  const int r = lora_r16(c->cfg.lora_rank);
  if (r <= 0) return;
  const Layer& L = k.layers[li];
  const float sc = c->cfg.lora_scale;
  G(c, s, 0, N, r, L.lin_out[i], dY, TrainC(c, k, L.lb[i]), du, nullptr, nullptr, sc);
  G(c, s, 2, r, L.lin_out[i], N, u, dY, k.grad + L.lb[i], nullptr, nullptr, sc);
  G(c, s, 2, r, L.lin_in[i], N, du, X, k.grad + L.la[i], nullptr, nullptr);
  G(c, s, 1, N, L.lin_in[i], r, du, TrainC(c, k, L.la[i]), dX, nullptr, dX);
}

void layer_fwd(zl_ctx* c, Chunk& k, int li, LayerSave& sv, const void* x, void* y, int B, int S, cudaStream_t s) {
  const int N = B * S, dt = c->dt;
  sv.x = x;
  NF(c, s, x, Wm(k, li, P_N1W), Wm(k, li, P_N1B), sv.xn1, sv.rstd1, sv.mean1, N);
  // Llama without LoRA on the QKV product: RoPE in the product's epilogue; otherwise a RoPE pass after
  // the product (and after the LoRA term, which the rotation must see)
  bool rotated = false;
  if (c->llama && dt == BF16 && lora_r16(c->cfg.lora_rank) <= 0) {
    const double e = (double)esz(c), M = N, Nq = c->qkvw, K = c->d;
    ProfScope p(c, s, PC_GEMM, 2.0 * M * Nq * K, e * (M * K + Nq * K + M * Nq));
    const GemmRope r{c->rope_cs, S, c->hd, (c->H + c->Hkv) * c->hd};
    rotated = gemm_tc_rope(N, c->qkvw, c->d, sv.xn1, Wc(c, k, li, P_WQKV), sv.qkv, Wm(k, li, P_BQKV), r, c->d_err,
                           s, c->pool);
    p.keep = rotated;
  }
  if (!rotated) {
    G(c, s, 0, N, c->qkvw, c->d, sv.xn1, Wc(c, k, li, P_WQKV), sv.qkv, Wm(k, li, P_BQKV), nullptr);
    lora_fwd(c, k, li, 0, sv.xn1, sv.qkv, sv.u[0], N, s);
    if (c->llama) {
      ProfScope p(c, s, PC_ELEM, 0, 2.0 * esz(c) * (double)N * (c->H + c->Hkv) * c->hd);
      launch_rope(dt, sv.qkv, c->rope_cs, N, S, c->H, c->Hkv, c->hd, 0, s);
    }
  }
  AF(c, s, sv.qkv, sv.att, sv.lse, B, S);
  G(c, s, 0, N, c->d, c->ad, sv.att, Wc(c, k, li, P_WO), sv.x2, Wm(k, li, P_BO), x);
  lora_fwd(c, k, li, 1, sv.att, sv.x2, sv.u[1], N, s);
  NF(c, s, sv.x2, Wm(k, li, P_N2W), Wm(k, li, P_N2B), sv.xn2, sv.rstd2, sv.mean2, N);
  G(c, s, 0, N, c->f1, c->d, sv.xn2, Wc(c, k, li, P_W1), sv.hid, Wm(k, li, P_B1), nullptr);
  lora_fwd(c, k, li, 2, sv.xn2, sv.hid, sv.u[2], N, s);
  {
    ProfScope p(c, s, PC_ELEM, 0, esz(c) * (double)N * (c->f1 + c->f));
    if (c->llama) launch_swiglu_fwd(dt, sv.hid, sv.act, N, c->f, s);
    else launch_gelu_fwd(dt, sv.hid, sv.act, (size_t)N * c->f, s);
  }
  G(c, s, 0, N, c->d, c->f, sv.act, Wc(c, k, li, P_W2), y, Wm(k, li, P_B2), sv.x2);
  lora_fwd(c, k, li, 3, sv.act, y, sv.u[3], N, s);
  CHECK_LAUNCH();
}

// Backward workspace of one chunk.
struct BwdWs {
  void *da, *dhid, *dxn, *dx2, *datt, *dqkv, *dy0, *dy1, *du;
  float *part_g, *part_b, *D;
  unsigned* counter;   // column-sum completion tickets, one per 256-column group (zero between launches)
};

size_t bwd_ws_bytes(zl_ctx* c, int N, int B, int S) {
  const size_t e = esz(c);
  const size_t wmax = std::max({(size_t)c->d, (size_t)c->qkvw, (size_t)c->f1, (size_t)c->f});
  size_t b = 0;
  auto add = [&](size_t x) { b += round_up(std::max<size_t>(x, 1), 256); };
  add((size_t)N * c->f * e);
  add((size_t)N * c->f1 * e);
  add((size_t)N * c->d * e);
  add((size_t)N * c->d * e);
  add((size_t)N * c->ad * e);
  add((size_t)N * c->qkvw * e);
  add((size_t)N * c->d * e);
  add((size_t)N * c->d * e);
  add((size_t)colsum_blocks(N) * wmax * 4);
  add((size_t)colsum_blocks(N) * wmax * 4);
  add((size_t)B * c->H * S * 4);
  add((size_t)colsum_groups((int)wmax) * 4);
  add((size_t)N * std::max(lora_r16(c->cfg.lora_rank), 1) * e);
  return b;
}

void carve_ws(zl_ctx* c, Arena& a, BwdWs& w, int N, int B, int S) {
  const size_t e = esz(c);
  const size_t wmax = std::max({(size_t)c->d, (size_t)c->qkvw, (size_t)c->f1, (size_t)c->f});
  w.da = a.take((size_t)N * c->f * e);
  w.dhid = a.take((size_t)N * c->f1 * e);
  w.dxn = a.take((size_t)N * c->d * e);
  w.dx2 = a.take((size_t)N * c->d * e);
  w.datt = a.take((size_t)N * c->ad * e);
  w.dqkv = a.take((size_t)N * c->qkvw * e);
  w.dy0 = a.take((size_t)N * c->d * e);
  w.dy1 = a.take((size_t)N * c->d * e);
  w.part_g = (float*)a.take((size_t)colsum_blocks(N) * wmax * 4);
  w.part_b = (float*)a.take((size_t)colsum_blocks(N) * wmax * 4);
  w.D = (float*)a.take((size_t)B * c->H * S * 4);
  w.counter = (unsigned*)a.take((size_t)colsum_groups((int)wmax) * 4);
  w.du = a.take((size_t)N * std::max(lora_r16(c->cfg.lora_rank), 1) * e);
}

// The column sums of one chunk backward (bias and norm-parameter gradients) run in order on the
// chunk's side stream: nothing reads them before the optimizer step, so they leave the layer-to-layer
// chain of the chunk stream. They share the workspace's partials and tickets, which nothing else uses.
// The main stream waits only where it overwrites a buffer that a queued sum still reads; every wait
// refers to a record made in the same backward (the flags), so none crosses a graph capture.
struct SideQ {
  Chunk* k;
  cudaStream_t s, sd;
  bool any = false, layer = false, ln2 = false, ln1 = false;
  bool on() const { return sd != s; }
  void fork() {   // the side stream waits for what the main stream has produced so far
    if (!on()) return;
    rec(k->ev_sin, s);
    wait_ev(sd, k->ev_sin);
    any = true;
  }
  bool mark(cudaEvent_t e) {   // record the side stream's position; true if recorded
    if (!on() || !any) return false;
    rec(e, sd);
    return true;
  }
  void need(cudaEvent_t e, bool recorded) {
    if (on() && recorded) wait_ev(s, e);
  }
};

void bias_grad(zl_ctx* c, const void* dY, int N, int cols, float* g, BwdWs& w, SideQ& q) {
  if (!g) return;
  q.fork();
  ProfScope p(c, q.sd, PC_ELEM, 0, esz(c) * (double)N * cols, 1);
  launch_colsum(c->dt, dY, w.part_b, N, cols, g, w.counter, q.sd);
}

void norm_param_grad(zl_ctx* c, const void* x, const float* rstd, const float* mean, const void* dyn, int N,
                     float* gw, float* gb, BwdWs& w, SideQ& q) {
  if (!gw) return;   // frozen norm
  const bool ln = !c->llama;
  q.fork();
  ProfScope p(c, q.sd, PC_NORM, 0, 2.0 * esz(c) * (double)N * c->d, 1);
  launch_norm_bwd_dparam(c->dt, ln, x, rstd, mean, dyn, w.part_g, w.part_b, N, c->d, gw, gb, w.counter, q.sd);
}

// dy: gradient w.r.t. the layer output; dx (may be NULL): gradient w.r.t. the layer input.
void layer_bwd(zl_ctx* c, Chunk& k, int li, LayerSave& sv, const void* dy, void* dx, BwdWs& w, int B, int S,
               cudaStream_t s, SideQ& q) {
  const int N = B * S, dt = c->dt;
  // the layer above queued sums over dy's buffer, dhid, dx2 and dqkv, which this layer overwrites
  q.need(k.ev_layer, q.layer);
  // Every dX product comes before the weight-gradient product of the same matrix, which may update the
  // matrix in place (fused update).
  // FFN
  G(c, s, 1, N, c->f, c->d, dy, Wc(c, k, li, P_W2), w.da, nullptr, nullptr);
  GW(c, s, k, li, P_W2, c->d, c->f, N, dy, sv.act);
  bias_grad(c, dy, N, c->d, Gm(k, li, P_B2), w, q);
  lora_bwd(c, k, li, 3, sv.act, sv.u[3], dy, w.da, w.du, N, s);
  {
    ProfScope p(c, s, PC_ELEM, 0, esz(c) * (double)N * (2.0 * c->f1 + c->f));
    if (c->llama) launch_swiglu_bwd(dt, sv.hid, w.da, w.dhid, N, c->f, s);
    else launch_gelu_bwd(dt, sv.hid, w.da, w.dhid, (size_t)N * c->f, s);
  }
  q.need(k.ev_ln1, q.ln1);   // the layer above's LN1 parameter sums read dxn
  G(c, s, 1, N, c->d, c->f1, w.dhid, Wc(c, k, li, P_W1), w.dxn, nullptr, nullptr);
  GW(c, s, k, li, P_W1, c->f1, c->d, N, w.dhid, sv.xn2);
  bias_grad(c, w.dhid, N, c->f1, Gm(k, li, P_B1), w, q);
  lora_bwd(c, k, li, 2, sv.xn2, sv.u[2], w.dhid, w.dxn, w.du, N, s);
  NBX(c, s, sv.x2, Wm(k, li, P_N2W), sv.rstd2, sv.mean2, w.dxn, dy, w.dx2, N);
  norm_param_grad(c, sv.x2, sv.rstd2, sv.mean2, w.dxn, N, Gm(k, li, P_N2W), Gm(k, li, P_N2B), w, q);
  q.ln2 = q.mark(k.ev_ln2);
  // attention
  G(c, s, 1, N, c->ad, c->d, w.dx2, Wc(c, k, li, P_WO), w.datt, nullptr, nullptr);
  GW(c, s, k, li, P_WO, c->d, c->ad, N, w.dx2, sv.att);
  bias_grad(c, w.dx2, N, c->d, Gm(k, li, P_BO), w, q);
  lora_bwd(c, k, li, 1, sv.att, sv.u[1], w.dx2, w.datt, w.du, N, s);
  AB(c, s, sv.qkv, sv.att, w.datt, sv.lse, w.D, w.dqkv, B, S);
  if (c->llama) {
    ProfScope p(c, s, PC_ELEM, 0, 2.0 * esz(c) * (double)N * (c->H + c->Hkv) * c->hd);
    launch_rope(dt, w.dqkv, c->rope_cs, N, S, c->H, c->Hkv, c->hd, 1, s);
  }
  q.need(k.ev_ln2, q.ln2);        // LN2 parameter sums read dxn, which the next product overwrites
  G(c, s, 1, N, c->d, c->qkvw, w.dqkv, Wc(c, k, li, P_WQKV), w.dxn, nullptr, nullptr);
  GW(c, s, k, li, P_WQKV, c->qkvw, c->d, N, w.dqkv, sv.xn1);
  bias_grad(c, w.dqkv, N, c->qkvw, Gm(k, li, P_BQKV), w, q);
  q.layer = q.mark(k.ev_layer);   // after this layer's sums over dy, dhid, dx2 and dqkv
  lora_bwd(c, k, li, 0, sv.xn1, sv.u[0], w.dqkv, w.dxn, w.du, N, s);
  norm_param_grad(c, sv.x, sv.rstd1, sv.mean1, w.dxn, N, Gm(k, li, P_N1W), Gm(k, li, P_N1B), w, q);
  q.ln1 = q.mark(k.ev_ln1);
  if (dx) NBX(c, s, sv.x, Wm(k, li, P_N1W), sv.rstd1, sv.mean1, w.dxn, w.dx2, dx, N);
  CHECK_LAUNCH();
}

// ----------------------------------------------------------------------------------------------
// Chunk forward (saving or not) and the chunk backward
// ----------------------------------------------------------------------------------------------
struct ChunkActs {
  void* mem = nullptr;
  std::vector<LayerSave> L;
};

// Saving forward: the arena holds every layer's activations; the chunk output goes to h_out.
void chunk_fwd_save(zl_ctx* c, Chunk& k, const void* h_in, void* h_out, int B, int S, ChunkActs& acts,
                    cudaStream_t s) {
  const int N = B * S, nl = k.l1 - k.l0;
  size_t bytes = 0;
  for (int i = 0; i < nl; ++i) bytes += layer_save_bytes(c, N, B, S, i + 1 < nl);
  Arena a;
  a.base = (char*)palloc(c, bytes, s);
  a.cap = bytes;
  acts.mem = a.base;
  acts.L.assign(nl, LayerSave{});
  const void* x = h_in;
  for (int i = 0; i < nl; ++i) {
    carve_layer(c, a, acts.L[i], N, B, S, i + 1 < nl);
    void* y = i + 1 < nl ? acts.L[i].y : h_out;
    layer_fwd(c, k, i, acts.L[i], x, y, B, S, s);
    x = y;
  }
}

// Forward without saving (one transient layer workspace, ping-pong outputs).
void chunk_fwd_nosave(zl_ctx* c, Chunk& k, const void* h_in, void* h_out, int B, int S, cudaStream_t s) {
  const int N = B * S, nl = k.l1 - k.l0;
  const size_t lb = layer_save_bytes(c, N, B, S, true) + round_up((size_t)N * c->d * esz(c), 256);
  Arena a;
  a.base = (char*)palloc(c, lb, s);
  a.cap = lb;
  LayerSave sv;
  carve_layer(c, a, sv, N, B, S, true);
  void* pong = a.take((size_t)N * c->d * esz(c));
  const void* x = h_in;
  for (int i = 0; i < nl; ++i) {
    void* y = (i + 1 == nl) ? h_out : ((i % 2 == 0) ? sv.y : pong);
    layer_fwd(c, k, i, sv, x, y, B, S, s);
    x = y;
  }
  pfree(a.base, s);
}

// Backward through the chunk from dh (gradient at its output). dh_in (may be NULL) receives the
// gradient at its input (only the backpropagation baseline needs it).
void chunk_bwd(zl_ctx* c, Chunk& k, ChunkActs& acts, const void* dh, void* dh_in, int B, int S, cudaStream_t s) {
  const int N = B * S, nl = k.l1 - k.l0;
  const size_t wb = bwd_ws_bytes(c, N, B, S);
  Arena a;
  a.base = (char*)palloc(c, wb, s);
  a.cap = wb;
  BwdWs w;
  carve_ws(c, a, w, N, B, S);
  const size_t wmax = std::max({(size_t)c->d, (size_t)c->qkvw, (size_t)c->f1, (size_t)c->f});
  CK(cudaMemsetAsync(w.counter, 0, (size_t)colsum_groups((int)wmax) * 4, s));
  SideQ q{&k, s, k.side ? k.side : s};
  const void* dy = dh;
  for (int i = nl - 1; i >= 0; --i) {
    void* dx = i > 0 ? ((i % 2) ? w.dy0 : w.dy1) : dh_in;
    layer_bwd(c, k, i, acts.L[i], dy, dx, w, B, S, s, q);
    dy = dx;
  }
  if (q.mark(k.ev_send)) wait_ev(s, k.ev_send);   // the sums are done before the workspace goes back
  pfree(a.base, s);
}

// Before the backward of one micro-batch of chunk k: when the fused update applies (one micro-batch per
// window, full fine-tune, cfg.unfused_update = 0), advance the step count and write this step's lr and
// bias corrections now, so the weight-gradient products can apply the step.
void window_begin(zl_ctx* c, Chunk& k, cudaStream_t s) {
  const zl_train_cfg& g = c->cfg;
  k.fuse = g.accum_m == 1 && !g.unfused_update && g.lora_rank == 0;
  if (k.fuse) launch_adamw_tick(k.d_t, k.d_hp, g.lr, g.lr_schedule, g.lr_gamma, g.beta1, g.beta2, s);
}

// After the backward: at the window's end the AdamW step of whatever the backward did not update (all of
// the slab, or, after a fused backward, its non-matrix ranges). adapters = false (the backpropagation
// step): the readout adapter, at the end of the slab, is left as is.
void adamw_window(zl_ctx* c, Chunk& k, cudaStream_t s, bool adapters = true) {
  k.micro += 1;
  if (k.micro < c->cfg.accum_m) return;
  k.t += 1;
  const zl_train_cfg& g = c->cfg;
  k.micro = 0;
  const float gscale = 1.f / (float)g.accum_m;
  if (k.fuse) {
    const int nr = adapters ? k.n_ranges : k.n_ranges_layers;
    double n = 0;
    for (int i = 0; i < nr; ++i) n += (double)k.h_ranges[2 * i + 1];
    ProfScope p(c, s, PC_ADAMW, 0, (c->dt == BF16 ? 34.0 : 32.0) * n);
    launch_adamw_ranges(k.master, k.grad, k.m, k.v, c->dt == BF16 ? k.comp : nullptr, k.d_ranges, nr, k.max_range,
                        k.d_hp, g.beta1, g.beta2, g.eps, g.weight_decay, gscale, s);
    k.fuse = false;
    CHECK_LAUNCH();
    return;
  }
  if (k.grad_n < k.n) raise_err(ZL_ERR_STATE, "internal: slab update without a full gradient accumulator");
  void* comp = c->dt == BF16 ? k.comp : nullptr;
  const bool skip_ad = !adapters && g.adapter_dim > 0;   // the slab but the adapter [ad_down, ad_end)
  const size_t n1 = skip_ad ? k.ad_down : k.n;
  const double nu = (double)(skip_ad ? k.n - (k.ad_end - k.ad_down) : k.n);
  ProfScope p(c, s, PC_ADAMW, 0, (c->dt == BF16 ? 34.0 : 32.0) * nu);
  launch_adamw(k.master, k.grad, k.m, k.v, comp, n1, k.d_t, k.d_hp, g.lr, g.lr_schedule, g.lr_gamma, g.beta1, g.beta2,
               g.eps, g.weight_decay, gscale, s);
  if (skip_ad)
    launch_adamw_span(k.master + k.ad_end, k.grad + k.ad_end, k.m + k.ad_end, k.v + k.ad_end,
                      comp ? (void*)((bf16*)comp + k.ad_end) : nullptr, k.n - k.ad_end, k.d_hp, g.beta1, g.beta2,
                      g.eps, g.weight_decay, gscale, s);
  CHECK_LAUNCH();
}

float alpha_of(zl_ctx* c, int k) { return (k == 1 && !c->cfg.consis_first) ? 1.f : c->cfg.alpha; }

// Keeps chunk k's input of micro-batch `seq` (h_{k-1} and the labels) in its hidden-state buffer.
void ring_put(zl_ctx* c, Chunk& ck, long seq, const void* h_in, const int32_t* labels, int B, int S, cudaStream_t s) {
  const int D = c->cfg.replay_depth;
  if (D <= 0) return;
  if ((int)ck.ring.size() != D) ck.ring.resize(D);
  Chunk::Entry& e = ck.ring[seq % D];
  const size_t N = (size_t)B * S;
  if (e.cap < N) {   // grow (rare): wait for this stream's use of the old buffers first
    CK(cudaStreamSynchronize(s));
    if (e.h) { CK(cudaFree(e.h)); c->static_bytes -= e.cap * c->d * esz(c); }
    if (e.labels) { CK(cudaFree(e.labels)); c->static_bytes -= e.cap * 4; }
    CK(cudaMalloc(&e.h, N * c->d * esz(c)));
    CK(cudaMalloc((void**)&e.labels, N * 4));
    c->static_bytes += N * c->d * esz(c) + N * 4;
    e.cap = N;
  }
  CK(cudaMemcpyAsync(e.h, h_in, N * c->d * esz(c), cudaMemcpyDeviceToDevice, s));
  CK(cudaMemcpyAsync(e.labels, labels, N * 4, cudaMemcpyDeviceToDevice, s));
  e.seq = seq;
  e.B = B;
  e.S = S;
}

// ----------------------------------------------------------------------------------------------
// Readout (Eq. 2) and its backward (frozen head: no parameter gradient)
// ----------------------------------------------------------------------------------------------
struct ReadoutSave {
  void* n = nullptr;
  float *rstd = nullptr, *mean = nullptr;
  void *a = nullptr, *u = nullptr;   // adapter: a_k(h) and h D^T
};

// z = Norm_f(x) W_lm^T with x = h, or x = a_k(h) = h + GELU(h D^T) U^T when `ad` (chunk k's readout
// adapter, Section III-B (b)) is given.
void readout_fwd(zl_ctx* c, const void* h, void* z, ReadoutSave* keep, int N, cudaStream_t s,
                 Chunk* ad = nullptr) {
  const size_t e = esz(c);
  const void* x = h;
  void *a = nullptr, *u = nullptr;
  if (ad && c->cfg.adapter_dim > 0) {
    const int ra = c->cfg.adapter_dim;
    u = palloc(c, (size_t)N * ra * e, s);
    void* gact = palloc(c, (size_t)N * ra * e, s);
    a = palloc(c, (size_t)N * c->d * e, s);
    G(c, s, 0, N, ra, c->d, h, TrainC(c, *ad, ad->ad_down), u, nullptr, nullptr);
    {
      ProfScope p(c, s, PC_ELEM, 0, 2.0 * e * (double)N * ra);
      launch_gelu_fwd(c->dt, u, gact, (size_t)N * ra, s);
    }
    G(c, s, 0, N, c->d, ra, gact, TrainC(c, *ad, ad->ad_up), a, nullptr, h);
    pfree(gact, s);
    x = a;
  }
  void* n = palloc(c, (size_t)N * c->d * e, s);
  float* st = (float*)palloc(c, (size_t)N * 8, s);
  NF(c, s, x, c->normf_w, c->normf_b, n, st, st + N, N);
  G(c, s, 0, N, c->Vp, c->d, n, c->lm_head, z, nullptr, nullptr);
  CHECK_LAUNCH();
  if (keep) {
    keep->n = n;
    keep->rstd = st;
    keep->mean = st + N;
    keep->a = a;
    keep->u = u;
  } else {
    pfree(n, s);
    pfree(st, s);
    pfree(a, s);
    pfree(u, s);
  }
}

// dh = d/dh of the readout: Norm_f'(x)^T (dz W_lm), through the adapter when it was applied:
// da = Norm_f'(a)^T dn;  dU += da^T GELU(u);  du = (da U) * GELU'(u);  dD += du^T h;  dh = da + du D.
void readout_bwd(zl_ctx* c, const void* h, ReadoutSave& rs, const void* dz, void* dh, int N, cudaStream_t s,
                 Chunk* ad = nullptr) {
  G(c, s, 1, N, c->d, c->Vp, dz, c->lm_head, rs.n, nullptr, nullptr);   // reuse n as dn
  if (!rs.a) {
    NBX(c, s, h, c->normf_w, rs.rstd, rs.mean, rs.n, nullptr, dh, N);
  } else {
    const int ra = c->cfg.adapter_dim;
    const size_t e = esz(c);
    void* da = palloc(c, (size_t)N * c->d * e, s);
    void* gact = palloc(c, (size_t)N * ra * e, s);
    void* dg = palloc(c, (size_t)N * ra * e, s);
    NBX(c, s, rs.a, c->normf_w, rs.rstd, rs.mean, rs.n, nullptr, da, N);
    {
      ProfScope p(c, s, PC_ELEM, 0, 2.0 * e * (double)N * ra);
      launch_gelu_fwd(c->dt, rs.u, gact, (size_t)N * ra, s);
    }
    G(c, s, 2, c->d, ra, N, da, gact, ad->grad + ad->ad_up, nullptr, nullptr);
    G(c, s, 1, N, ra, c->d, da, TrainC(c, *ad, ad->ad_up), dg, nullptr, nullptr);
    {
      ProfScope p(c, s, PC_ELEM, 0, 3.0 * e * (double)N * ra);
      launch_gelu_bwd(c->dt, rs.u, dg, gact, (size_t)N * ra, s);   // gact now holds du
    }
    G(c, s, 2, ra, c->d, N, gact, h, ad->grad + ad->ad_down, nullptr, nullptr);
    G(c, s, 1, N, c->d, ra, gact, TrainC(c, *ad, ad->ad_down), dh, nullptr, da);
    pfree(da, s);
    pfree(gact, s);
    pfree(dg, s);
    pfree(rs.a, s);
    pfree(rs.u, s);
  }
  CHECK_LAUNCH();
  pfree(rs.n, s);
  pfree(rs.rstd, s);
  rs = ReadoutSave{};
}

// Readout (Eq. 2), local objective (Eq. 3-5) and head backward over row slices of R rows, so that the
// vocab-sized logits exist for R rows at a time only (the head fused with the loss): for each slice
// z_s = n_s W^T, t_s = tn_s W^T (the stop-gradient teacher, when tn is given), the fused loss writes
// dz_s in place of z_s and the per-row losses, and (backward) dn_s = dz_s W. n, tn [N, d]: the final-norm
// outputs of the chunk's hidden state and of its input; W [Vp, d] the frozen head (rows >= V zero);
// count: |Omega| of all N rows (already counted); dn [N, d] may be n (slice s of n is read before dn_s
// is written, in stream order); zb, tb: [R, Vp] slice buffers. c may be NULL (no profiling).
void head_loss_rows(zl_ctx* c, int dt, const void* n, const void* tn, const void* W, const int32_t* labels, int N,
                    int d, int V, int Vp, float alpha, int kl_dir, int R, const int* count, void* dn, float* rl,
                    void* zb, void* tb, bool backward, cudaStream_t s, unsigned* err, cudaMemPool_t pool) {
  const size_t e = dt_size(dt);
  const double ed = (double)e;
  auto gm = [&](int mode, int M, int Nn, int K, const void* A, const void* B, void* C) {
    ProfScope p(c, s, PC_GEMM_HEAD, 2.0 * M * Nn * (double)K, ed * ((double)M * K + (double)Nn * K + (double)M * Nn));
    gemm(dt, mode, M, Nn, K, A, B, C, nullptr, nullptr, s, err, pool);
  };
  const bool teacher = alpha < 1.f && tn;
  for (int r0 = 0; r0 < N; r0 += R) {
    const int rows = std::min(R, N - r0);
    const size_t ro = (size_t)r0 * d * e;
    gm(0, rows, Vp, d, (const char*)n + ro, W, zb);
    if (teacher) gm(0, rows, Vp, d, (const char*)tn + ro, W, tb);
    {
      ProfScope p(c, s, PC_LOSS, 0, (teacher ? 3.0 : 2.0) * ed * (double)rows * Vp);
      launch_local_loss(dt, zb, teacher ? tb : nullptr, labels + r0, rows, V, Vp, alpha, kl_dir, count, zb, rl + r0, s);
    }
    if (backward) gm(1, rows, d, Vp, zb, W, (char*)dn + ro);
  }
}

// The readout, local objective and head backward of one chunk with the logits in row slices of
// cfg.loss_rows rows (head_loss_rows): the teacher p_{k-1} is the frozen head on h_prev, the loss goes to
// d_losses[slot] and, with backward, dh receives Norm_f'(h)^T dn. alpha == 1: no teacher (h_prev unused).
void readout_loss_sliced(zl_ctx* c, const void* h, const void* h_prev, const int32_t* labels, float alpha, int N,
                         int slot, void* dh, bool backward, cudaStream_t s) {
  const size_t e = esz(c);
  const int R = std::min(N, c->cfg.loss_rows);
  void* n = palloc(c, (size_t)N * c->d * e, s);
  float* st = (float*)palloc(c, (size_t)N * 8, s);
  NF(c, s, h, c->normf_w, c->normf_b, n, st, st + N, N);
  void *tn = nullptr, *tb = nullptr;
  float* tst = nullptr;
  if (alpha < 1.f) {
    tn = palloc(c, (size_t)N * c->d * e, s);
    tst = (float*)palloc(c, (size_t)N * 8, s);
    NF(c, s, h_prev, c->normf_w, c->normf_b, tn, tst, tst + N, N);
    tb = palloc(c, (size_t)R * c->Vp * e, s);
  }
  void* zb = palloc(c, (size_t)R * c->Vp * e, s);
  float* rl = (float*)palloc(c, (size_t)N * 4, s);
  launch_count_valid(labels, N, c->V, c->d_count + slot, c->d_err, s);
  head_loss_rows(c, c->dt, n, tn, c->lm_head, labels, N, c->d, c->V, c->Vp, alpha, c->cfg.kl_dir, R, c->d_count + slot,
                 n, rl, zb, tb, backward, s, c->d_err, c->pool);
  launch_loss_reduce(rl, N, c->d_count + slot, c->d_losses + slot, s);
  if (backward) NBX(c, s, h, c->normf_w, st, st + N, n, nullptr, dh, N);
  CHECK_LAUNCH();
  for (void* p : {(void*)rl, zb, tb, tn, (void*)tst, n, (void*)st}) pfree(p, s);
}

// Loss of chunk slot `slot` into d_losses[slot]; returns dz (pool memory, caller frees).
void* local_loss(zl_ctx* c, const void* z, const void* t, const int32_t* labels, float alpha, int N, int slot,
                 cudaStream_t s) {
  void* dz = palloc(c, (size_t)N * c->Vp * esz(c), s);
  float* rl = (float*)palloc(c, (size_t)N * 4, s);
  launch_count_valid(labels, N, c->V, c->d_count + slot, c->d_err, s);
  {
    ProfScope p(c, s, PC_LOSS, 0, (alpha < 1.f ? 3.0 : 2.0) * esz(c) * (double)N * c->Vp);
    launch_local_loss(c->dt, z, alpha < 1.f ? t : nullptr, labels, N, c->V, c->Vp, alpha, c->cfg.kl_dir,
                      c->d_count + slot, dz, rl, s);
  }
  launch_loss_reduce(rl, N, c->d_count + slot, c->d_losses + slot, s);
  CHECK_LAUNCH();
  pfree(rl, s);
  return dz;
}

// ----------------------------------------------------------------------------------------------
// synchronisation
// ----------------------------------------------------------------------------------------------
void join_all(zl_ctx* c) {
  for (int k = 1; k <= c->K; ++k) {
    rec(c->ch[k].ev_done, c->ch[k].s);
    wait_ev(c->user, c->ch[k].ev_done);
  }
  rec(c->ev_aux, c->aux);
  wait_ev(c->user, c->ev_aux);
}

zl_status sync_all(zl_ctx* c, int timeout_ms) {
  join_all(c);
  rec(c->ev_sync, c->user);
  const auto t0 = std::chrono::steady_clock::now();
  for (;;) {
    cudaError_t e = cudaEventQuery(c->ev_sync);
    if (e == cudaSuccess) break;
    if (e != cudaErrorNotReady) CK(e);
    if (timeout_ms >= 0 &&
        std::chrono::duration_cast<std::chrono::milliseconds>(std::chrono::steady_clock::now() - t0).count() >
            timeout_ms)
      raise_err(ZL_ERR_TIMEOUT, "zl_synchronize: queued work did not finish in time");
    std::this_thread::sleep_for(std::chrono::microseconds(50));
  }
  unsigned err = 0;
  CK(cudaMemcpy(&err, c->d_err, 4, cudaMemcpyDeviceToHost));
  if (err) {
    CK(cudaMemset(c->d_err, 0, 4));
    std::string m = "device-side argument error:";
    if (err & ZL_DEVERR_BAD_ID) m += " token id out of [0, vocab);";
    if (err & ZL_DEVERR_BAD_LABEL) m += " label out of [-1, vocab);";
    if (err & ZL_DEVERR_TIMEOUT) m += " bounded wait expired in a kernel;";
    raise_err(ZL_ERR_ARG, m);
  }
  return ZL_OK;
}

void start_on(zl_ctx* c, cudaStream_t s) {   // order s after the user's stream
  rec(c->ev_start, c->user);
  wait_ev(s, c->ev_start);
}

void check_bs(zl_ctx* c, int B, int S) {
  if (B <= 0 || S <= 0) raise_err(ZL_ERR_ARG, "empty micro-batch (B and S must be >= 1)");
  if (S > c->dims.max_seq) raise_err(ZL_ERR_ARG, "S exceeds max_seq");
  // |Omega| is counted in fp32 partial sums, exact up to 2^24 positions
  if ((long)B * S > (1L << 24)) raise_err(ZL_ERR_ARG, "B*S above 2^24 tokens");
  if (B > 65535) raise_err(ZL_ERR_ARG, "B above 65535");
}

// ----------------------------------------------------------------------------------------------
// Name lookup
// ----------------------------------------------------------------------------------------------
struct Found {
  void* dev = nullptr;          // compute-dtype or fp32 pointer of the tensor
  bool fp32 = true;
  size_t numel = 0;
  Chunk* chunk = nullptr;       // trainable: owning chunk
  size_t off = 0;
  int frozen = 0;               // 1 tok_emb, 2 pos_emb, 3 norm_f.weight, 4 norm_f.bias, 5 lm_head
  int trows = 0, tcols = 0;     // > 0: user layout [tcols, trows], stored transposed as [trows, tcols]
  int brows = 0, bcols = 0;     // > 0: master and moments stored in the blocked layout of [brows, bcols]
};

bool lookup(zl_ctx* c, const std::string& name, Found& f) {
  const size_t Vd = (size_t)c->V * c->d;
  if (name == "tok_emb") { f = Found{c->tok_emb, c->dt == F32, Vd, nullptr, 0, 1}; return true; }
  if (name == "pos_emb" && !c->llama) {
    f = Found{c->pos_emb, c->dt == F32, (size_t)c->dims.max_seq * c->d, nullptr, 0, 2};
    return true;
  }
  if (name == "norm_f.weight") { f = Found{c->normf_w, true, (size_t)c->d, nullptr, 0, 3}; return true; }
  if (name == "norm_f.bias" && !c->llama) { f = Found{c->normf_b, true, (size_t)c->d, nullptr, 0, 4}; return true; }
  if (name == "lm_head" && c->llama) { f = Found{c->lm_head, c->dt == F32, Vd, nullptr, 0, 5}; return true; }
  if (name.rfind("adapters.", 0) == 0 && c->cfg.adapter_dim > 0) {
    const size_t dot = name.find('.', 9);
    if (dot == std::string::npos) return false;
    int k = -1;
    try { k = std::stoi(name.substr(9, dot - 9)); } catch (...) { return false; }
    if (k < 1 || k > c->K || name.substr(9, dot - 9) != std::to_string(k)) return false;
    Chunk& ck = c->ch[k];
    const std::string suf = name.substr(dot + 1);
    const size_t n = (size_t)c->cfg.adapter_dim * c->d;
    if (suf == "down") { f = Found{ck.master + ck.ad_down, true, n, &ck, ck.ad_down, 0}; return true; }
    if (suf == "up") { f = Found{ck.master + ck.ad_up, true, n, &ck, ck.ad_up, 0}; return true; }
    return false;
  }
  if (name.rfind("layers.", 0) != 0) return false;
  const size_t dot = name.find('.', 7);
  if (dot == std::string::npos) return false;
  int l = -1;
  try { l = std::stoi(name.substr(7, dot - 7)); } catch (...) { return false; }
  if (l < 0 || l >= c->dims.n_layers) return false;
  const std::string suf = name.substr(dot + 1);
  for (int k = 1; k <= c->K; ++k) {
    Chunk& ck = c->ch[k];
    if (l < ck.l0 || l >= ck.l1) continue;
    const Layer& L = ck.layers[l - ck.l0];
    for (int p = 0; p < P_COUNT; ++p)
      if (L.has[p] && suf == kPName[p]) {
        if (L.slab[p] == S_TRAIN) {
          f = Found{ck.master + L.off[p], true, L.numel[p], &ck, L.off[p], 0};
          if (L.blk[p]) { f.brows = L.rows[p]; f.bcols = L.cols[p]; }
        }
        else if (L.slab[p] == S_FVEC) f = Found{ck.fvec + L.off[p], true, L.numel[p], nullptr, 0, 0};
        else f = Found{(char*)ck.fmat + L.off[p] * esz(c), c->dt == F32, L.numel[p], nullptr, 0, 0};
        return true;
      }
    if (c->cfg.lora_rank > 0)
      for (int i = 0; i < 4; ++i) {
        const std::string base = kPName[kLoraP[i]];
        const size_t r = (size_t)c->cfg.lora_rank;
        if (suf == base + ".lora_a") { f = Found{ck.master + L.la[i], true, r * L.lin_in[i], &ck, L.la[i], 0}; return true; }
        if (suf == base + ".lora_b") {
          f = Found{ck.master + L.lb[i], true, r * L.lin_out[i], &ck, L.lb[i], 0};
          f.trows = (int)r;
          f.tcols = L.lin_out[i];
          return true;
        }
      }
  }
  return false;
}

void free_ctx(zl_ctx* c) {
  if (!c) return;
  cudaDeviceSynchronize();
  for (zl_ctx::StepGraph* g : {&c->zg, &c->bg}) {
    if (g->exec) cudaGraphExecDestroy(g->exec);
    if (g->ids) cudaFree(g->ids);
    if (g->labels) cudaFree(g->labels);
  }
  if (c->cap) cudaStreamDestroy(c->cap);
  const bool shared = c->cfg.serialize != 0;
  for (int k = 1; k < (int)c->ch.size(); ++k) {
    Chunk& ck = c->ch[k];
    for (auto& e : ck.ring) {
      if (e.h) cudaFree(e.h);
      if (e.labels) cudaFree(e.labels);
    }
    if (ck.s && (!shared || k == 1)) cudaStreamDestroy(ck.s);
    if (ck.side && !shared) cudaStreamDestroy(ck.side);
    for (cudaEvent_t e : {ck.ev_h, ck.ev_z, ck.ev_loss, ck.ev_hb, ck.ev_done, ck.ev_sin, ck.ev_ln2, ck.ev_layer,
                          ck.ev_ln1, ck.ev_send})
      if (e) cudaEventDestroy(e);
  }
  for (cudaEvent_t e : c->live_ring) cudaEventDestroy(e);
  for (cudaEvent_t e : {c->ev_start, c->ev_aux, c->ev_sync})
    if (e) cudaEventDestroy(e);
  if (c->aux && !shared) cudaStreamDestroy(c->aux);
  for (void* p : c->statics) cudaFree(p);
  if (c->h_losses) cudaFreeHost(c->h_losses);
  if (c->pool) cudaMemPoolDestroy(c->pool);
  delete c;
}

template <typename F>
zl_status guarded(zl_ctx* c, F&& fn) {
  if (c && c->broken) { g_err = "context unusable after an earlier sticky CUDA error"; return ZL_ERR_STATE; }
  try {
    return fn();
  } catch (const ZlError& e) {
    g_err = e.msg;
    if (c && e.st == ZL_ERR_STATE) c->broken = true;
    return e.st;
  } catch (const std::exception& e) {
    g_err = std::string("internal error: ") + e.what();
    return ZL_ERR_CUDA;
  }
}

}  // namespace

// ================================================================================================
// C ABI
// ================================================================================================
extern "C" {

const char* zl_last_error(void) { return g_err.c_str(); }

}  // extern "C"

namespace zl {
void set_last_error(const char* msg) { g_err = msg ? msg : ""; }
}  // namespace zl

extern "C" {

zl_status zl_create(const zl_model_dims* dims, int K, const int* bounds, const zl_train_cfg* cfg, zl_ctx** out) {
  if (!dims || !bounds || !cfg || !out) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  *out = nullptr;
  const zl_model_dims& D = *dims;
  std::string why;
  if (D.arch != ZL_ARCH_LLAMA && D.arch != ZL_ARCH_GPT2) why = "arch";
  else if (D.dtype != ZL_DTYPE_F32 && D.dtype != ZL_DTYPE_BF16) why = "dtype";
  else if (D.n_layers < 1 || D.d_model < 8 || D.n_heads < 1 || D.n_kv_heads < 1 || D.d_ff < 8 || D.vocab < 2 ||
           D.max_seq < 1) why = "non-positive dimension";
  else if (D.d_model % D.n_heads != 0) why = "d_model must be n_heads * head_dim";
  else if ((D.d_model / D.n_heads) % 2 != 0 || D.d_model / D.n_heads > 128) why = "head_dim must be even and <= 128";
  else if (D.n_heads % D.n_kv_heads != 0) why = "n_heads must be a multiple of n_kv_heads";
  else if (D.arch == ZL_ARCH_GPT2 && D.n_kv_heads != D.n_heads) why = "GPT-2 blocks use n_kv_heads == n_heads";
  else if (D.d_model % 8 != 0 || D.d_ff % 8 != 0) why = "d_model and d_ff must be multiples of 8";
  else if (D.d_model > 16384) why = "d_model above 16384 is not supported";
  else if (cfg->adapter_dim < 0 || cfg->adapter_dim % 16 != 0 || cfg->adapter_dim > D.d_model)
    why = "adapter_dim must be 0 or a multiple of 16 up to d_model";
  else if (!(D.norm_eps > 0.f)) why = "norm_eps";
  else if (K < 1 || K > D.n_layers) why = "K must be in [1, n_layers]";
  else if (bounds[0] != 0 || bounds[K] != D.n_layers) why = "bounds[0] must be 0 and bounds[K] n_layers";
  else if (!(cfg->alpha > 0.f && cfg->alpha <= 1.f)) why = "alpha must be in (0, 1]";
  else if (cfg->kl_dir != 0 && cfg->kl_dir != 1) why = "kl_dir must be 0 or 1";
  else if (cfg->accum_m < 1) why = "accum_m must be >= 1";
  else if (cfg->max_live_chunks < 0) why = "max_live_chunks must be >= 0";
  else if (cfg->lr_schedule != 0 && cfg->lr_schedule != 1) why = "lr_schedule";
  else if (cfg->lr_schedule == 1 && !(cfg->lr_gamma > 0.f)) why = "lr_gamma must be > 0";
  else if (cfg->serialize != 0 && cfg->serialize != 1) why = "serialize must be 0 or 1";
  else if (cfg->lora_rank < 0 || cfg->lora_rank > 256) why = "lora_rank must be in [0, 256]";
  else if (cfg->replay_depth < 0 || cfg->replay_depth > 4096) why = "replay_depth must be in [0, 4096]";
  else if (cfg->lora_rank > 0 && !(std::isfinite(cfg->lora_scale))) why = "lora_scale must be finite";
  else if (cfg->fuzz_delay_us < 0 || cfg->fuzz_delay_us > 100000) why = "fuzz_delay_us must be in [0, 100000]";
  else if (cfg->unfused_update != 0 && cfg->unfused_update != 1) why = "unfused_update must be 0 or 1";
  else if (cfg->loss_rows < 0) why = "loss_rows must be >= 0";
  for (int k = 1; why.empty() && k <= K; ++k)
    if (bounds[k] <= bounds[k - 1]) why = "bounds must be strictly increasing";
  if (!why.empty()) { g_err = "zl_create: " + why; return ZL_ERR_ARG; }
  if (cfg->loss_rows > 0 && cfg->adapter_dim > 0) {
    g_err = "zl_create: the row-sliced head (loss_rows > 0) does not take readout adapters";
    return ZL_ERR_UNSUPPORTED;
  }

  zl_ctx* c = new zl_ctx();
  zl_status st = guarded(nullptr, [&]() -> zl_status {
    c->dims = D;
    c->cfg = *cfg;
    c->fuzz_state = (uint64_t)cfg->fuzz_seed * 0x9E3779B97F4A7C15ull;
    c->K = K;
    c->bounds.assign(bounds, bounds + K + 1);
    c->dt = D.dtype;
    c->llama = D.arch == ZL_ARCH_LLAMA;
    c->d = D.d_model;
    c->H = D.n_heads;
    c->Hkv = D.n_kv_heads;
    c->hd = D.d_model / D.n_heads;
    c->qkvw = (c->H + 2 * c->Hkv) * c->hd;
    c->ad = c->H * c->hd;
    c->f = D.d_ff;
    c->f1 = c->llama ? 2 * D.d_ff : D.d_ff;
    c->V = D.vocab;
    c->Vp = (int)round_up((size_t)D.vocab, 128);
    const size_t e = esz(c);

    int dev = 0;
    CK(cudaGetDevice(&dev));
    cudaMemPoolProps props = {};
    props.allocType = cudaMemAllocationTypePinned;
    props.location.type = cudaMemLocationTypeDevice;
    props.location.id = dev;
    CK(cudaMemPoolCreate(&c->pool, &props));
    uint64_t thr = UINT64_MAX;
    CK(cudaMemPoolSetAttribute(c->pool, cudaMemPoolAttrReleaseThreshold, &thr));

    // frozen tensors
    c->tok_emb = salloc(c, (size_t)c->V * c->d * e);
    CK(cudaMemset(c->tok_emb, 0, (size_t)c->V * c->d * e));
    if (!c->llama) {
      c->pos_emb = salloc(c, (size_t)D.max_seq * c->d * e);
      CK(cudaMemset(c->pos_emb, 0, (size_t)D.max_seq * c->d * e));
    }
    c->normf_w = (float*)salloc(c, (size_t)c->d * 4);
    c->normf_b = (float*)salloc(c, (size_t)c->d * 4);
    {
      std::vector<float> ones(c->d, 1.f);
      CK(cudaMemcpy(c->normf_w, ones.data(), (size_t)c->d * 4, cudaMemcpyHostToDevice));
      CK(cudaMemset(c->normf_b, 0, (size_t)c->d * 4));
    }
    c->lm_head = salloc(c, (size_t)c->Vp * c->d * e);   // padded rows stay zero
    CK(cudaMemset(c->lm_head, 0, (size_t)c->Vp * c->d * e));
    if (c->llama) {   // rotary table (cos, sin) for positions 0..max_seq-1, computed in double
      const int half = c->hd / 2;
      std::vector<float> cs((size_t)D.max_seq * half * 2);
      for (int s = 0; s < D.max_seq; ++s)
        for (int i = 0; i < half; ++i) {
          const double ang = (double)s * std::pow((double)D.rope_theta, -2.0 * i / c->hd);
          cs[((size_t)s * half + i) * 2] = (float)std::cos(ang);
          cs[((size_t)s * half + i) * 2 + 1] = (float)std::sin(ang);
        }
      c->rope_cs = (float*)salloc(c, cs.size() * 4);
      CK(cudaMemcpy(c->rope_cs, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice));
    }

    // chunks
    const int d = c->d;
    c->ch.resize(K + 1);
    for (int k = 1; k <= K; ++k) {
      Chunk& ck = c->ch[k];
      ck.k = k;
      ck.l0 = bounds[k - 1];
      ck.l1 = bounds[k];
      // Full fine-tune: every layer tensor in the trainable slab. LoRA: the base matrices and the
      // vectors are frozen and only the factors A [r, in], B [out, r] of the four linears train.
      const int r = cfg->lora_rank;
      // Trainable slab layout: every layer's vectors (norm gains, biases), then the readout adapter, then
      // every layer's matrices (or LoRA factors). The gradient accumulator may stop after the adapter: with
      // the fused update the matrices never need one.
      size_t off = 0, fvec = 0, fmat = 0;
      const bool is_mat[P_COUNT] = {false, false, true, false, true, false, false, false, true, false, true, false};
      for (int l = ck.l0; l < ck.l1; ++l) {
        Layer L;
        for (int p = 0; p < P_COUNT; ++p) { L.blk[p] = false; L.rows[p] = L.cols[p] = 0; }
        size_t shp[P_COUNT] = {(size_t)d, (size_t)d, (size_t)c->qkvw * d, (size_t)c->qkvw, (size_t)d * c->ad, (size_t)d,
                               (size_t)d, (size_t)d, (size_t)c->f1 * d, (size_t)c->f, (size_t)d * c->f, (size_t)d};
        for (int p = 0; p < P_COUNT; ++p) {
          const bool bias = (p == P_N1B || p == P_BQKV || p == P_BO || p == P_N2B || p == P_B1 || p == P_B2);
          L.has[p] = !(c->llama && bias);
          L.numel[p] = L.has[p] ? shp[p] : 0;
          L.slab[p] = r == 0 ? S_TRAIN : (is_mat[p] ? S_FMAT : S_FVEC);
          L.off[p] = 0;
          if (L.slab[p] == S_TRAIN && is_mat[p]) continue;   // second pass
          size_t& cur = L.slab[p] == S_TRAIN ? off : (L.slab[p] == S_FMAT ? fmat : fvec);
          L.off[p] = cur;
          if (L.has[p]) cur += round_up(shp[p], 64);
        }
        ck.layers.push_back(L);
      }
      ck.ad_down = ck.ad_up = off;
      if (cfg->adapter_dim > 0) {
        const size_t ra = (size_t)cfg->adapter_dim;
        ck.ad_down = off;
        off += round_up(ra * d, 64);
        ck.ad_up = off;
        off += round_up((size_t)d * ra, 64);
      }
      ck.ad_end = off;
      for (Layer& L : ck.layers) {
        for (int p = 0; p < P_COUNT; ++p)
          if (L.has[p] && L.slab[p] == S_TRAIN && is_mat[p]) {
            L.off[p] = off;
            off += round_up(L.numel[p], 64);
          }
        // LoRA factors are stored with the rank padded to a multiple of 16 (rows beyond r stay exactly
        // zero: zero start, zero gradient), A as [r16, in] and B transposed as [r16, out], so every
        // LoRA product is a tensor-core GEMM.
        const int ins[4] = {d, c->ad, d, c->f}, outs[4] = {c->qkvw, d, c->f1, d};
        const size_t r16 = (size_t)lora_r16(r);
        for (int i = 0; i < 4; ++i) {
          L.lin_in[i] = ins[i];
          L.lin_out[i] = outs[i];
          L.rows[kLoraP[i]] = outs[i];
          L.cols[kLoraP[i]] = ins[i];
          L.la[i] = L.lb[i] = 0;
          if (r > 0) {
            L.la[i] = off;
            off += round_up(r16 * ins[i], 64);
            L.lb[i] = off;
            off += round_up(r16 * outs[i], 64);
          }
        }
      }
      ck.n = std::max<size_t>(off, 64);
      ck.fvec_n = fvec;
      ck.fmat_n = fmat;
      if (fvec) {
        ck.fvec = (float*)salloc(c, fvec * 4);
        CK(cudaMemset(ck.fvec, 0, fvec * 4));
      }
      if (fmat) {
        ck.fmat = salloc(c, fmat * esz(c));
        CK(cudaMemset(ck.fmat, 0, fmat * esz(c)));
      }
      ck.d_t = (long long*)salloc(c, 64);
      ck.d_hp = (float*)(ck.d_t + 1);
      CK(cudaMemset(ck.d_t, 0, 64));
      // the trainable ranges a fused backward leaves to the range update: every vector of the layers,
      // then the readout adapter (lengths rounded up to 4 inside the slab's 64-element padding)
      if (r == 0) {
        for (const Layer& L : ck.layers)
          for (int p = 0; p < P_COUNT; ++p)
            if (L.has[p] && L.slab[p] == S_TRAIN && p != P_WQKV && p != P_WO && p != P_W1 && p != P_W2) {
              ck.h_ranges.push_back((long long)L.off[p]);
              ck.h_ranges.push_back((long long)round_up(L.numel[p], 4));
            }
        ck.n_ranges_layers = (int)ck.h_ranges.size() / 2;
        if (cfg->adapter_dim > 0)
          for (size_t o : {ck.ad_down, ck.ad_up}) {
            ck.h_ranges.push_back((long long)o);
            ck.h_ranges.push_back((long long)round_up((size_t)cfg->adapter_dim * d, 4));
          }
        ck.n_ranges = (int)ck.h_ranges.size() / 2;
        for (int i = 0; i < ck.n_ranges; ++i) ck.max_range = std::max(ck.max_range, (size_t)ck.h_ranges[2 * i + 1]);
        if (ck.n_ranges > 65535) raise_err(ZL_ERR_UNSUPPORTED, "too many trainable vectors in one chunk");
        if (ck.n_ranges > 0) {
          ck.d_ranges = (long long*)salloc(c, ck.h_ranges.size() * sizeof(long long));
          CK(cudaMemcpy(ck.d_ranges, ck.h_ranges.data(), ck.h_ranges.size() * sizeof(long long),
                        cudaMemcpyHostToDevice));
        }
      }
      // With the fused update always on (bf16 on the tensor cores, one micro-batch per window, full
      // fine-tune) the matrices never hold a gradient: the accumulator covers the vectors and adapter only.
      const bool fused_always = c->dt == BF16 && cfg->accum_m == 1 && !cfg->unfused_update && r == 0 &&
                                gemm_tc_available();
      ck.grad_n = fused_always ? std::max<size_t>(ck.ad_end, 64) : ck.n;
      // ... and, where the shape allows it, their master and moments take the blocked layout the fused
      // update streams fastest (the weight-gradient products are then the only kernels that step them)
      for (Layer& L : ck.layers)
        for (int i = 0; i < 4; ++i) {
          const int p = kLoraP[i];
          L.blk[p] = fused_always && L.has[p] && L.slab[p] == S_TRAIN && L.rows[p] % 16 == 0 && L.cols[p] % 32 == 0;
        }
      ck.master = (float*)salloc(c, ck.n * 4);
      ck.grad = (float*)salloc(c, ck.grad_n * 4);
      ck.m = (float*)salloc(c, ck.n * 4);
      ck.v = (float*)salloc(c, ck.n * 4);
      CK(cudaMemset(ck.master, 0, ck.n * 4));
      CK(cudaMemset(ck.grad, 0, ck.grad_n * 4));
      CK(cudaMemset(ck.m, 0, ck.n * 4));
      CK(cudaMemset(ck.v, 0, ck.n * 4));
      if (c->dt == BF16) {
        ck.comp = salloc(c, ck.n * 2);
        CK(cudaMemset(ck.comp, 0, ck.n * 2));
      }
      // norm gains start at one
      std::vector<float> ones(d, 1.f);
      for (auto& L : ck.layers)
        for (PK p : {P_N1W, P_N2W})
          CK(cudaMemcpy((L.slab[p] == S_FVEC ? ck.fvec : ck.master) + L.off[p], ones.data(), (size_t)d * 4,
                        cudaMemcpyHostToDevice));
      if (c->dt == BF16) launch_f32_to_bf16(ck.master, ck.comp, ck.n, 0);
      if (cfg->serialize && k > 1) ck.s = c->ch[1].s;   // one stream for every chunk
      else CK(cudaStreamCreateWithFlags(&ck.s, cudaStreamNonBlocking));
      if (cfg->serialize) ck.side = ck.s;
      else CK(cudaStreamCreateWithFlags(&ck.side, cudaStreamNonBlocking));
      for (cudaEvent_t* e2 : {&ck.ev_h, &ck.ev_z, &ck.ev_loss, &ck.ev_hb, &ck.ev_done, &ck.ev_sin, &ck.ev_ln2,
                              &ck.ev_layer, &ck.ev_ln1, &ck.ev_send})
        CK(cudaEventCreateWithFlags(e2, cudaEventDisableTiming));
    }
    if (cfg->serialize) c->aux = c->ch[1].s;
    else CK(cudaStreamCreateWithFlags(&c->aux, cudaStreamNonBlocking));
    for (cudaEvent_t* e2 : {&c->ev_start, &c->ev_aux, &c->ev_sync}) CK(cudaEventCreateWithFlags(e2, cudaEventDisableTiming));
    const int cap = cfg->max_live_chunks > 0 ? std::min(cfg->max_live_chunks, K) : K;
    c->live_ring.resize(cap);
    for (auto& e2 : c->live_ring) CK(cudaEventCreateWithFlags(&e2, cudaEventDisableTiming));
    c->d_err = (unsigned*)salloc(c, 4);
    CK(cudaMemset(c->d_err, 0, 4));
    c->d_count = (int*)salloc(c, (size_t)(K + 1) * 4);
    c->d_losses = (float*)salloc(c, (size_t)(K + 1) * 4);
    CK(cudaMemset(c->d_losses, 0, (size_t)(K + 1) * 4));
    CK(cudaMallocHost(&c->h_losses, (size_t)(K + 1) * 4));
    CK(cudaDeviceSynchronize());
    return ZL_OK;
  });
  if (st != ZL_OK) {
    std::string keep = g_err;
    free_ctx(c);
    g_err = keep;
    return st;
  }
  *out = c;
  return ZL_OK;
}

void zl_free(zl_ctx* ctx) { free_ctx(ctx); }

zl_status zl_set_stream(zl_ctx* c, void* stream) {
  if (!c) { g_err = "NULL context"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    c->user = (cudaStream_t)stream;
    return ZL_OK;
  });
}

zl_status zl_param_numel(zl_ctx* c, const char* name, size_t* numel) {
  if (!c || !name || !numel) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  Found f;
  if (!lookup(c, name, f)) { *numel = 0; g_err = std::string("unknown tensor ") + name; return ZL_ERR_ARG; }
  *numel = f.numel;
  return ZL_OK;
}

zl_status zl_set_param(zl_ctx* c, const char* name, const void* src, size_t bytes, int on_device) {
  if (!c || !name || !src) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    Found f;
    if (!lookup(c, name, f)) raise_err(ZL_ERR_ARG, std::string("unknown tensor ") + name);
    if (bytes != f.numel * 4) raise_err(ZL_ERR_ARG, std::string("byte count mismatch for ") + name);
    sync_all(c, -1);
    const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    if (f.trows > 0) {   // user layout [tcols, trows] -> stored [trows, tcols]
      std::vector<float> h(f.numel), t(f.numel);
      CK(cudaMemcpy(h.data(), src, bytes, on_device ? cudaMemcpyDeviceToHost : cudaMemcpyHostToHost));
      for (int o = 0; o < f.tcols; ++o)
        for (int j = 0; j < f.trows; ++j) t[(size_t)j * f.tcols + o] = h[(size_t)o * f.trows + j];
      CK(cudaMemcpy(f.dev, t.data(), bytes, cudaMemcpyHostToDevice));
      if (c->dt == BF16) launch_f32_to_bf16((const float*)f.dev, (bf16*)f.chunk->comp + f.off, f.numel, 0);
    } else if (f.chunk && f.brows > 0) {   // row-major in, blocked master; the compute copy from the row-major
      float* tmp = nullptr;
      CK(cudaMalloc(&tmp, bytes));
      CK(cudaMemcpy(tmp, src, bytes, kind));
      launch_blk_permute(tmp, (float*)f.dev, f.brows, f.bcols, 1, 0);
      if (c->dt == BF16) launch_f32_to_bf16(tmp, (bf16*)f.chunk->comp + f.off, f.numel, 0);
      CK(cudaDeviceSynchronize());
      CK(cudaFree(tmp));
    } else if (f.chunk) {
      CK(cudaMemcpy(f.dev, src, bytes, kind));
      if (c->dt == BF16) launch_f32_to_bf16((const float*)f.dev, (bf16*)f.chunk->comp + f.off, f.numel, 0);
    } else if (f.fp32) {
      CK(cudaMemcpy(f.dev, src, bytes, kind));
    } else {   // frozen tensor held in bf16
      float* tmp = nullptr;
      CK(cudaMalloc(&tmp, bytes));
      CK(cudaMemcpy(tmp, src, bytes, kind));
      launch_f32_to_bf16(tmp, f.dev, f.numel, 0);
      CK(cudaDeviceSynchronize());
      CK(cudaFree(tmp));
    }
    // the LM head copy: lm_head (Llama) or the tied token embedding (GPT-2)
    if ((f.frozen == 5) || (f.frozen == 1 && !c->llama))
      CK(cudaMemcpy(c->lm_head, f.dev, (size_t)c->V * c->d * esz(c), cudaMemcpyDeviceToDevice));
    CK(cudaDeviceSynchronize());
    return ZL_OK;
  });
}

zl_status zl_load_weights(zl_ctx* c, const char* name, const void* src, size_t bytes, int on_device) {
  return zl_set_param(c, name, src, bytes, on_device);
}

zl_status zl_get_param(zl_ctx* c, const char* name, int which, void* dst, size_t bytes, int on_device) {
  if (!c || !name || !dst) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    Found f;
    if (!lookup(c, name, f)) raise_err(ZL_ERR_ARG, std::string("unknown tensor ") + name);
    if (bytes != f.numel * 4) raise_err(ZL_ERR_ARG, std::string("byte count mismatch for ") + name);
    if (which < 0 || which > 3 || (which > 0 && !f.chunk)) raise_err(ZL_ERR_ARG, "which: 0..3, 1..3 trainable only");
    sync_all(c, -1);
    const void* srcp = f.dev;
    if (which == 1 && f.off >= f.chunk->grad_n) {   // a matrix whose gradient is never stored: it is zero
      if (on_device) CK(cudaMemset(dst, 0, bytes));
      else std::memset(dst, 0, bytes);
      return ZL_OK;
    }
    if (which > 0) {
      float* base = which == 1 ? f.chunk->grad : which == 2 ? f.chunk->m : f.chunk->v;
      srcp = base + f.off;
    }
    const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
    if (f.trows > 0) {   // stored [trows, tcols] -> user layout [tcols, trows]
      std::vector<float> h(f.numel), t(f.numel);
      CK(cudaMemcpy(h.data(), srcp, bytes, cudaMemcpyDeviceToHost));
      for (int j = 0; j < f.trows; ++j)
        for (int o = 0; o < f.tcols; ++o) t[(size_t)o * f.trows + j] = h[(size_t)j * f.tcols + o];
      CK(cudaMemcpy(dst, t.data(), bytes, on_device ? cudaMemcpyHostToDevice : cudaMemcpyHostToHost));
    } else if (f.brows > 0) {   // blocked master or moment -> row-major
      float* tmp = nullptr;
      CK(cudaMalloc(&tmp, bytes));
      launch_blk_permute((const float*)srcp, tmp, f.brows, f.bcols, 0, 0);
      CK(cudaDeviceSynchronize());
      CK(cudaMemcpy(dst, tmp, bytes, kind));
      CK(cudaFree(tmp));
    } else if (f.fp32 || which > 0) {
      CK(cudaMemcpy(dst, srcp, bytes, kind));
    } else {
      std::vector<uint16_t> h(f.numel);
      CK(cudaMemcpy(h.data(), srcp, f.numel * 2, cudaMemcpyDeviceToHost));
      std::vector<float> o(f.numel);
      for (size_t i = 0; i < f.numel; ++i) {
        uint32_t u = (uint32_t)h[i] << 16;
        std::memcpy(&o[i], &u, 4);
      }
      CK(cudaMemcpy(dst, o.data(), bytes, on_device ? cudaMemcpyHostToDevice : cudaMemcpyHostToHost));
    }
    return ZL_OK;
  });
}

zl_status zl_embed(zl_ctx* c, const int32_t* ids, int B, int S, void* h0_out) {
  if (!c || !ids || !h0_out) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    check_bs(c, B, S);
    cudaStream_t s = c->ch[1].s;
    start_on(c, s);
    launch_embed(c->dt, ids, c->tok_emb, c->pos_emb, h0_out, B * S, S, c->d, c->V, c->d_err, s);
    CHECK_LAUNCH();
    return ZL_OK;
  });
}

zl_status zl_forward_chunk(zl_ctx* c, int k, const void* h_in, const int32_t* ids, void* h_out, int B, int S) {
  if (!c || !h_out) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    check_bs(c, B, S);
    if (k < 1 || k > c->K) raise_err(ZL_ERR_ARG, "chunk index out of [1, K]");
    if (!h_in && (k != 1 || !ids)) raise_err(ZL_ERR_ARG, "h_in may be NULL only for k = 1 with ids");
    Chunk& ck = c->ch[k];
    cudaStream_t s = ck.s;
    start_on(c, s);
    const int N = B * S;
    void* h0 = nullptr;
    if (!h_in) {
      h0 = palloc(c, (size_t)N * c->d * esz(c), s);
      launch_embed(c->dt, ids, c->tok_emb, c->pos_emb, h0, N, S, c->d, c->V, c->d_err, s);
      h_in = h0;
    }
    chunk_fwd_nosave(c, ck, h_in, h_out, B, S, s);
    pfree(h0, s);
    return ZL_OK;
  });
}

// Steps S1-S3 of Section III-B for chunk k on one micro-batch, queued on the chunk's stream.
void local_step_impl(zl_ctx* c, int k, const void* h_in, const int32_t* ids, const int32_t* labels, int B, int S,
                     void* h_out) {
  Chunk& ck = c->ch[k];
  cudaStream_t s = ck.s;
  const int N = B * S;
  const size_t hb = (size_t)N * c->d * esz(c), zb = (size_t)N * c->Vp * esz(c);
  NvtxPhases ph(c);
  ph.next("zl chunk %d forward", k);
  void* h0 = nullptr;
  if (!h_in) {
    h0 = palloc(c, hb, s);
    launch_embed(c->dt, ids, c->tok_emb, c->pos_emb, h0, N, S, c->d, c->V, c->d_err, s);
    h_in = h0;
  }
  const float a = alpha_of(c, k);
  const bool sliced = c->cfg.loss_rows > 0;
  void* t = nullptr;
  if (a < 1.f && !sliced) {   // teacher p_{k-1} = readout(h_{k-1}), recomputed from the detached input
    t = palloc(c, zb, s);
    readout_fwd(c, h_in, t, nullptr, N, s);
  }
  void* hk = palloc(c, hb, s);
  ChunkActs acts;
  chunk_fwd_save(c, ck, h_in, hk, B, S, acts, s);
  if (h_out) CK(cudaMemcpyAsync(h_out, hk, hb, cudaMemcpyDeviceToDevice, s));
  void* dh = palloc(c, hb, s);
  if (sliced) {
    ph.next("zl chunk %d readout, loss and head backward", k);
    readout_loss_sliced(c, hk, h_in, labels, a, N, k, dh, true, s);
    ph.next("zl chunk %d backward", k);
  } else {
    ph.next("zl chunk %d readout", k);
    void* z = palloc(c, zb, s);
    ReadoutSave rs;
    Chunk* ad = c->cfg.adapter_dim > 0 ? &ck : nullptr;
    readout_fwd(c, hk, z, &rs, N, s, ad);
    ph.next("zl chunk %d loss", k);
    void* dz = local_loss(c, z, t, labels, a, N, k, s);
    pfree(z, s);
    pfree(t, s);
    ph.next("zl chunk %d backward", k);
    readout_bwd(c, hk, rs, dz, dh, N, s, ad);
    pfree(dz, s);
  }
  window_begin(c, ck, s);
  chunk_bwd(c, ck, acts, dh, nullptr, B, S, s);
  pfree(dh, s);
  pfree(acts.mem, s);
  pfree(hk, s);
  pfree(h0, s);
  ph.next("zl chunk %d adamw", k);
  adamw_window(c, ck, s);
  ph.end();
  ck.done += 1;
}

zl_status zl_local_step(zl_ctx* c, int k, const void* h_in, const int32_t* ids, const int32_t* labels, int B, int S,
                        void* h_out, float* loss_out) {
  if (!c || !labels) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    check_bs(c, B, S);
    if (k < 1 || k > c->K) raise_err(ZL_ERR_ARG, "chunk index out of [1, K]");
    if (!h_in && (k != 1 || !ids)) raise_err(ZL_ERR_ARG, "h_in may be NULL only for k = 1 with ids");
    start_on(c, c->ch[k].s);
    local_step_impl(c, k, h_in, ids, labels, B, S, h_out);
    if (loss_out) {
      CK(cudaMemcpyAsync(c->h_losses + k, c->d_losses + k, 4, cudaMemcpyDeviceToHost, c->ch[k].s));
      sync_all(c, -1);
      *loss_out = c->h_losses[k];
    }
    return ZL_OK;
  });
}

// Catch chunk k up to the pipeline frontier from its hidden-state buffer (reactive recovery,
// Section III-B-3): re-runs its local steps for every buffered micro-batch after its progress.
zl_status zl_replay(zl_ctx* c, int k, int* replayed, float* loss_out) {
  if (!c) { g_err = "NULL context"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    if (k < 1 || k > c->K) raise_err(ZL_ERR_ARG, "chunk index out of [1, K]");
    Chunk& ck = c->ch[k];
    const int D = c->cfg.replay_depth;
    if (ck.done > c->seq) raise_err(ZL_ERR_STATE, "chunk progress is ahead of the pipeline frontier");
    if (ck.done < c->seq && (D <= 0 || c->seq - ck.done > D))
      raise_err(ZL_ERR_ARG, "the micro-batches to replay are no longer in the hidden-state buffer");
    start_on(c, ck.s);
    int n = 0;
    for (long q = ck.done; q < c->seq; ++q) {
      Chunk::Entry& e = ck.ring[q % D];
      if (e.seq != q) raise_err(ZL_ERR_ARG, "hidden-state buffer entry missing");
      local_step_impl(c, k, e.h, nullptr, e.labels, e.B, e.S, nullptr);
      ++n;
    }
    if (replayed) *replayed = n;
    if (loss_out && n > 0) {
      CK(cudaMemcpyAsync(c->h_losses + k, c->d_losses + k, 4, cudaMemcpyDeviceToHost, ck.s));
      sync_all(c, -1);
      *loss_out = c->h_losses[k];
    }
    return ZL_OK;
  });
}

// Per-chunk checkpoint (proactive checkpointing, Section III-B-3): header, then the trainable
// slab's fp32 master, gradient accumulator and AdamW moments.
struct CkptHeader {
  uint64_t magic;
  int32_t k, l0, l1, lora_rank;
  int64_t n, t, done;
  int32_t micro, dtype;
};
constexpr uint64_t kCkptMagic = 0x31304B434C5A4C5AULL;   // "ZLZLCK01"

bool has_blocked(const Chunk& ck) {
  for (const Layer& L : ck.layers)
    for (int p = 0; p < P_COUNT; ++p)
      if (L.blk[p]) return true;
  return false;
}
// Copies one slab-sized fp32 array (n floats) between device buffers, turning every blocked matrix into
// row-major (to_blk = 0) or back (1), so checkpoints hold the same row-major layout whatever the engine's.
void slab_xfer(Chunk& ck, const float* src, float* dst, int to_blk) {
  CK(cudaMemcpy(dst, src, ck.n * sizeof(float), cudaMemcpyDeviceToDevice));
  for (const Layer& L : ck.layers)
    for (int p = 0; p < P_COUNT; ++p)
      if (L.blk[p]) launch_blk_permute(src + L.off[p], dst + L.off[p], L.rows[p], L.cols[p], to_blk, 0);
  CK(cudaDeviceSynchronize());
}

zl_status zl_chunk_state_bytes(zl_ctx* c, int k, size_t* bytes) {
  if (!c || !bytes) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if (k < 1 || k > c->K) { g_err = "chunk index out of [1, K]"; return ZL_ERR_ARG; }
  *bytes = sizeof(CkptHeader) + 4 * c->ch[k].n * sizeof(float);
  return ZL_OK;
}

zl_status zl_chunk_save(zl_ctx* c, int k, void* dst, size_t bytes) {
  if (!c || !dst) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    if (k < 1 || k > c->K) raise_err(ZL_ERR_ARG, "chunk index out of [1, K]");
    Chunk& ck = c->ch[k];
    if (bytes != sizeof(CkptHeader) + 4 * ck.n * sizeof(float)) raise_err(ZL_ERR_ARG, "checkpoint size mismatch");
    sync_all(c, -1);
    CkptHeader h{kCkptMagic, k, ck.l0, ck.l1, c->cfg.lora_rank, (int64_t)ck.n, ck.t, ck.done, ck.micro, c->dt};
    std::memcpy(dst, &h, sizeof h);
    float* p = reinterpret_cast<float*>(static_cast<char*>(dst) + sizeof h);
    const size_t sz = ck.n * sizeof(float);
    float* tmp = nullptr;
    if (has_blocked(ck)) CK(cudaMalloc(&tmp, sz));
    auto out = [&](const float* a, float* h) {   // row-major copy of a slab array to the host
      if (tmp) slab_xfer(ck, a, tmp, 0);
      CK(cudaMemcpy(h, tmp ? tmp : a, sz, cudaMemcpyDeviceToHost));
    };
    out(ck.master, p);
    CK(cudaMemcpy(p + ck.n, ck.grad, ck.grad_n * sizeof(float), cudaMemcpyDeviceToHost));
    std::memset(p + ck.n + ck.grad_n, 0, (ck.n - ck.grad_n) * sizeof(float));   // unstored gradients are zero
    out(ck.m, p + 2 * ck.n);
    out(ck.v, p + 3 * ck.n);
    if (tmp) CK(cudaFree(tmp));
    return ZL_OK;
  });
}

zl_status zl_chunk_load(zl_ctx* c, int k, const void* src, size_t bytes) {
  if (!c || !src) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    if (k < 1 || k > c->K) raise_err(ZL_ERR_ARG, "chunk index out of [1, K]");
    Chunk& ck = c->ch[k];
    if (bytes != sizeof(CkptHeader) + 4 * ck.n * sizeof(float)) raise_err(ZL_ERR_ARG, "checkpoint size mismatch");
    CkptHeader h;
    std::memcpy(&h, src, sizeof h);
    if (h.magic != kCkptMagic || h.k != k || h.l0 != ck.l0 || h.l1 != ck.l1 || h.lora_rank != c->cfg.lora_rank ||
        h.n != (int64_t)ck.n || h.dtype != c->dt)
      raise_err(ZL_ERR_ARG, "checkpoint does not belong to this chunk");
    sync_all(c, -1);
    const float* p = reinterpret_cast<const float*>(static_cast<const char*>(src) + sizeof h);
    const size_t sz = ck.n * sizeof(float);
    if (has_blocked(ck)) {   // the blob is row-major: through a device copy into the blocked layout
      float* tmp = nullptr;
      CK(cudaMalloc(&tmp, sz));
      CK(cudaMemcpy(tmp, p, sz, cudaMemcpyHostToDevice));
      slab_xfer(ck, tmp, ck.master, 1);
      if (c->dt == BF16) launch_f32_to_bf16(tmp, ck.comp, ck.n, 0);
      CK(cudaMemcpy(tmp, p + 2 * ck.n, sz, cudaMemcpyHostToDevice));
      slab_xfer(ck, tmp, ck.m, 1);
      CK(cudaMemcpy(tmp, p + 3 * ck.n, sz, cudaMemcpyHostToDevice));
      slab_xfer(ck, tmp, ck.v, 1);
      CK(cudaFree(tmp));
    } else {
      CK(cudaMemcpy(ck.master, p, sz, cudaMemcpyHostToDevice));
      CK(cudaMemcpy(ck.m, p + 2 * ck.n, sz, cudaMemcpyHostToDevice));
      CK(cudaMemcpy(ck.v, p + 3 * ck.n, sz, cudaMemcpyHostToDevice));
      if (c->dt == BF16) launch_f32_to_bf16(ck.master, ck.comp, ck.n, 0);
    }
    CK(cudaMemcpy(ck.grad, p + ck.n, ck.grad_n * sizeof(float), cudaMemcpyHostToDevice));
    CK(cudaDeviceSynchronize());
    ck.t = h.t;
    const long long tt = h.t;
    CK(cudaMemcpy(ck.d_t, &tt, sizeof(tt), cudaMemcpyHostToDevice));
    ck.done = h.done;
    ck.micro = h.micro;
    return ZL_OK;
  });
}

// The concurrent ZeroLock step: chunk k runs on stream s_k; its forward waits only for the
// readiness event of h_{k-1} (early forwarding), its loss waits for the teacher logits z_{k-1},
// and at most `cap` chunks hold activation arenas at once.
}  // extern "C"

namespace {

// CUDA graphs (cfg.graph): a step is captured once per micro-batch shape and replayed. The first call
// at a shape runs eagerly (it also performs the one-time set-up some launches do); the inputs are
// staged into context-owned buffers that the graph reads. Graphs are used only where a step's work
// is the same every time: no profiling, one micro-batch per window, no replay buffer.
bool graph_ok(zl_ctx* c) {
  return c->cfg.graph != 0 && !c->prof && c->cfg.accum_m == 1 && c->cfg.replay_depth == 0;
}

template <typename E, typename A>
bool run_graph(zl_ctx* c, zl_ctx::StepGraph& g, const int32_t* ids, const int32_t* labels, int B, int S, E&& enqueue,
               A&& advance) {
  if (!graph_ok(c)) return false;
  const size_t N = (size_t)B * S;
  if (g.B != B || g.S != S) {
    if (g.exec) {
      sync_all(c, -1);
      CK(cudaGraphExecDestroy(g.exec));
      g.exec = nullptr;
    }
    g.B = B;
    g.S = S;
    g.seen = 0;
  }
  if (g.seen++ < 1) return false;
  if (g.cap < N) {   // (re)allocate the staging buffers, outside any capture
    sync_all(c, -1);
    if (g.ids) CK(cudaFree(g.ids));
    if (g.labels) CK(cudaFree(g.labels));
    g.ids = g.labels = nullptr;
    g.cap = 0;
    CK(cudaMalloc((void**)&g.ids, N * 4));
    CK(cudaMalloc((void**)&g.labels, N * 4));
    g.cap = N;
  }
  CK(cudaMemcpyAsync(g.ids, ids, N * 4, cudaMemcpyDeviceToDevice, c->user));
  CK(cudaMemcpyAsync(g.labels, labels, N * 4, cudaMemcpyDeviceToDevice, c->user));
  join_all(c);   // every stream's earlier work before the graph
  if (!g.exec) {
    // capture on a stream of the context, standing in for the user's stream
    if (!c->cap) CK(cudaStreamCreateWithFlags(&c->cap, cudaStreamNonBlocking));
    const cudaStream_t user = c->user;
    CK(cudaStreamBeginCapture(c->cap, cudaStreamCaptureModeThreadLocal));
    c->capturing = true;
    c->user = c->cap;
    const unsigned long long n0 = g_launches.load();
    try {
      enqueue(g.ids, g.labels);
      join_all(c);
      g.launches = g_launches.load() - n0;
    } catch (...) {
      c->capturing = false;
      c->user = user;
      cudaGraph_t junk = nullptr;
      cudaStreamEndCapture(c->cap, &junk);
      if (junk) cudaGraphDestroy(junk);
      cudaGetLastError();
      throw;
    }
    c->capturing = false;
    c->user = user;
    cudaGraph_t graph = nullptr;
    CK(cudaStreamEndCapture(c->cap, &graph));
    const cudaError_t e = cudaGraphInstantiate(&g.exec, graph, 0);
    cudaGraphDestroy(graph);
    CK(e);
  } else {
    advance();
    note_launch((int)g.launches);   // the replay runs the same kernels
  }
  CK(cudaGraphLaunch(g.exec, c->user));
  // The context's events were last recorded inside the capture, which does not count as a record
  // outside it: record them all after the graph (a later point than the one they stood for, so every
  // later wait on them stays correct). Later work on the chunk and auxiliary streams (loss read-back,
  // the next eager step) follows the graph.
  for (cudaEvent_t e : c->live_ring) rec(e, c->user);
  for (int k = 1; k <= c->K; ++k)
    for (cudaEvent_t e : {c->ch[k].ev_h, c->ch[k].ev_z, c->ch[k].ev_loss, c->ch[k].ev_hb, c->ch[k].ev_done})
      rec(e, c->user);
  for (cudaEvent_t e : {c->ev_aux, c->ev_sync}) rec(e, c->user);
  rec(c->ev_start, c->user);
  for (int k = 1; k <= c->K; ++k) wait_ev(c->ch[k].s, c->ev_start);
  wait_ev(c->aux, c->ev_start);
  return true;
}

// The work of one zl_step, queued on the chunk streams (eagerly or into a capture).
void step_enqueue(zl_ctx* c, const int32_t* ids, const int32_t* labels, int B, int S) {
  const int N = B * S, K = c->K;
  const size_t hb = (size_t)N * c->d * esz(c), zb = (size_t)N * c->Vp * esz(c);
  rec(c->ev_start, c->user);
  for (int k = 1; k <= K; ++k) wait_ev(c->ch[k].s, c->ev_start);
  wait_ev(c->aux, c->ev_start);
  NvtxPhases ph(c);
  ph.next("zl step embedding and teacher");
  std::vector<void*> h(K + 1, nullptr), z(K + 1, nullptr);
  // h_0 = E(x) on s_1; the teacher of chunk 1, z_0 = readout(h_0), on the auxiliary stream
  cudaStream_t s1 = c->ch[1].s;
  h[0] = palloc(c, hb, s1);
  launch_embed(c->dt, ids, c->tok_emb, c->pos_emb, h[0], N, S, c->d, c->V, c->d_err, s1);
  CHECK_LAUNCH();
  rec(c->ch[1].ev_h, s1);   // reused below as "h_0 ready" before chunk 1 records h_1
  cudaEvent_t ev_h0 = c->ev_aux;
  const float a1 = alpha_of(c, 1);
  const bool sliced = c->cfg.loss_rows > 0;   // each chunk forms its teacher slices from h_{k-1} itself
  if (a1 < 1.f && !sliced) {
    wait_ev(c->aux, c->ch[1].ev_h);
    z[0] = palloc(c, zb, c->aux);
    readout_fwd(c, h[0], z[0], nullptr, N, c->aux);
  }
  rec(ev_h0, c->aux);      // z_0 ready (and aux done reading h_0)
  const int cap = (int)c->live_ring.size();
  const bool adp = c->cfg.adapter_dim > 0;
  for (int k = 1; k <= K; ++k) {
    Chunk& ck = c->ch[k];
    cudaStream_t s = ck.s;
    const float a = alpha_of(c, k);
    ph.next("zl chunk %d forward", k);
    // S1: the upstream entry (h_{k-1}) and a free arena slot
    if (k > 1) wait_ev(s, c->ch[k - 1].ev_h);
    ring_put(c, ck, c->seq, h[k - 1], labels, B, S, s);
    ck.done += 1;
    // a capture sees only this step's events: slots are numbered within the step (graph launches
    // on the user stream already order one step after the previous one)
    const long seq0 = c->live_seq++;
    const long seq = c->capturing ? (long)(k - 1) : seq0;
    if (seq >= cap) wait_ev(s, c->live_ring[seq % cap]);
    // S2: forward, then hand h_k downstream before the local backward (early forwarding)
    h[k] = palloc(c, hb, s);
    ChunkActs acts;
    chunk_fwd_save(c, ck, h[k - 1], h[k], B, S, acts, s);
    rec(ck.ev_h, s);
    void* dh = palloc(c, hb, s);
    if (sliced) {
      // readout, local objective against the frozen head on h_{k-1}, head backward, in row slices
      ph.next("zl chunk %d readout, loss and head backward", k);
      readout_loss_sliced(c, h[k], h[k - 1], labels, a, N, k, dh, true, s);
      rec(ck.ev_z, s);
      rec(ck.ev_loss, s);
      rec(ck.ev_hb, s);
      ph.next("zl chunk %d backward", k);
    } else {
      ph.next("zl chunk %d readout", k);
      z[k] = palloc(c, zb, s);
      ReadoutSave rs;
      readout_fwd(c, h[k], z[k], &rs, N, s, adp ? &ck : nullptr);
      rec(ck.ev_z, s);
      ph.next("zl chunk %d loss", k);
      // S3: local objective against the stop-gradient teacher: the frozen head on h_{k-1}, which is
      // chunk k-1's own readout z_{k-1} (reused) unless chunk k-1 read out through its adapter
      void* teacher = nullptr;
      void* own_t = nullptr;
      if (a < 1.f) {
        if (k == 1) {
          wait_ev(s, ev_h0);
          teacher = z[0];
        } else if (adp) {
          own_t = palloc(c, zb, s);
          readout_fwd(c, h[k - 1], own_t, nullptr, N, s);
          teacher = own_t;
        } else {
          wait_ev(s, c->ch[k - 1].ev_z);
          teacher = z[k - 1];
        }
      }
      void* dz = local_loss(c, z[k], teacher, labels, a, N, k, s);
      rec(ck.ev_loss, s);
      pfree(own_t, s);
      // z_{k-1} is no longer needed once this loss and chunk k-1's own loss are done
      if (k == 1) {
        if (z[0]) { wait_ev(s, ev_h0); pfree(z[0], s); }
      } else if (!adp) {
        wait_ev(s, c->ch[k - 1].ev_loss);
        pfree(z[k - 1], s);
      }
      if (k == K || adp) pfree(z[k], s);   // with adapters no later chunk reads z_k
      ph.next("zl chunk %d backward", k);
      readout_bwd(c, h[k], rs, dz, dh, N, s, adp ? &ck : nullptr);
      pfree(dz, s);
      rec(ck.ev_hb, s);
    }
    window_begin(c, ck, s);
    chunk_bwd(c, ck, acts, dh, nullptr, B, S, s);
    pfree(dh, s);
    pfree(acts.mem, s);
    rec(c->live_ring[seq % cap], s);
    // h_{k-1}: read by this chunk's backward and by chunk k-1's readout backward
    if (k == 1) wait_ev(s, ev_h0);
    else wait_ev(s, c->ch[k - 1].ev_hb);
    pfree(h[k - 1], s);
    if (k == K) pfree(h[K], s);
    ph.next("zl chunk %d adamw", k);
    adamw_window(c, ck, s);
  }
  ph.end();
  c->last_nloss = K;
  c->seq += 1;
}

}  // namespace

extern "C" {

zl_status zl_step(zl_ctx* c, const int32_t* ids, const int32_t* labels, int B, int S, float* losses_out) {
  if (!c || !ids || !labels) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    check_bs(c, B, S);
    const int K = c->K;
    const bool graphed = run_graph(
        c, c->zg, ids, labels, B, S, [&](const int32_t* gi, const int32_t* gl) { step_enqueue(c, gi, gl, B, S); },
        [&]() {   // the host bookkeeping step_enqueue does, for a replay
          for (int k = 1; k <= K; ++k) {
            c->ch[k].done += 1;
            c->ch[k].t += 1;
          }
          c->live_seq += K;
          c->last_nloss = K;
          c->seq += 1;
        });
    if (!graphed) step_enqueue(c, ids, labels, B, S);
    if (losses_out) {
      for (int k = 1; k <= K; ++k)
        CK(cudaMemcpyAsync(c->h_losses + k, c->d_losses + k, 4, cudaMemcpyDeviceToHost, c->ch[k].s));
      sync_all(c, -1);
      for (int k = 1; k <= K; ++k) losses_out[k - 1] = c->h_losses[k];
    }
    return ZL_OK;
  });
}

// Backpropagation through all chunks (the same kernels, one stream, every arena alive until
// the backward reaches it).
}  // extern "C"

namespace {

// The work of one zl_bp_step (eagerly or into a capture).
void bp_enqueue(zl_ctx* c, const int32_t* ids, const int32_t* labels, int B, int S) {
  const int N = B * S, K = c->K;
  const size_t hb = (size_t)N * c->d * esz(c), zb = (size_t)N * c->Vp * esz(c);
  cudaStream_t s = c->ch[1].s;
  rec(c->ev_start, c->user);
  wait_ev(s, c->ev_start);
  wait_ev(c->aux, c->ev_start);    // (keeps every stream of the context in a capture)
  if (!c->capturing)
    for (int k = 2; k <= K; ++k) {   // previous work of the other chunk streams
      rec(c->ch[k].ev_done, c->ch[k].s);
      wait_ev(s, c->ch[k].ev_done);
    }
  NvtxPhases ph(c);
  ph.next("zl bp forward");
  std::vector<void*> h(K + 1, nullptr);
  std::vector<ChunkActs> acts(K + 1);
  h[0] = palloc(c, hb, s);
  launch_embed(c->dt, ids, c->tok_emb, c->pos_emb, h[0], N, S, c->d, c->V, c->d_err, s);
  for (int k = 1; k <= K; ++k) {
    h[k] = palloc(c, hb, s);
    chunk_fwd_save(c, c->ch[k], h[k - 1], h[k], B, S, acts[k], s);
  }
  ph.next("zl bp readout and loss");
  void* dh = palloc(c, hb, s);
  void* dh2 = palloc(c, hb, s);
  if (c->cfg.loss_rows > 0) {
    readout_loss_sliced(c, h[K], nullptr, labels, 1.f, N, 0, dh, true, s);
    ph.next("zl bp backward");
  } else {
    void* z = palloc(c, zb, s);
    ReadoutSave rs;
    readout_fwd(c, h[K], z, &rs, N, s);
    void* dz = local_loss(c, z, nullptr, labels, 1.f, N, 0, s);
    pfree(z, s);
    ph.next("zl bp backward");
    readout_bwd(c, h[K], rs, dz, dh, N, s);
    pfree(dz, s);
  }
  for (int k = K; k >= 1; --k) {
    window_begin(c, c->ch[k], s);
    chunk_bwd(c, c->ch[k], acts[k], dh, k > 1 ? dh2 : nullptr, B, S, s);
    std::swap(dh, dh2);
    pfree(acts[k].mem, s);
    pfree(h[k], s);
  }
  pfree(h[0], s);
  pfree(dh, s);
  pfree(dh2, s);
  ph.next("zl bp adamw");
  for (int k = 1; k <= K; ++k) {
    if (k > 1) {   // the optimizer step of chunk k stays on its own stream
      rec(c->ch[1].ev_done, s);
      wait_ev(c->ch[k].s, c->ch[1].ev_done);
    }
    adamw_window(c, c->ch[k], k == 1 ? s : c->ch[k].s, false);
  }
  c->last_nloss = 1;
  for (int k = 1; k <= K; ++k) c->ch[k].done += 1;
}

}  // namespace

extern "C" {

zl_status zl_bp_step(zl_ctx* c, const int32_t* ids, const int32_t* labels, int B, int S, float* loss_out) {
  if (!c || !ids || !labels) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    check_bs(c, B, S);
    const int K = c->K;
    const bool graphed = run_graph(
        c, c->bg, ids, labels, B, S, [&](const int32_t* gi, const int32_t* gl) { bp_enqueue(c, gi, gl, B, S); },
        [&]() {
          for (int k = 1; k <= K; ++k) {
            c->ch[k].done += 1;
            c->ch[k].t += 1;
          }
          c->last_nloss = 1;
        });
    if (!graphed) bp_enqueue(c, ids, labels, B, S);
    const cudaStream_t s = c->ch[1].s;
    if (loss_out) {
      CK(cudaMemcpyAsync(c->h_losses, c->d_losses, 4, cudaMemcpyDeviceToHost, s));
      sync_all(c, -1);
      *loss_out = c->h_losses[0];
    }
    return ZL_OK;
  });
}

zl_status zl_eval_global_loss(zl_ctx* c, const int32_t* ids, const int32_t* labels, int B, int S, float* loss_out) {
  if (!c || !ids || !labels || !loss_out) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    check_bs(c, B, S);
    const int N = B * S, K = c->K;
    const size_t hb = (size_t)N * c->d * esz(c), zb = (size_t)N * c->Vp * esz(c);
    cudaStream_t s = c->aux;
    rec(c->ev_start, c->user);
    wait_ev(s, c->ev_start);
    for (int k = 1; k <= K; ++k) {
      rec(c->ch[k].ev_done, c->ch[k].s);
      wait_ev(s, c->ch[k].ev_done);
    }
    void* a = palloc(c, hb, s);
    void* b = palloc(c, hb, s);
    launch_embed(c->dt, ids, c->tok_emb, c->pos_emb, a, N, S, c->d, c->V, c->d_err, s);
    for (int k = 1; k <= K; ++k) {
      chunk_fwd_nosave(c, c->ch[k], a, b, B, S, s);
      std::swap(a, b);
    }
    if (c->cfg.loss_rows > 0) {
      readout_loss_sliced(c, a, nullptr, labels, 1.f, N, 0, nullptr, false, s);
    } else {
      void* z = palloc(c, zb, s);
      readout_fwd(c, a, z, nullptr, N, s);
      void* dz = local_loss(c, z, nullptr, labels, 1.f, N, 0, s);
      pfree(dz, s);
      pfree(z, s);
    }
    pfree(a, s);
    pfree(b, s);
    CK(cudaMemcpyAsync(c->h_losses, c->d_losses, 4, cudaMemcpyDeviceToHost, s));
    sync_all(c, -1);
    *loss_out = c->h_losses[0];
    return ZL_OK;
  });
}

zl_status zl_read_losses(zl_ctx* c, float* out, int n) {
  if (!c || !out) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    if (n != c->last_nloss) raise_err(ZL_ERR_ARG, "n must be K after zl_step, 1 after zl_bp_step");
    sync_all(c, -1);
    CK(cudaMemcpy(out, c->d_losses + (c->last_nloss == 1 ? 0 : 1), (size_t)n * 4, cudaMemcpyDeviceToHost));
    return ZL_OK;
  });
}

zl_status zl_join(zl_ctx* c) {
  if (!c) { g_err = "NULL context"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    join_all(c);
    return ZL_OK;
  });
}

zl_status zl_synchronize(zl_ctx* c, int timeout_ms) {
  if (!c) { g_err = "NULL context"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status { return sync_all(c, timeout_ms); });
}

zl_status zl_peak_bytes(zl_ctx* c, size_t* peak, size_t* current) {
  if (!c) { g_err = "NULL context"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    uint64_t hi = 0, cur = 0;
    CK(cudaMemPoolGetAttribute(c->pool, cudaMemPoolAttrUsedMemHigh, &hi));
    CK(cudaMemPoolGetAttribute(c->pool, cudaMemPoolAttrUsedMemCurrent, &cur));
    if (c->cfg.graph) {   // a captured step's activations live in the device's graph memory
      int dev = 0;
      uint64_t ghi = 0, gcur = 0;
      CK(cudaGetDevice(&dev));
      CK(cudaDeviceGetGraphMemAttribute(dev, cudaGraphMemAttrUsedMemHigh, &ghi));
      CK(cudaDeviceGetGraphMemAttribute(dev, cudaGraphMemAttrUsedMemCurrent, &gcur));
      hi += ghi;
      cur += gcur;
    }
    if (peak) *peak = c->static_bytes + hi;
    if (current) *current = c->static_bytes + cur;
    return ZL_OK;
  });
}

zl_status zl_reset_peak(zl_ctx* c) {
  if (!c) { g_err = "NULL context"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    sync_all(c, -1);
    uint64_t zero = 0;
    CK(cudaMemPoolSetAttribute(c->pool, cudaMemPoolAttrUsedMemHigh, &zero));
    if (c->cfg.graph) {
      int dev = 0;
      CK(cudaGetDevice(&dev));
      CK(cudaDeviceSetGraphMemAttribute(dev, cudaGraphMemAttrUsedMemHigh, &zero));
    }
    return ZL_OK;
  });
}

zl_status zl_profile(zl_ctx* c, int on) {
  if (!c) { g_err = "NULL context"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    if (on && c->evpool.size() < 8192) {
      while (c->evpool.size() < 8192) {
        cudaEvent_t e;
        CK(cudaEventCreate(&e));
        c->evpool.push_back(e);
      }
    }
    c->prof = on != 0;
    return ZL_OK;
  });
}

zl_status zl_profile_read(zl_ctx* c, char* buf, size_t cap) {
  if (!c || !buf || cap == 0) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  return guarded(c, [&]() -> zl_status {
    sync_all(c, -1);
    double ms[PC_COUNT] = {}, fl[PC_COUNT] = {}, by[PC_COUNT] = {}, nl[PC_COUNT] = {};
    for (const ProfRec& r : c->recs) {
      float t = 0.f;
      CK(cudaEventElapsedTime(&t, r.a, r.b));
      ms[r.cls] += t;
      fl[r.cls] += r.flops;
      by[r.cls] += r.bytes;
      nl[r.cls] += r.launches;
    }
    c->recs.clear();
    c->evnext = 0;
    std::string js = "{";
    for (int i = 0; i < PC_COUNT; ++i) {
      char tmp[256];
      std::snprintf(tmp, sizeof tmp, "%s\"%s\": {\"launches\": %.0f, \"ms\": %.6f, \"flops\": %.6e, \"bytes\": %.6e}",
                    i ? ", " : "", kPCName[i], nl[i], ms[i], fl[i], by[i]);
      js += tmp;
    }
    js += "}";
    std::snprintf(buf, cap, "%s", js.c_str());
    return ZL_OK;
  });
}

zl_status zl_kernel_launches(uint64_t* count) {
  if (!count) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  *count = (uint64_t)launches_so_far();
  return ZL_OK;
}

zl_status zl_op_local_loss(int dtype, const void* z, const void* t, const int32_t* labels, int N, int V, int ldz,
                           float alpha, int kl_dir, void* dz, float* row_loss, float* loss, void* stream) {
  if (!z || !labels || !dz || !row_loss || !loss) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if (dtype != 0 && dtype != 1) { g_err = "dtype"; return ZL_ERR_ARG; }
  if (N < 1 || V < 2 || ldz < V || ldz % 8 != 0) { g_err = "need N >= 1, V >= 2, ldz >= V, ldz % 8 == 0"; return ZL_ERR_ARG; }
  if (N > (1 << 24)) { g_err = "N above 2^24 rows (|Omega| is counted exactly up to 2^24)"; return ZL_ERR_ARG; }
  if (!(alpha > 0.f && alpha <= 1.f) || (alpha < 1.f && !t) || (kl_dir != 0 && kl_dir != 1)) {
    g_err = "alpha in (0,1], t required when alpha < 1, kl_dir 0/1";
    return ZL_ERR_ARG;
  }
  return guarded(nullptr, [&]() -> zl_status {
    cudaStream_t s = (cudaStream_t)stream;
    int* cnt = nullptr;
    unsigned* err = nullptr;
    CK(cudaMallocAsync((void**)&cnt, 256, s));
    err = (unsigned*)((char*)cnt + 128);
    CK(cudaMemsetAsync(err, 0, 4, s));
    launch_count_valid(labels, N, V, cnt, err, s);
    launch_local_loss(dtype, z, t, labels, N, V, ldz, alpha, kl_dir, cnt, dz, row_loss, s);
    launch_loss_reduce(row_loss, N, cnt, loss, s);
    CHECK_LAUNCH();
    CK(cudaFreeAsync(cnt, s));
    return ZL_OK;
  });
}

zl_status zl_op_head_loss(int dtype, const void* n, const void* tn, const void* W, const int32_t* labels, int N, int d,
                          int V, int ldw, float alpha, int kl_dir, int rows_per_slice, void* dn, float* row_loss,
                          float* loss, void* stream) {
  if (!n || !W || !labels || !dn || !row_loss || !loss) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if (dtype != 0 && dtype != 1) { g_err = "dtype"; return ZL_ERR_ARG; }
  if (N < 1 || d < 8 || d % 8 != 0 || V < 2 || ldw < V || ldw % 8 != 0 || rows_per_slice < 1) {
    g_err = "need N >= 1, d >= 8 with d % 8 == 0, V >= 2, ldw >= V with ldw % 8 == 0, rows_per_slice >= 1";
    return ZL_ERR_ARG;
  }
  if (N > (1 << 24)) { g_err = "N above 2^24 rows (|Omega| is counted exactly up to 2^24)"; return ZL_ERR_ARG; }
  if (!(alpha > 0.f && alpha <= 1.f) || (alpha < 1.f && !tn) || (kl_dir != 0 && kl_dir != 1)) {
    g_err = "alpha in (0,1], tn required when alpha < 1, kl_dir 0/1";
    return ZL_ERR_ARG;
  }
  return guarded(nullptr, [&]() -> zl_status {
    cudaStream_t s = (cudaStream_t)stream;
    const int R = std::min(N, rows_per_slice);
    const size_t zb = (size_t)R * ldw * dt_size(dtype);
    int* cnt = nullptr;
    void *z = nullptr, *t = nullptr;
    CK(cudaMallocAsync((void**)&cnt, 256, s));
    CK(cudaMallocAsync(&z, zb, s));
    if (alpha < 1.f) CK(cudaMallocAsync(&t, zb, s));
    unsigned* err = (unsigned*)((char*)cnt + 128);
    CK(cudaMemsetAsync(err, 0, 4, s));
    launch_count_valid(labels, N, V, cnt, err, s);
    head_loss_rows(nullptr, dtype, n, alpha < 1.f ? tn : nullptr, W, labels, N, d, V, ldw, alpha, kl_dir, R, cnt, dn,
                   row_loss, z, t, true, s, nullptr, nullptr);
    launch_loss_reduce(row_loss, N, cnt, loss, s);
    CHECK_LAUNCH();
    CK(cudaFreeAsync(z, s));
    if (t) CK(cudaFreeAsync(t, s));
    CK(cudaFreeAsync(cnt, s));
    return ZL_OK;
  });
}

static bool attn_args_ok(int dtype, int B, int S, int H, int Hkv, int hd) {
  return (dtype == 0 || dtype == 1) && B >= 1 && B <= 65535 && S >= 1 && (long)B * S <= (1L << 26) && H >= 1 &&
         Hkv >= 1 && H % Hkv == 0 && hd >= 2 && hd <= 128 && hd % 2 == 0;
}

zl_status zl_op_attention(int dtype, const void* qkv, void* out, float* lse, int B, int S, int H, int Hkv, int hd,
                          void* stream) {
  if (!qkv || !out || !lse) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if (!attn_args_ok(dtype, B, S, H, Hkv, hd)) { g_err = "bad attention shape"; return ZL_ERR_ARG; }
  return guarded(nullptr, [&]() -> zl_status {
    attn_fwd(dtype, qkv, out, lse, B, S, H, Hkv, hd, (cudaStream_t)stream);
    CHECK_LAUNCH();
    return ZL_OK;
  });
}

zl_status zl_op_attention_bwd(int dtype, const void* qkv, const void* out, const void* dout, const float* lse,
                              void* dqkv, int B, int S, int H, int Hkv, int hd, void* stream) {
  if (!qkv || !out || !dout || !lse || !dqkv) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if (!attn_args_ok(dtype, B, S, H, Hkv, hd)) { g_err = "bad attention shape"; return ZL_ERR_ARG; }
  return guarded(nullptr, [&]() -> zl_status {
    cudaStream_t s = (cudaStream_t)stream;
    float* D = nullptr;
    CK(cudaMallocAsync((void**)&D, (size_t)B * H * S * 4, s));
    attn_bwd(dtype, qkv, out, dout, lse, D, dqkv, B, S, H, Hkv, hd, s);
    CHECK_LAUNCH();
    CK(cudaFreeAsync(D, s));
    return ZL_OK;
  });
}

zl_status zl_op_gemm(int dtype, int mode, int M, int N, int K, const void* A, const void* B, void* C, void* stream) {
  if (!A || !B || !C) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if ((dtype != 0 && dtype != 1) || mode < 0 || mode > 2 || M < 0 || N < 0 || K < 0) {
    g_err = "bad dtype/mode/size";
    return ZL_ERR_ARG;
  }
  return guarded(nullptr, [&]() -> zl_status {
    gemm(dtype, mode, M, N, K, A, B, C, nullptr, nullptr, (cudaStream_t)stream);
    CHECK_LAUNCH();
    return ZL_OK;
  });
}

zl_status zl_op_qkv_rope(int dtype, int M, int N, int K, const void* A, const void* B, void* C, const float* bias,
                         const float* cs, int S, int hd, int rot_cols, void* stream) {
  if (!A || !B || !C || !cs) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if ((dtype != 0 && dtype != 1) || M < 0 || N < 0 || K < 0 || S < 1 || hd < 2 || hd % 2 != 0 || rot_cols < 0 ||
      rot_cols % hd != 0 || rot_cols > N) {
    g_err = "bad dtype/size, or rot_cols not whole heads within N";
    return ZL_ERR_ARG;
  }
  return guarded(nullptr, [&]() -> zl_status {
    cudaStream_t s = (cudaStream_t)stream;
    const GemmRope r{cs, S, hd, rot_cols};
    if (!(dtype == BF16 && M > 0 && gemm_tc_rope(M, N, K, A, B, C, bias, r, nullptr, s, nullptr))) {
      gemm(dtype, 0, M, N, K, A, B, C, bias, nullptr, s);
      if (M > 0 && rot_cols > 0) launch_rope_heads(dtype, C, cs, M, S, rot_cols / hd, hd, N, 0, s);
    }
    CHECK_LAUNCH();
    return ZL_OK;
  });
}

zl_status zl_op_gemm_ex(int dtype, int mode, int M, int N, int K, const void* A, const void* B, void* C,
                        float* bias, const void* R, int r_mode, void* stream) {
  if (!A || !B || !C) { g_err = "NULL argument"; return ZL_ERR_ARG; }
  if ((dtype != 0 && dtype != 1) || mode < 0 || mode > 2 || M < 0 || N < 0 || K < 0 || (r_mode != 0 && r_mode != 1) ||
      (r_mode == 1 && !R) || (mode == 2 && (R || r_mode))) {
    g_err = "bad dtype/mode/size/r_mode (r_mode 1 needs R; mode 2 takes no R)";
    return ZL_ERR_ARG;
  }
  if (mode == 2 && bias && M % 8 != 0) { g_err = "mode 2 column sums need M % 8 == 0"; return ZL_ERR_ARG; }
  return guarded(nullptr, [&]() -> zl_status {
    cudaStream_t s = (cudaStream_t)stream;
    gemm(dtype, mode, M, N, K, A, B, C, mode == 2 ? nullptr : bias, R, s, nullptr, nullptr, 1.f, r_mode);
    if (mode == 2 && bias && K > 0) {   // the column sums of A: the column-sum kernel of the bias gradients
      float* part = nullptr;
      unsigned* cnt = nullptr;
      CK(cudaMallocAsync((void**)&part, (size_t)colsum_blocks(K) * M * 4, s));
      CK(cudaMallocAsync((void**)&cnt, (size_t)colsum_groups(M) * 4, s));
      CK(cudaMemsetAsync(cnt, 0, (size_t)colsum_groups(M) * 4, s));
      launch_colsum(dtype, A, part, K, M, bias, cnt, s);
      CK(cudaFreeAsync(part, s));
      CK(cudaFreeAsync(cnt, s));
    }
    CHECK_LAUNCH();
    return ZL_OK;
  });
}

}  // extern "C"
