"""ctypes binding of libzerolock.so (include/zerolock.h): argument marshalling only.

Functions keep the C names (zl_create, zl_step, ...). Device arrays are passed as
``tensor.data_ptr()``; streams as ``torch.cuda.Stream.cuda_stream``. Importing this
module fails loudly if the library has not been built: there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Dict, List, Optional, Sequence

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libzerolock.so")

ZL_OK, ZL_ERR_ARG, ZL_ERR_CUDA, ZL_ERR_OOM, ZL_ERR_STATE, ZL_ERR_TIMEOUT, ZL_ERR_UNSUPPORTED = 0, -1, -2, -3, -4, -5, -6
ZL_ARCH_LLAMA, ZL_ARCH_GPT2 = 0, 1
ZL_DEVERR_BAD_ID, ZL_DEVERR_BAD_LABEL, ZL_DEVERR_TIMEOUT = 1, 2, 4
ZL_DTYPE_F32, ZL_DTYPE_BF16 = 0, 1
ZL_NOALLOC_MAX_ROWS = 65536   # rows of zl_op_local_loss_noalloc's static scratch (include/zerolock.h)

#: every symbol include/zerolock.h declares
EXPORTS = ["zl_create", "zl_free", "zl_set_stream", "zl_set_param", "zl_load_weights", "zl_get_param", "zl_param_numel",
           "zl_embed", "zl_forward_chunk", "zl_local_step", "zl_step", "zl_bp_step", "zl_eval_global_loss",
           "zl_read_losses", "zl_join", "zl_synchronize", "zl_peak_bytes", "zl_reset_peak", "zl_last_error",
           "zl_op_local_loss", "zl_op_local_loss_noalloc", "zl_op_head_loss", "zl_op_gemm", "zl_op_gemm_ex", "zl_op_qkv_rope", "zl_op_attention", "zl_op_attention_bwd", "zl_profile", "zl_profile_read", "zl_kernel_launches", "zl_chunk_state_bytes", "zl_chunk_save",
           "zl_chunk_load", "zl_replay", "zl_wait_selftest"]


class zl_model_dims(C.Structure):
    _fields_ = [("arch", C.c_int), ("dtype", C.c_int), ("n_layers", C.c_int), ("d_model", C.c_int),
                ("n_heads", C.c_int), ("n_kv_heads", C.c_int), ("d_ff", C.c_int), ("vocab", C.c_int),
                ("max_seq", C.c_int), ("norm_eps", C.c_float), ("rope_theta", C.c_float)]


class zl_train_cfg(C.Structure):
    _fields_ = [("alpha", C.c_float), ("kl_dir", C.c_int), ("consis_first", C.c_int), ("lr", C.c_float),
                ("beta1", C.c_float), ("beta2", C.c_float), ("eps", C.c_float), ("weight_decay", C.c_float),
                ("accum_m", C.c_int), ("max_live_chunks", C.c_int), ("lr_schedule", C.c_int),
                ("lr_gamma", C.c_float), ("serialize", C.c_int), ("lora_rank", C.c_int),
                ("lora_scale", C.c_float), ("replay_depth", C.c_int), ("adapter_dim", C.c_int),
                ("graph", C.c_int), ("unfused_update", C.c_int), ("loss_rows", C.c_int), ("fuzz_delay_us", C.c_int),
                ("fuzz_seed", C.c_uint)]


class ZLError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"zerolock status {status}: {msg}")
        self.status = status


def _load() -> C.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                          "(the CUDA library is required; there is no CPU path)")
    lib = C.CDLL(LIB_PATH)
    vp, i, f, sz = C.c_void_p, C.c_int, C.c_float, C.c_size_t
    sig = {
        "zl_create": [C.POINTER(zl_model_dims), i, C.POINTER(C.c_int), C.POINTER(zl_train_cfg), C.POINTER(vp)],
        "zl_free": [vp],
        "zl_set_stream": [vp, vp],
        "zl_set_param": [vp, C.c_char_p, vp, sz, i],
        "zl_load_weights": [vp, C.c_char_p, vp, sz, i],
        "zl_get_param": [vp, C.c_char_p, i, vp, sz, i],
        "zl_param_numel": [vp, C.c_char_p, C.POINTER(sz)],
        "zl_embed": [vp, vp, i, i, vp],
        "zl_forward_chunk": [vp, i, vp, vp, vp, i, i],
        "zl_local_step": [vp, i, vp, vp, vp, i, i, vp, C.POINTER(f)],
        "zl_step": [vp, vp, vp, i, i, C.POINTER(f)],
        "zl_bp_step": [vp, vp, vp, i, i, C.POINTER(f)],
        "zl_eval_global_loss": [vp, vp, vp, i, i, C.POINTER(f)],
        "zl_read_losses": [vp, C.POINTER(f), i],
        "zl_join": [vp],
        "zl_synchronize": [vp, i],
        "zl_peak_bytes": [vp, C.POINTER(sz), C.POINTER(sz)],
        "zl_reset_peak": [vp],
        "zl_last_error": [],
        "zl_op_local_loss": [i, vp, vp, vp, i, i, i, f, i, vp, vp, vp, vp],
        "zl_op_local_loss_noalloc": [i, vp, vp, vp, i, i, i, f, i, vp, vp, vp],
        "zl_op_head_loss": [i, vp, vp, vp, vp, i, i, i, i, f, i, i, vp, vp, vp, vp],
        "zl_op_gemm": [i, i, i, i, i, vp, vp, vp, vp],
        "zl_op_gemm_ex": [i, i, i, i, i, vp, vp, vp, vp, vp, i, vp],
        "zl_op_qkv_rope": [i, i, i, i, vp, vp, vp, vp, vp, i, i, i, vp],
        "zl_op_attention": [i, vp, vp, vp, i, i, i, i, i, vp],
        "zl_op_attention_bwd": [i, vp, vp, vp, vp, vp, i, i, i, i, i, vp],
        "zl_profile": [vp, i],
        "zl_profile_read": [vp, C.c_char_p, sz],
        "zl_kernel_launches": [C.POINTER(C.c_uint64)],
        "zl_chunk_state_bytes": [vp, i, C.POINTER(sz)],
        "zl_chunk_save": [vp, i, vp, sz],
        "zl_chunk_load": [vp, i, vp, sz],
        "zl_replay": [vp, i, C.POINTER(C.c_int), C.POINTER(f)],
        "zl_wait_selftest": [C.POINTER(C.c_uint)],
    }
    for name, args in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = C.c_char_p if name == "zl_last_error" else (None if name == "zl_free" else C.c_int)
    return lib


_lib = _load()


def last_error() -> str:
    return (_lib.zl_last_error() or b"").decode()


def _check(st: int) -> None:
    if st != ZL_OK:
        raise ZLError(st, last_error())


def _p(x) -> Optional[int]:
    """Pointer of a torch tensor (or None / int)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


# ---- thin wrappers with the C names -------------------------------------------------------------
def zl_create(dims: zl_model_dims, K: int, bounds: Sequence[int], cfg: zl_train_cfg) -> C.c_void_p:
    arr = (C.c_int * len(bounds))(*bounds)
    out = C.c_void_p()
    _check(_lib.zl_create(C.byref(dims), K, arr, C.byref(cfg), C.byref(out)))
    return out


def zl_free(ctx) -> None:
    _lib.zl_free(ctx)


def zl_set_stream(ctx, stream: int) -> None:
    _check(_lib.zl_set_stream(ctx, stream))


def zl_set_param(ctx, name: str, t) -> None:
    """t: fp32 torch tensor (host or CUDA), contiguous."""
    t = t.contiguous()
    _check(_lib.zl_set_param(ctx, name.encode(), t.data_ptr(), t.numel() * 4, int(t.is_cuda)))


def zl_load_weights(ctx, name: str, t) -> None:
    """Same as zl_set_param (the problem statement's name for loading a weight). t: fp32 tensor."""
    t = t.contiguous()
    _check(_lib.zl_load_weights(ctx, name.encode(), t.data_ptr(), t.numel() * 4, int(t.is_cuda)))


def zl_param_numel(ctx, name: str) -> int:
    n = C.c_size_t()
    _check(_lib.zl_param_numel(ctx, name.encode(), C.byref(n)))
    return n.value


def zl_get_param(ctx, name: str, which: int = 0):
    import torch
    n = zl_param_numel(ctx, name)
    out = torch.empty(n, dtype=torch.float32)
    _check(_lib.zl_get_param(ctx, name.encode(), which, out.data_ptr(), n * 4, 0))
    return out


def zl_embed(ctx, ids, B: int, S: int, h0_out) -> None:
    _check(_lib.zl_embed(ctx, _p(ids), B, S, _p(h0_out)))


def zl_forward_chunk(ctx, k: int, h_in, ids, h_out, B: int, S: int) -> None:
    _check(_lib.zl_forward_chunk(ctx, k, _p(h_in), _p(ids), _p(h_out), B, S))


def zl_local_step(ctx, k: int, h_in, ids, labels, B: int, S: int, h_out=None, want_loss: bool = True):
    loss = C.c_float()
    _check(_lib.zl_local_step(ctx, k, _p(h_in), _p(ids), _p(labels), B, S, _p(h_out),
                              C.byref(loss) if want_loss else None))
    return loss.value if want_loss else None


def zl_step(ctx, ids, labels, B: int, S: int, K: int, want_losses: bool = True):
    if want_losses:
        arr = (C.c_float * K)()
        _check(_lib.zl_step(ctx, _p(ids), _p(labels), B, S, arr))
        return list(arr)
    _check(_lib.zl_step(ctx, _p(ids), _p(labels), B, S, None))
    return None


def zl_bp_step(ctx, ids, labels, B: int, S: int, want_loss: bool = True):
    loss = C.c_float()
    _check(_lib.zl_bp_step(ctx, _p(ids), _p(labels), B, S, C.byref(loss) if want_loss else None))
    return loss.value if want_loss else None


def zl_eval_global_loss(ctx, ids, labels, B: int, S: int) -> float:
    loss = C.c_float()
    _check(_lib.zl_eval_global_loss(ctx, _p(ids), _p(labels), B, S, C.byref(loss)))
    return loss.value


def zl_read_losses(ctx, n: int) -> List[float]:
    arr = (C.c_float * n)()
    _check(_lib.zl_read_losses(ctx, arr, n))
    return list(arr)


def zl_join(ctx) -> None:
    _check(_lib.zl_join(ctx))


def zl_synchronize(ctx, timeout_ms: int = -1) -> None:
    _check(_lib.zl_synchronize(ctx, timeout_ms))


def zl_peak_bytes(ctx):
    pk, cur = C.c_size_t(), C.c_size_t()
    _check(_lib.zl_peak_bytes(ctx, C.byref(pk), C.byref(cur)))
    return pk.value, cur.value


def zl_reset_peak(ctx) -> None:
    _check(_lib.zl_reset_peak(ctx))


def _need(t, dtypes, what):
    if t is not None and not isinstance(t, int) and str(t.dtype).replace("torch.", "") not in dtypes:
        raise TypeError(f"{what}: dtype {t.dtype}, expected {dtypes}")


def _need_numel(t, n: int, what: str) -> None:
    """Raise ZLError(ZL_ERR_ARG) when a tensor argument holds fewer than n elements."""
    if t is not None and not isinstance(t, int) and t.numel() < n:
        raise ZLError(ZL_ERR_ARG, f"{what}: {t.numel()} elements, the call reads or writes {n}")


def _loss_sizes(z, t, labels, dz, N: int, ldz: int, loss, row_loss=None) -> None:
    if N >= 1 and ldz >= 1:
        for x, nm in ((z, "z"), (t, "t"), (dz, "dz")):
            _need_numel(x, N * ldz, nm)
        _need_numel(labels, N, "labels")
        _need_numel(row_loss, N, "row_loss")
        _need_numel(loss, 1, "loss")


def zl_op_local_loss(dtype: int, z, t, labels, N: int, V: int, ldz: int, alpha: float, kl_dir: int, dz, row_loss,
                     loss, stream: int = 0) -> None:
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    for x, nm in ((z, "z"), (t, "t"), (dz, "dz")):
        _need(x, act, nm)
    _need(labels, ("int32",), "labels")
    _need(row_loss, ("float32",), "row_loss")
    _need(loss, ("float32",), "loss")
    _loss_sizes(z, t, labels, dz, N, ldz, loss, row_loss)
    _check(_lib.zl_op_local_loss(dtype, _p(z), _p(t), _p(labels), N, V, ldz, alpha, kl_dir, _p(dz), _p(row_loss),
                                 _p(loss), stream))


def zl_op_local_loss_noalloc(dtype: int, z, t, labels, N: int, V: int, ldz: int, alpha: float, kl_dir: int, dz,
                             loss, stream: int = 0) -> None:
    """zl_op_local_loss without any device allocation (scratch in a static device array)."""
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    for x, nm in ((z, "z"), (t, "t"), (dz, "dz")):
        _need(x, act, nm)
    _need(labels, ("int32",), "labels")
    _need(loss, ("float32",), "loss")
    if N <= ZL_NOALLOC_MAX_ROWS:   # larger N is the library's own error (beyond its scratch)
        _loss_sizes(z, t, labels, dz, N, ldz, loss)
    _check(_lib.zl_op_local_loss_noalloc(dtype, _p(z), _p(t), _p(labels), N, V, ldz, alpha, kl_dir, _p(dz),
                                         _p(loss), stream))


def zl_op_head_loss(dtype: int, n, tn, W, labels, N: int, d: int, V: int, ldw: int, alpha: float, kl_dir: int,
                    rows_per_slice: int, dn, row_loss, loss, stream: int = 0) -> None:
    """The frozen head fused with the local objective over row slices (include/zerolock.h)."""
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    for x, nm in ((n, "n"), (tn, "tn"), (W, "W"), (dn, "dn")):
        _need(x, act, nm)
    _need(labels, ("int32",), "labels")
    _need(row_loss, ("float32",), "row_loss")
    _need(loss, ("float32",), "loss")
    if N >= 1 and d >= 1:
        for x, nm in ((n, "n"), (tn, "tn"), (dn, "dn")):
            _need_numel(x, N * d, nm)
        _need_numel(W, ldw * d, "W")
        _need_numel(labels, N, "labels")
        _need_numel(row_loss, N, "row_loss")
        _need_numel(loss, 1, "loss")
    _check(_lib.zl_op_head_loss(dtype, _p(n), _p(tn), _p(W), _p(labels), N, d, V, ldw, alpha, kl_dir, rows_per_slice,
                                _p(dn), _p(row_loss), _p(loss), stream))


def zl_op_attention(dtype: int, qkv, out, lse, B: int, S: int, H: int, Hkv: int, hd: int, stream: int = 0) -> None:
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    _need(qkv, act, "qkv")
    _need(out, act, "out")
    _need(lse, ("float32",), "lse")
    _check(_lib.zl_op_attention(dtype, _p(qkv), _p(out), _p(lse), B, S, H, Hkv, hd, stream))


def zl_op_attention_bwd(dtype: int, qkv, out, dout, lse, dqkv, B: int, S: int, H: int, Hkv: int, hd: int,
                        stream: int = 0) -> None:
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    for x, nm in ((qkv, "qkv"), (out, "out"), (dout, "dout"), (dqkv, "dqkv")):
        _need(x, act, nm)
    _need(lse, ("float32",), "lse")
    _check(_lib.zl_op_attention_bwd(dtype, _p(qkv), _p(out), _p(dout), _p(lse), _p(dqkv), B, S, H, Hkv, hd, stream))


def zl_op_gemm(dtype: int, mode: int, M: int, N: int, K: int, A, B, Cm, stream: int = 0) -> None:
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    _need(A, act, "A")
    _need(B, act, "B")
    _need(Cm, ("float32",) if mode == 2 else act, "C")
    _check(_lib.zl_op_gemm(dtype, mode, M, N, K, _p(A), _p(B), _p(Cm), stream))


def zl_op_gemm_ex(dtype: int, mode: int, M: int, N: int, K: int, A, B, Cm, bias=None, R=None, r_mode: int = 0,
                  stream: int = 0) -> None:
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    _need(A, act, "A")
    _need(B, act, "B")
    _need(Cm, ("float32",) if mode == 2 else act, "C")
    if bias is not None:
        _need(bias, ("float32",), "bias")
    if R is not None:
        _need(R, act, "R")
    _check(_lib.zl_op_gemm_ex(dtype, mode, M, N, K, _p(A), _p(B), _p(Cm), _p(bias) if bias is not None else None,
                              _p(R) if R is not None else None, r_mode, stream))


def zl_op_qkv_rope(dtype: int, M: int, N: int, K: int, A, B, Cm, cs, S: int, hd: int, rot_cols: int, bias=None,
                   stream: int = 0) -> None:
    """C = A B^T (+ bias), then rotate-half RoPE of the first rot_cols columns (heads of hd) of row n by
    position n % S; cs: fp32 [S, hd/2, 2] (cos, sin)."""
    act = ("bfloat16",) if dtype == ZL_DTYPE_BF16 else ("float32",)
    _need(A, act, "A")
    _need(B, act, "B")
    _need(Cm, act, "C")
    _need(cs, ("float32",), "cs")
    if bias is not None:
        _need(bias, ("float32",), "bias")
        _need_numel(bias, N, "bias")
    _need_numel(A, M * K, "A")
    _need_numel(B, N * K, "B")
    _need_numel(Cm, M * N, "C")
    _need_numel(cs, S * hd, "cs")
    _check(_lib.zl_op_qkv_rope(dtype, M, N, K, _p(A), _p(B), _p(Cm), _p(bias) if bias is not None else None, _p(cs),
                               S, hd, rot_cols, stream))


def zl_profile(ctx, on: bool) -> None:
    _check(_lib.zl_profile(ctx, int(on)))


def zl_profile_read(ctx) -> dict:
    import json
    buf = C.create_string_buffer(1 << 16)
    _check(_lib.zl_profile_read(ctx, buf, len(buf)))
    return json.loads(buf.value.decode() or "{}")


def zl_kernel_launches() -> int:
    n = C.c_uint64()
    _check(_lib.zl_kernel_launches(C.byref(n)))
    return n.value


def zl_chunk_save(ctx, k: int) -> bytes:
    n = C.c_size_t()
    _check(_lib.zl_chunk_state_bytes(ctx, k, C.byref(n)))
    buf = C.create_string_buffer(n.value)
    _check(_lib.zl_chunk_save(ctx, k, buf, n.value))
    return buf.raw


def zl_chunk_load(ctx, k: int, blob: bytes) -> None:
    _check(_lib.zl_chunk_load(ctx, k, blob, len(blob)))


def zl_replay(ctx, k: int):
    n, loss = C.c_int(), C.c_float()
    _check(_lib.zl_replay(ctx, k, C.byref(n), C.byref(loss)))
    return n.value, loss.value


def zl_wait_selftest() -> int:
    """Runs the bounded-wait self-test (seconds); returns the kernel's device error bits."""
    bits = C.c_uint()
    _check(_lib.zl_wait_selftest(C.byref(bits)))
    return bits.value


# ---- convenience object ----------------------------------------------------------------------
class ZeroLock:
    """One engine context: a model cut into K chunks, its AdamW state and K CUDA streams."""

    def __init__(self, dims, K: int, bounds: Sequence[int], *, dtype: str = "bf16", alpha: float = 0.5,
                 kl_dir: int = 0, consis_first: int = 1, lr: float = 1e-3, beta1: float = 0.9,
                 beta2: float = 0.999, eps: float = 1e-8, weight_decay: float = 0.01, accum_m: int = 1,
                 max_live_chunks: int = 0, lr_schedule: int = 0, lr_gamma: float = 1.0, serialize: bool = False,
                 lora_rank: int = 0, lora_scale: float = 1.0, replay_depth: int = 0, adapter_dim: int = 0,
                 graph: bool = False, unfused_update: bool = False, loss_rows: int = 0, fuzz_delay_us: int = 0,
                 fuzz_seed: int = 0, stream=None):
        import torch
        self.dims = dims
        self.K = K
        self.dtype = dtype
        self.adapter_dim = adapter_dim
        md = zl_model_dims(dims.arch, ZL_DTYPE_BF16 if dtype == "bf16" else ZL_DTYPE_F32, dims.n_layers,
                           dims.d_model, dims.n_heads, dims.n_kv_heads, dims.d_ff, dims.vocab, dims.max_seq,
                           dims.norm_eps, dims.rope_theta)
        cfg = zl_train_cfg(alpha, kl_dir, consis_first, lr, beta1, beta2, eps, weight_decay, accum_m,
                           max_live_chunks, lr_schedule, lr_gamma, int(serialize), lora_rank, lora_scale,
                           replay_depth, adapter_dim, int(graph), int(unfused_update), loss_rows, fuzz_delay_us,
                           fuzz_seed)
        self.ctx = zl_create(md, K, list(bounds), cfg)
        s = stream if stream is not None else torch.cuda.current_stream()
        zl_set_stream(self.ctx, s.cuda_stream)
        self._keep = []          # inputs borrowed by queued work, released at synchronize()

    @property
    def torch_dtype(self):
        import torch
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def load(self, params: Dict[str, "torch.Tensor"]) -> None:
        for n, t in params.items():
            zl_set_param(self.ctx, n, t.float())

    def get(self, name: str, which: int = 0):
        return zl_get_param(self.ctx, name, which)

    def step(self, ids, labels, want_losses: bool = True):
        B, S = ids.shape
        self._keep += [ids, labels]
        out = zl_step(self.ctx, ids, labels, B, S, self.K, want_losses)
        if want_losses:
            self._keep.clear()
        return out

    def bp_step(self, ids, labels, want_loss: bool = True):
        B, S = ids.shape
        self._keep += [ids, labels]
        out = zl_bp_step(self.ctx, ids, labels, B, S, want_loss)
        if want_loss:
            self._keep.clear()
        return out

    def local_step(self, k: int, h_in, ids, labels, h_out=None):
        B, S = labels.shape
        return zl_local_step(self.ctx, k, h_in, ids, labels, B, S, h_out, True)

    def forward_chunk(self, k: int, h_in, ids, B: int, S: int):
        import torch
        out = torch.empty(B * S, self.dims.d_model, dtype=self.torch_dtype, device="cuda")
        zl_forward_chunk(self.ctx, k, h_in, ids, out, B, S)
        self.synchronize()
        return out

    def embed(self, ids):
        import torch
        B, S = ids.shape
        out = torch.empty(B * S, self.dims.d_model, dtype=self.torch_dtype, device="cuda")
        zl_embed(self.ctx, ids, B, S, out)
        self.synchronize()
        return out

    def global_loss(self, ids, labels) -> float:
        B, S = ids.shape
        return zl_eval_global_loss(self.ctx, ids, labels, B, S)

    def read_losses(self, n: Optional[int] = None):
        out = zl_read_losses(self.ctx, self.K if n is None else n)
        self._keep.clear()
        return out

    def synchronize(self, timeout_ms: int = -1) -> None:
        zl_synchronize(self.ctx, timeout_ms)
        self._keep.clear()

    def peak_bytes(self):
        return zl_peak_bytes(self.ctx)

    def reset_peak(self) -> None:
        zl_reset_peak(self.ctx)

    def close(self) -> None:
        if getattr(self, "ctx", None):
            zl_free(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
