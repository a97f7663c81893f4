"""DC-Leap denoise step on one GB300: Python binding of libdcleap.so.

Argument marshalling only: every step of the decoding path runs in the CUDA
kernels of ``libdcleap.so`` (built in-tree by ``paper_2607_20467_gb300.build``).
There is no CPU fallback: if the library is missing, ``lib()`` raises.

Two layers:
* ``lib()`` - the raw ctypes functions, under their C names (``dcl_create``, ...);
* ``Context`` - a thin object over one ``dcl_ctx*`` whose methods take torch
  tensors (device buffers) or numpy arrays (host buffers) and raise ``DcleapError``
  on a non-zero status.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdcleap.so")

DCL_TILE_PAIR = 2
DCL_OK, DCL_ERR_INVALID_ARG, DCL_ERR_STATE, DCL_ERR_OOM, DCL_ERR_CUDA, DCL_ERR_TIMEOUT, \
    DCL_ERR_UNSUPPORTED = range(7)
STATUS_NAMES = ["OK", "INVALID_ARG", "STATE", "OOM", "CUDA", "TIMEOUT", "UNSUPPORTED"]

(DCL_W_EMBED, DCL_W_ATTN_NORM, DCL_W_Q, DCL_W_K, DCL_W_V, DCL_W_O, DCL_W_MLP_NORM, DCL_W_GATE,
 DCL_W_UP, DCL_W_DOWN, DCL_W_FINAL_NORM, DCL_W_LM_HEAD) = range(12)

KERNEL_KINDS = ["embed", "rmsnorm", "gemm_qkv", "attention", "gemm_o", "gemm_gateup",
                "gemm_down", "gemm_lmhead", "combine", "dcv", "v_transpose", "row_plan", "gemm_mlp"]


class ModelConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("n_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("ffn_dim", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("mask_id", ctypes.c_int32),
                ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float)]


class DecodeConfig(ctypes.Structure):
    _fields_ = [("tau_commit", ctypes.c_float), ("tau_draft", ctypes.c_float),
                ("max_window", ctypes.c_int32), ("block_len", ctypes.c_int32),
                ("gen_len", ctypes.c_int32), ("kv_cache", ctypes.c_int32),
                ("min_commit", ctypes.c_int32), ("contiguous_drafts", ctypes.c_int32),
                ("confidence", ctypes.c_int32), ("acceptance", ctypes.c_int32)]


class Stats(ctypes.Structure):
    _fields_ = [("steps", ctypes.c_int64), ("tokens", ctypes.c_int64),
                ("elapsed_ms", ctypes.c_double), ("done", ctypes.c_int32),
                ("jpde_bound", ctypes.c_double)]


class Allocator(ctypes.Structure):
    _fields_ = [("alloc", ctypes.c_void_p), ("free", ctypes.c_void_p), ("user", ctypes.c_void_p)]


_P = ctypes.c_void_p
_I = ctypes.c_int32
_F = ctypes.c_float
# name: (restype, argtypes)
SIGNATURES = {
    "dcl_create": (_I, [ctypes.POINTER(ModelConfig), _I, _I, _P, ctypes.POINTER(Allocator),
                        ctypes.POINTER(_P)]),
    "dcl_set_weight": (_I, [_P, _I, _I, _P, _I]),
    "dcl_init_random_weights": (_I, [_P, ctypes.c_uint64, _F, _F, _F]),
    "dcl_set_prompt": (_I, [_P, _I, _P, _I, ctypes.POINTER(DecodeConfig)]),
    "dcl_step": (_I, [_P, _P]),
    "dcl_generate": (_I, [_P, _I, _P, ctypes.POINTER(Stats)]),
    "dcl_restart": (_I, [_P]),
    "dcl_get_state": (_I, [_P, _P, _P]),
    "dcl_set_state": (_I, [_P, _P, _P]),
    "dcl_forward_debug": (_I, [_P, _P, _P, _P, _P, _P, _P]),
    "dcl_debug_hidden": (_I, [_P, _I, _P]),
    "dcl_forward_debug_from": (_I, [_P, _I, _P, _I, _P, _P, _P, _P, _P, _P]),
    "dcl_launch_floor": (_I, [_P, _I, _I, ctypes.POINTER(ctypes.c_float)]),
    "dcl_accept": (_I, [_P, _P, _I, _I, _I, _P, _P, ctypes.POINTER(DecodeConfig), _P]),
    "dcl_accept_noalloc": (_I, [_P, _I, _I, _I, _P, _P, ctypes.POINTER(DecodeConfig), _P, _P]),
    "dcl_fp8_quantise": (_I, [_P, ctypes.c_int64, ctypes.c_int64, _P, _P]),
    "dcl_op_rmsnorm": (_I, [_P, _P, _P, _P, _I, _I, _F]),
    "dcl_op_linear": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _I]),
    "dcl_op_attention": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I]),
    "dcl_op_lmhead_top2": (_I, [_P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _I]),
    "dcl_op_generate": (_I, [_P, _P, ctypes.c_uint64, _I, ctypes.c_int64, ctypes.c_int64, _F, _F]),
    "dcl_selftest_wait_timeout": (_I, [_P, _I]),
    "dcl_set_profiling": (_I, [_P, _I]),
    "dcl_profile_last_step": (_I, [_P, _P, _P, _I, _P]),
    "dcl_last_error": (ctypes.c_char_p, [_P]),
    "dcl_destroy": (None, [_P]),
}

_lib = None


def lib():
    """The loaded libdcleap.so with typed functions (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with "
                              "`python -m paper_2607_20467_gb300.build` (no CPU fallback exists)")
        handle = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(handle, name)
            fn.restype = res
            fn.argtypes = args
        _lib = handle
    return _lib


def __getattr__(name):  # module-level access to the raw C functions: dcl_step, ...
    if name in SIGNATURES:
        return getattr(lib(), name)
    raise AttributeError(name)


class DcleapError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"{STATUS_NAMES[status] if 0 <= status < 7 else status}: {message}")
        self.status = status


def _ptr(t):
    """Device pointer of a torch tensor / host pointer of a numpy array / None."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        if not t.flags["C_CONTIGUOUS"]:
            raise ValueError("host array must be C-contiguous")
        return t.ctypes.data
    if hasattr(t, "data_ptr"):
        if not t.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return t.data_ptr()
    if isinstance(t, int):
        return t
    raise TypeError(f"cannot pass {type(t)} as a pointer")


def _dev(t, name, itemsize, count=0):
    """Device pointer for a ``*_dev`` argument: a contiguous CUDA tensor of ``itemsize``-byte
    elements holding at least ``count`` of them (None passes as NULL, an int as a raw device
    address).  A host array, a CPU tensor, another element size or a short buffer is
    refused here, before a kernel could read or write past it."""
    if t is None or isinstance(t, int):
        return t
    if isinstance(t, np.ndarray) or not getattr(t, "is_cuda", False):
        raise ValueError(f"{name}: a device buffer (a CUDA tensor) is required")
    if t.element_size() != itemsize:
        raise TypeError(f"{name}: elements of {itemsize} bytes expected, got {t.dtype}")
    if t.numel() < count:
        raise ValueError(f"{name}: at least {count} elements needed, {t.numel()} given")
    return _ptr(t)


def weight_elements(shape, kind) -> int:
    """Elements of weight tensor `kind` (DCL_W_*) of a model of this shape: matrices in the
    nn.Linear layout [out_features][in_features], gains [d_model]."""
    d, hd, H, G, F, V = shape.d_model, shape.head_dim, shape.n_heads, shape.n_kv_heads, shape.ffn_dim, shape.vocab
    return {DCL_W_EMBED: V * d, DCL_W_ATTN_NORM: d, DCL_W_Q: H * hd * d, DCL_W_K: G * hd * d,
            DCL_W_V: G * hd * d, DCL_W_O: d * H * hd, DCL_W_MLP_NORM: d, DCL_W_GATE: F * d,
            DCL_W_UP: F * d, DCL_W_DOWN: d * F, DCL_W_FINAL_NORM: d, DCL_W_LM_HEAD: V * d}[kind]


def fp8_quantise(w_bits: np.ndarray):
    """dcl_fp8_quantise on a host bf16 weight (uint16 bit patterns [rows][cols]): returns
    (codes uint8 [rows][cols], exps int32 [rows]), row n storing w[n] ~ value(codes[n]) *
    2^exps[n] (E4M3, one power-of-two scale per row).  Host only: no GPU is used."""
    w_bits = np.ascontiguousarray(w_bits)
    if w_bits.dtype != np.uint16 or w_bits.ndim != 2:
        raise TypeError("w_bits: a 2-D array of bf16 bit patterns (uint16)")
    rows, cols = w_bits.shape
    codes = np.empty((rows, cols), np.uint8)
    exps = np.empty(rows, np.int32)
    st = lib().dcl_fp8_quantise(_ptr(w_bits), rows, cols, _ptr(codes), _ptr(exps))
    if st != DCL_OK:
        raise DcleapError(st, lib().dcl_last_error(None).decode())
    return codes, exps


def model_config(shape) -> ModelConfig:
    return ModelConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads,
                       shape.head_dim, shape.ffn_dim, shape.vocab, shape.mask_id,
                       shape.rope_theta, shape.rms_eps)


def decode_config(tau_commit=0.70, tau_draft=0.98, max_window=0, block_len=32, gen_len=0,
                  kv_cache=0, min_commit=1, contiguous_drafts=0, confidence=0,
                  acceptance=0) -> DecodeConfig:
    """confidence: 0 = top-1 probability, 1 = exp(-entropy); acceptance: 0 = DCV (contiguous),
    1 = Eq. threshold_pd in the semi-autoregressive block."""
    return DecodeConfig(tau_commit, tau_draft, max_window, block_len, gen_len, kv_cache,
                        min_commit, int(bool(contiguous_drafts)), confidence, acceptance)


class Context:
    """One dcl_ctx: a model (or ops-only when shape is None) on the current device."""

    def __init__(self, shape=None, max_batch=1, max_seq=1, stream=None):
        L = lib()
        self._L = L
        self.shape = shape
        self.stream = stream  # None: the context owns a blocking stream
        out = ctypes.c_void_p()
        cfg = model_config(shape) if shape is not None else None
        st = L.dcl_create(ctypes.byref(cfg) if cfg is not None else None, max_batch, max_seq,
                          self.stream, None, ctypes.byref(out))
        if st != DCL_OK:
            raise DcleapError(st, L.dcl_last_error(None).decode())
        self.ptr = out.value
        self.batch = 0
        self.n_prompt = 0
        self.gen_len = 0

    # ------------------------------------------------------------------ plumbing
    def _check(self, st):
        if st != DCL_OK:
            raise DcleapError(st, self._L.dcl_last_error(self.ptr).decode())

    def close(self):
        if getattr(self, "ptr", None):
            self._L.dcl_destroy(self.ptr)
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    # ------------------------------------------------------------------ the ABI
    def set_weight(self, kind, layer, src):
        """src: numpy bf16 bits (uint16) on the host, or a torch bf16 tensor on the device."""
        is_dev = 0 if isinstance(src, np.ndarray) else int(src.is_cuda)
        if isinstance(src, np.ndarray) and src.dtype != np.uint16:
            raise TypeError("host weights are bf16 bit patterns (uint16)")
        if not isinstance(src, np.ndarray) and src.element_size() != 2:
            raise TypeError(f"weights are bf16 (2-byte elements), got {src.dtype}")
        if self.shape is not None and 0 <= kind <= DCL_W_LM_HEAD:
            need = weight_elements(self.shape, kind)
            have = src.size if isinstance(src, np.ndarray) else src.numel()
            if have < need:
                raise ValueError(f"weight {kind}: {need} elements needed, {have} given")
        self._check(self._L.dcl_set_weight(self.ptr, kind, layer, _ptr(src), is_dev))

    def init_random_weights(self, seed, std=0.02, lm_head_scale=1.0, norm_gain_std=0.0):
        self._check(self._L.dcl_init_random_weights(self.ptr, seed, std, lm_head_scale, norm_gain_std))

    def set_prompt(self, prompt, cfg: DecodeConfig):
        prompt = np.ascontiguousarray(np.atleast_2d(prompt), dtype=np.int32)
        self._check(self._L.dcl_set_prompt(self.ptr, prompt.shape[0], _ptr(prompt), prompt.shape[1],
                                           ctypes.byref(cfg)))
        self.batch, self.n_prompt, self.gen_len = prompt.shape[0], prompt.shape[1], cfg.gen_len
        self.dcfg = cfg

    def step(self, return_k=False):
        if return_k:
            k = np.zeros(self.batch, np.int32)
            self._check(self._L.dcl_step(self.ptr, _ptr(k)))
            return k
        self._check(self._L.dcl_step(self.ptr, None))
        return None

    def generate(self, max_steps=1 << 20, out=True, check=True):
        """Returns (x[N:N+M] per row as int32 [batch][M] or None, Stats, status).
        ``out`` may be a preallocated (e.g. pinned) int32 [batch][M] host array."""
        if isinstance(out, np.ndarray):
            buf = out
        else:
            buf = np.zeros((self.batch, self.gen_len), np.int32) if out else None
        st = Stats()
        status = self._L.dcl_generate(self.ptr, max_steps, _ptr(buf), ctypes.byref(st))
        if check and status not in (DCL_OK,):
            self._check(status)
        return buf, st, status

    def restart(self):
        self._check(self._L.dcl_restart(self.ptr))

    def get_state(self):
        x = np.zeros((self.batch, self.n_prompt + self.gen_len), np.int32)
        p = np.zeros(self.batch, np.int32)
        self._check(self._L.dcl_get_state(self.ptr, _ptr(x), _ptr(p)))
        return x, p

    def set_state(self, x, p):
        x = np.ascontiguousarray(x, dtype=np.int32)
        p = np.ascontiguousarray(p, dtype=np.int32)
        self._check(self._L.dcl_set_state(self.ptr, _ptr(x), _ptr(p)))

    def _outs(self, logits, top1, p1, p2, conf, entropy):
        """Device pointers of the per-position outputs of a forward ([batch][M], logits
        [batch][M][vocab])."""
        n = self.batch * self.gen_len
        vocab = self.shape.vocab if self.shape is not None else 0
        return (_dev(logits, "logits", 2, n * vocab), _dev(top1, "top1", 4, n), _dev(p1, "p1", 4, n),
                _dev(p2, "p2", 4, n), _dev(conf, "conf", 4, n), _dev(entropy, "entropy", 4, n))

    def _stream_elems(self):
        """Elements of a residual stream buffer: float [batch*(N+M)][d_model]."""
        d = self.shape.d_model if self.shape is not None else 0
        return self.batch * (self.n_prompt + self.gen_len) * d

    def forward_debug(self, logits=None, top1=None, p1=None, p2=None, conf=None, entropy=None):
        self._check(self._L.dcl_forward_debug(self.ptr, *self._outs(logits, top1, p1, p2, conf, entropy)))

    def debug_hidden(self, layer, h):
        self._check(self._L.dcl_debug_hidden(self.ptr, layer, _dev(h, "h", 4, self._stream_elems())))

    def forward_debug_from(self, layer, h, commit=False, logits=None, top1=None, p1=None, p2=None, conf=None,
                           entropy=None):
        self._check(self._L.dcl_forward_debug_from(self.ptr, layer, _dev(h, "h", 4, self._stream_elems()),
                                                   int(bool(commit)),
                                                   *self._outs(logits, top1, p1, p2, conf, entropy)))

    def accept(self, logits, committed, x, cfg: DecodeConfig, k):
        B, P, V = logits.shape
        self._check(self._L.dcl_accept(self.ptr, _dev(logits, "logits", 2, B * P * V),
                                       B, P, V, _dev(committed, "committed", 4, B), _dev(x, "x", 4, B * P),
                                       ctypes.byref(cfg), _dev(k, "k", 4, B)))

    def op_rmsnorm(self, x, gain, y, eps):
        rows, d = x.shape
        self._check(self._L.dcl_op_rmsnorm(self.ptr, _dev(x, "x", 4, rows * d), _dev(gain, "gain", 2, d),
                                           _dev(y, "y", 2, rows * d), rows, d, eps))

    def op_linear(self, a, w, out, mode=0, tile=0):
        M, K = a.shape
        N = w.shape[0]
        self._check(self._L.dcl_op_linear(self.ptr, _dev(a, "a", 2, M * K), _dev(w, "w", 2, N * K),
                                          _dev(out, "out", 4 if mode == 1 else 2, M * N), M, N, K, mode, tile))

    def op_attention(self, qkv, out, batch, T, H, G, hd, q_rows=0):
        rows = batch * T
        self._check(self._L.dcl_op_attention(self.ptr, _dev(qkv, "qkv", 2, rows * (H + 2 * G) * hd),
                                             _dev(out, "out", 2, rows * H * hd), batch, T, H, G, hd, q_rows))

    def op_lmhead_top2(self, x, w, top1, p1, p2, tile=0, entropy=None):
        R, d = x.shape
        V = w.shape[0]
        self._check(self._L.dcl_op_lmhead_top2(self.ptr, _dev(x, "x", 2, R * d), _dev(w, "w", 2, V * d), R, V, d,
                                               _dev(top1, "top1", 4, R), _dev(p1, "p1", 4, R),
                                               _dev(p2, "p2", 4, R), _dev(entropy, "entropy", 4, R), tile))

    def op_generate(self, dst, seed, tid, start, count, std, mean=0.0):
        self._check(self._L.dcl_op_generate(self.ptr, _dev(dst, "dst", 2, count), seed, tid, start, count, std,
                                            mean))

    def selftest_wait_timeout(self, which):
        """Status of the bounded-wait self-test (DCL_ERR_TIMEOUT is the expected one)."""
        return self._L.dcl_selftest_wait_timeout(self.ptr, which)

    def launch_floor(self, n_kernels, reps=200):
        """Mean ms of a CUDA graph of n_kernels empty dependent launches."""
        ms = ctypes.c_float()
        self._check(self._L.dcl_launch_floor(self.ptr, n_kernels, reps, ctypes.byref(ms)))
        return ms.value

    def set_profiling(self, enable):
        self._check(self._L.dcl_set_profiling(self.ptr, int(bool(enable))))

    def profile_last_step(self, cap=4096):
        ms = np.zeros(cap, np.float32)
        kind = np.zeros(cap, np.int32)
        n = ctypes.c_int32(0)
        self._check(self._L.dcl_profile_last_step(self.ptr, _ptr(ms), _ptr(kind), cap, ctypes.byref(n)))
        return ms[:n.value].copy(), kind[:n.value].copy()

    # ------------------------------------------------------------------ helpers
    def load_weights(self, weights: dict):
        """Upload a dict of float32 (bf16-exact) arrays: embed, final_norm, lm_head and
        per-layer attn_norm, wq, wk, wv, wo, mlp_norm, w_gate, w_up, w_down."""
        import torch

        def up(kind, layer, a):
            bits = torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(torch.bfloat16)
            self.set_weight(kind, layer, bits.view(torch.int16).numpy().view(np.uint16))
        up(DCL_W_EMBED, 0, weights["embed"])
        up(DCL_W_FINAL_NORM, 0, weights["final_norm"])
        up(DCL_W_LM_HEAD, 0, weights["lm_head"])
        names = [(DCL_W_ATTN_NORM, "attn_norm"), (DCL_W_Q, "wq"), (DCL_W_K, "wk"), (DCL_W_V, "wv"),
                 (DCL_W_O, "wo"), (DCL_W_MLP_NORM, "mlp_norm"), (DCL_W_GATE, "w_gate"),
                 (DCL_W_UP, "w_up"), (DCL_W_DOWN, "w_down")]
        for li, lw in enumerate(weights["layers"]):
            for kind, key in names:
                up(kind, li, lw[key])


def exported_symbols():
    """Names declared in include/dcleap.h (for the ABI test)."""
    return [n for n in SIGNATURES]
