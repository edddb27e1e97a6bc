"""Python binding of libkforcing.so: the C ABI in include/kforcing.h.

Argument marshalling only.  Every step of the decode path runs in the CUDA
library; if the library is missing this module raises instead of computing
anything itself.  Functions keep the C names (kf_init, kf_prefill,
kf_decode_step, ...); ``Decoder`` is a thin object wrapper over them.

Buffers may be numpy arrays (host) or torch tensors (host or CUDA); the
library classifies each pointer itself.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkforcing.so")

KF_OK, KF_E_ARG, KF_E_CAPACITY, KF_E_OOM, KF_E_CUDA, KF_E_DEVICE, KF_E_STATE = 0, -1, -2, -3, -4, -5, -6
KF_POS_ROPE, KF_POS_LEARNED = 0, 1
KF_DTYPE_FP32, KF_DTYPE_BF16 = 0, 1
KF_MAP_ICDF, KF_MAP_ARGMAX = 0, 1
KF_FLAG_NO_GRAPH, KF_FLAG_SIMT_GEMM, KF_FLAG_NO_PDL, KF_FLAG_NO_PERSISTENT_GEMM = 1, 2, 4, 16
KF_FLAG_NO_SKINNY = 32
KIND_NAMES = ["rowmap", "embed", "noise_gemm", "rmsnorm", "gemm_qkv", "rope_kv", "attention",
              "attn_combine", "gemm_o", "gemm_up", "gemm_down", "head_norm", "gemm_head",
              "head_select", "commit"]
KF_KIND_COUNT = len(KIND_NAMES)

EXPORTED = ["kf_init", "kf_prefill", "kf_decode_step", "kf_teacher_step", "kf_admit",
            "kf_debug_logits", "kf_rewind", "kf_get_lengths", "kf_set_stream", "kf_sync",
            "kf_profile_step", "kf_free", "kf_last_error"]


class KfError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"kforcing error {code}: {msg}")
        self.code = code


class kf_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "n_layer", "d_model", "n_head", "d_ff", "vocab", "max_len", "noise_hidden",
        "pos_kind", "dtype", "map_kind", "max_batch", "max_k", "page_size", "n_pages",
        "prefill_rows", "flags")] + [(n, ctypes.c_float) for n in (
        "tau", "rms_eps", "rope_theta", "noise_scale")] + [("mtp_k", ctypes.c_int32)]


WEIGHT_FIELDS = ("tok_emb", "pos_emb", "attn_norm", "wqkv", "wo", "mlp_norm", "w_up", "w_down",
                 "final_norm", "w_head", "ne_w1", "ne_b1", "ne_w2", "ne_b2", "w_mtp")


class kf_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in WEIGHT_FIELDS]


_lib = None


def load_library(path: str = LIB_PATH):
    """Load libkforcing.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build() "
                           "(there is no CPU fallback)")
    lib = ctypes.CDLL(path)
    P, I32, VP = ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p
    lib.kf_init.argtypes = [ctypes.POINTER(kf_config), ctypes.POINTER(kf_weights), VP,
                            ctypes.POINTER(P)]
    lib.kf_prefill.argtypes = [P, I32, VP, VP]
    lib.kf_decode_step.argtypes = [P, I32, I32, VP, VP]
    lib.kf_teacher_step.argtypes = [P, I32, I32, VP, VP]
    lib.kf_admit.argtypes = [P, I32, VP, VP, VP]
    lib.kf_debug_logits.argtypes = [P, VP]
    lib.kf_rewind.argtypes = [P]
    lib.kf_get_lengths.argtypes = [P, VP]
    lib.kf_set_stream.argtypes = [P, VP]
    lib.kf_sync.argtypes = [P]
    lib.kf_profile_step.argtypes = [P, I32, I32, VP, VP, VP, VP]
    lib.kf_free.argtypes = [P]
    lib.kf_last_error.argtypes = [P]
    lib.kf_last_error.restype = ctypes.c_char_p
    for n in EXPORTED:
        if n != "kf_last_error":
            getattr(lib, n).restype = ctypes.c_int
    _lib = lib
    return lib


def _ptr(a):
    """Data pointer of a numpy array or torch tensor (must be contiguous)."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError("array must be C-contiguous")
        return a.ctypes.data
    if hasattr(a, "data_ptr"):
        if not a.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return a.data_ptr()
    raise TypeError(f"unsupported buffer type {type(a)}")


def _check(rc, ctx=None):
    if rc != KF_OK:
        msg = load_library().kf_last_error(ctx)
        raise KfError(rc, msg.decode() if msg else "")


def make_config(model, max_batch: int, max_k: int, n_pages: int = 0, flags: int = 0,
                prefill_rows: int = 0) -> kf_config:
    """kf_config from a model description with the attributes of
    ``synth.ModelConfig`` (n_layer, d_model, ..., pos, dtype, map)."""
    c = kf_config()
    c.n_layer, c.d_model, c.n_head = model.n_layer, model.d_model, model.n_head
    c.d_ff, c.vocab, c.max_len = model.d_ff, model.vocab, model.max_len
    c.noise_hidden = model.noise_hidden
    c.pos_kind = KF_POS_LEARNED if model.pos == "learned" else KF_POS_ROPE
    c.dtype = KF_DTYPE_BF16 if model.dtype == "bf16" else KF_DTYPE_FP32
    c.map_kind = KF_MAP_ARGMAX if model.map == "argmax" else KF_MAP_ICDF
    c.max_batch, c.max_k, c.page_size, c.n_pages = max_batch, max_k, 16, n_pages
    c.prefill_rows, c.flags = prefill_rows, flags
    c.tau, c.rms_eps, c.rope_theta, c.noise_scale = (model.tau, model.rms_eps, model.rope_theta,
                                                     model.noise_scale)
    c.mtp_k = getattr(model, "mtp_k", 0)
    return c


# ------------------------------------------------------------------ C names

def kf_init(cfg: kf_config, weights: dict, stream: int = 0):
    lib = load_library()
    w = kf_weights()
    keep = []
    for n in WEIGHT_FIELDS:
        a = weights.get(n)
        if a is not None:
            if isinstance(a, np.ndarray):
                a = np.ascontiguousarray(a, np.float32)
            keep.append(a)
        setattr(w, n, _ptr(a))
    ctx = ctypes.c_void_p()
    _check(lib.kf_init(ctypes.byref(cfg), ctypes.byref(w), ctypes.c_void_p(stream or None),
                       ctypes.byref(ctx)))
    del keep
    return ctx


def kf_prefill(ctx, B: int, tokens, lens):
    lens = np.ascontiguousarray(lens, np.int32)
    if isinstance(tokens, np.ndarray):
        tokens = np.ascontiguousarray(tokens, np.int32)
    _check(load_library().kf_prefill(ctx, B, _ptr(tokens), _ptr(lens)), ctx)


def kf_decode_step(ctx, B: int, k: int, noise, out_tokens):
    _check(load_library().kf_decode_step(ctx, B, k, _ptr(noise), _ptr(out_tokens)), ctx)


def kf_teacher_step(ctx, B: int, k: int, noise, out_tokens):
    _check(load_library().kf_teacher_step(ctx, B, k, _ptr(noise), _ptr(out_tokens)), ctx)


def kf_admit(ctx, n: int, slots, tokens, lens):
    _check(load_library().kf_admit(ctx, n, _ptr(slots), _ptr(tokens), _ptr(lens)), ctx)


def kf_debug_logits(ctx, out):
    _check(load_library().kf_debug_logits(ctx, _ptr(out)), ctx)


def kf_rewind(ctx):
    _check(load_library().kf_rewind(ctx), ctx)


def kf_get_lengths(ctx, out):
    _check(load_library().kf_get_lengths(ctx, _ptr(out)), ctx)


def kf_set_stream(ctx, stream: int):
    _check(load_library().kf_set_stream(ctx, ctypes.c_void_p(stream or None)), ctx)


def kf_sync(ctx):
    _check(load_library().kf_sync(ctx), ctx)


def kf_profile_step(ctx, B, k, noise, out_tokens, ms_per_kind, launches_per_kind):
    _check(load_library().kf_profile_step(ctx, B, k, _ptr(noise), _ptr(out_tokens),
                                          _ptr(ms_per_kind), _ptr(launches_per_kind)), ctx)


def kf_free(ctx):
    if ctx:
        load_library().kf_free(ctx)


def kf_last_error(ctx=None) -> str:
    m = load_library().kf_last_error(ctx)
    return m.decode() if m else ""


class Decoder:
    """Owns one context: ``prefill(prompts)`` then ``step(k, noise)``."""

    def __init__(self, model, weights: dict, max_batch: int, max_k: int, stream: int = 0,
                 n_pages: int = 0, flags: int = 0, prefill_rows: int = 0):
        self.model = model
        self.cfg = make_config(model, max_batch, max_k, n_pages, flags, prefill_rows)
        self.ctx = kf_init(self.cfg, weights, stream)
        self.B = 0

    def prefill(self, prompts):
        lens = np.array([len(p) for p in prompts], np.int32)
        toks = np.concatenate([np.asarray(p, np.int32) for p in prompts])
        kf_prefill(self.ctx, len(prompts), toks, lens)
        self.B = len(prompts)

    def step(self, k: int, noise, out=None):
        """noise [B, max(k,1)] fp32 (host or device); returns int32 tokens."""
        if out is None:
            out = np.zeros((self.B, max(k, 1)), np.int32)
        kf_decode_step(self.ctx, self.B, k, noise, out)
        return out

    def teacher_step(self, k: int, noise, out=None):
        """k AR steps in one call (the G* teacher); noise [B, k]; returns [B, k]."""
        if out is None:
            out = np.zeros((self.B, k), np.int32)
        kf_teacher_step(self.ctx, self.B, k, noise, out)
        return out

    def admit(self, slots, prompts):
        """Replace the sequences `slots` (an int or a list) by new prompts at a
        step boundary."""
        if np.isscalar(slots):
            slots, prompts = [slots], [prompts]
        sl = np.asarray(slots, np.int32)
        lens = np.array([len(p) for p in prompts], np.int32)
        toks = np.concatenate([np.asarray(p, np.int32) for p in prompts]) if len(prompts) else \
            np.zeros(0, np.int32)
        kf_admit(self.ctx, len(sl), sl, np.ascontiguousarray(toks), lens)

    def logits(self, nout: int):
        out = np.zeros((self.B, nout, self.model.vocab), np.float32)
        kf_debug_logits(self.ctx, out)
        return out

    def lengths(self):
        out = np.zeros(self.B, np.int32)
        kf_get_lengths(self.ctx, out)
        return out

    def rewind(self):
        kf_rewind(self.ctx)

    def sync(self):
        kf_sync(self.ctx)

    def close(self):
        if self.ctx:
            kf_free(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
