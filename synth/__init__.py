"""Seeded synthetic inputs for the joint next-k-token decode step.

This module is shared by the CPU oracle and by the CUDA path's tests and
benchmark.  It holds workload descriptions and random-number draws only:
none of the method's arithmetic (no norms, attention, noise encoding or
noise-to-token map) lives here.

Recipe (the paper's datasets and checkpoints are not available, so these
stand in for them):
  * weights: every matrix N(0, 0.02) (embeddings, learned positions,
    projections, LM head, noise-encoder layers); norm gains 1; biases 0.
    Each tensor is drawn from its own stream ``default_rng([seed, idx])`` so
    that changing one shape never shifts another tensor's values.  For bf16
    workloads the fp32 draws are rounded to the nearest bf16 value (ties to
    even) here, so both sides start from identical, bf16-exact weights.
  * prompts: token ids uniform over [0, V).
  * noise: fp32 uniform on [0, 1), one value per (step, sequence, slot).
  * ragged prompt lengths: integers uniform on [lo, hi].
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass

import numpy as np

SEED_WEIGHTS = 0
SEED_PROMPTS = 1
SEED_NOISE = 2
SEED_LENGTHS = 3
SEED_REQUESTS = 4


@dataclass(frozen=True)
class ModelConfig:
    """Shape and numeric mode of the push-forward causal Transformer."""

    n_layer: int
    d_model: int
    n_head: int
    d_ff: int
    vocab: int
    max_len: int
    pos: str = "rope"          # "rope" | "learned"
    dtype: str = "bf16"        # "fp32" | "bf16"
    noise_hidden: int = 0      # 0 => 4 * d_model
    tau: float = 1.0
    rms_eps: float = 1e-6
    rope_theta: float = 10000.0
    noise_scale: float = 1000.0
    map: str = "icdf"          # "icdf" | "argmax"
    mtp_k: int = 0             # 0: fully causal (k noise tokens, shared head);
                               # > 0: standard MTP (Sec. 3.3): one noise token, mtp_k heads

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_head

    @property
    def ne_hidden(self) -> int:
        return self.noise_hidden or 4 * self.d_model

    def replace(self, **kw) -> "ModelConfig":
        return dataclasses.replace(self, **kw)


@dataclass(frozen=True)
class Workload:
    """A decode workload: model, batch, prompt lengths and generation length."""

    name: str
    model: ModelConfig
    batch: int
    prompt_len: int            # fixed prompt length (ignored if ragged)
    gen_len: int               # tokens generated per sequence
    ks: tuple = (4,)
    ragged: tuple | None = None  # (lo, hi) for per-sequence prompt lengths
    page_size: int = 16


TINY = ModelConfig(n_layer=2, d_model=128, n_head=4, d_ff=512, vocab=1000,
                   max_len=64, pos="learned", dtype="fp32")
LM1B = ModelConfig(n_layer=12, d_model=768, n_head=12, d_ff=3072, vocab=30522,
                   max_len=128, pos="rope", dtype="bf16")
OWT = ModelConfig(n_layer=12, d_model=768, n_head=12, d_ff=3072, vocab=50257,
                  max_len=1024, pos="rope", dtype="bf16")
MEDIUM = ModelConfig(n_layer=24, d_model=1024, n_head=16, d_ff=4096,
                     vocab=50257, max_len=2048, pos="rope", dtype="bf16")

# standard-MTP variants of the same backbones (the architecture ablation of Sec. 3.3)
TINY_MTP = TINY.replace(mtp_k=3)
LM1B_MTP = LM1B.replace(mtp_k=4)

WORKLOADS = {
    # tiny fp32 parity case: one k=2 step after a 32-token prompt
    "tiny": Workload("tiny", TINY, batch=2, prompt_len=32, gen_len=2, ks=(2,)),
    # LM1B-shaped: prompt 32 -> 128, k=4 and the k=1 AR teacher step, batch 64
    "lm1b": Workload("lm1b", LM1B, batch=64, prompt_len=32, gen_len=96,
                     ks=(4, 2, 1)),
    # OWT-shaped: prompt 512 -> 1024
    "owt": Workload("owt", OWT, batch=8, prompt_len=512, gen_len=512,
                    ks=(4, 2, 1)),
    # OWT-shaped high-load paged serving: ragged prompts in [128, 896], 128 new
    "owt_paged": Workload("owt_paged", OWT, batch=512, prompt_len=0,
                          gen_len=128, ks=(4, 1), ragged=(128, 896)),
    # the standard-MTP variant of the LM1B-shaped model (Sec. 3.3 ablation)
    "lm1b_mtp": Workload("lm1b_mtp", LM1B_MTP, batch=64, prompt_len=32, gen_len=96,
                         ks=(4, 1)),
    # medium stress shape: prompt 1024 -> 2048
    "medium": Workload("medium", MEDIUM, batch=256, prompt_len=1024,
                       gen_len=1024, ks=(8, 4, 1)),
}


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16-representable fp32 (ties to even)."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    bits = a.view(np.uint32)
    bias = ((bits >> 16) & np.uint32(1)) + np.uint32(0x7FFF)
    out = ((bits + bias) & np.uint32(0xFFFF0000)).view(np.float32)
    return out


def weight_shapes(cfg: ModelConfig) -> dict:
    """Names and shapes of every weight tensor (nn.Linear layout: [out, in])."""
    L, d, F, V = cfg.n_layer, cfg.d_model, cfg.d_ff, cfg.vocab
    h = cfg.ne_hidden
    shapes = {
        "tok_emb": (V, d),
        "attn_norm": (L, d),
        "wqkv": (L, 3 * d, d),
        "wo": (L, d, d),
        "mlp_norm": (L, d),
        "w_up": (L, F, d),
        "w_down": (L, d, F),
        "final_norm": (d,),
        "w_head": (V, d),
        "ne_w1": (h, d * max(1, cfg.mtp_k)),
        "ne_b1": (h,),
        "ne_w2": (d, h),
        "ne_b2": (d,),
    }
    if cfg.pos == "learned":
        shapes["pos_emb"] = (cfg.max_len, d)
    if cfg.mtp_k:
        shapes["w_mtp"] = (cfg.mtp_k, V, d)
    return shapes


_ONES = ("attn_norm", "mlp_norm", "final_norm")
_ZEROS = ("ne_b1", "ne_b2")


def make_weights(cfg: ModelConfig, seed: int = SEED_WEIGHTS,
                 std: float = 0.02) -> dict:
    """All weights as C-contiguous float32 arrays (bf16-exact for bf16 models)."""
    out = {}
    for idx, (name, shape) in enumerate(sorted(weight_shapes(cfg).items())):
        if name in _ONES:
            a = np.ones(shape, np.float32)
        elif name in _ZEROS:
            a = np.zeros(shape, np.float32)
        else:
            rng = np.random.default_rng([seed, idx])
            a = rng.standard_normal(int(np.prod(shape)), dtype=np.float32)
            a *= np.float32(std)
            a = a.reshape(shape)
        if cfg.dtype == "bf16":
            a = round_to_bf16(a)
        out[name] = np.ascontiguousarray(a, dtype=np.float32)
    return out


def make_prompt_lengths(batch: int, lo: int, hi: int,
                        seed: int = SEED_LENGTHS) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return rng.integers(lo, hi + 1, size=batch).astype(np.int32)


def make_prompts(lengths, vocab: int, seed: int = SEED_PROMPTS) -> list:
    """One int32 array of uniform token ids per sequence."""
    rng = np.random.default_rng(seed)
    return [rng.integers(0, vocab, size=int(n)).astype(np.int32)
            for n in lengths]


def make_noise(n_steps: int, batch: int, k: int,
               seed: int = SEED_NOISE) -> np.ndarray:
    """fp32 U[0,1) noise, shape [n_steps, batch, max(k, 1)]."""
    rng = np.random.default_rng(seed)
    return rng.random((n_steps, batch, max(k, 1)), dtype=np.float32)


def make_requests(n: int, prompt_len: int, gen_lo: int, gen_hi: int, k: int, vocab: int,
                  seed: int = SEED_REQUESTS) -> list:
    """Serving requests: (prompt of uniform ids, generation length uniform in
    [gen_lo, gen_hi] rounded down to a multiple of k)."""
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        g = int(rng.integers(gen_lo, gen_hi + 1)) // k * k
        out.append((rng.integers(0, vocab, size=prompt_len).astype(np.int32), max(k, g)))
    return out


def workload_prompts(w: Workload, batch: int | None = None) -> list:
    b = w.batch if batch is None else batch
    if w.ragged is not None:
        lens = make_prompt_lengths(b, *w.ragged)
    else:
        lens = np.full(b, w.prompt_len, np.int32)
    return make_prompts(lens, w.model.vocab)
