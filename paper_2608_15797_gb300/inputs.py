"""Seeded synthetic inputs and workload geometries.

This module holds no arithmetic of the method: it only draws the random
queries, keys and values that both the CUDA path and the fp64 oracle consume,
and lists the workload shapes.  Values are drawn in float32 with numpy's PCG64
and rounded to the kernel's element type (bfloat16 round-to-nearest-even via
torch) before either side sees them, so both sides read bit-identical inputs
(the oracle widens them exactly to double).

Geometries follow the paper's Table 4 (Qwen2.5-Math 7B / 72B / 1.5B: layers,
KV heads, head dim 128) and the evaluation setup of Sec. 4.1 (budgets
B in {64, 128, 256, 512}); the synthetic Gaussian streams stand in for the
paper's Qwen2.5-Math decode traces, which cannot be reproduced without the
models and benchmarks.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

try:  # torch rounds float32 to bfloat16 with round-to-nearest-even
    import torch
except ImportError:  # pragma: no cover - torch is always present here
    torch = None


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    n_kv_heads: int
    group: int
    head_dim: int
    dtype: str            # "bf16" or "f32"
    budget: int           # B
    window: int           # W
    prompt: int           # prompt length loaded before decoding
    steps: int            # decode steps
    n_seq: int = 1
    n_cand: int = 1       # candidates per step (1 = plain decode)
    cand_step: int = 64   # tokens per candidate step
    sigma: float = 1.0    # std of q, k, v
    heavy_frac: float = 0.0   # fraction of keys scaled by heavy_scale
    heavy_scale: float = 3.0
    heavy_exact: bool = False  # exact count per (layer, head) of the prompt

    @property
    def n_q_heads(self):
        return self.n_kv_heads * self.group


_S7 = 1.0 / math.sqrt(128.0)

WORKLOADS = {
    # 1 layer, 4 q / 2 kv heads, d=64, fp32; prompt 128 + 256 steps, B=16, W=8,
    # 5% of prompt keys x3 (exact count per head).
    "tiny": Workload("tiny", 1, 2, 2, 64, "f32", 16, 8, 128, 256,
                     heavy_frac=0.05, heavy_exact=True),
    # Qwen2.5-Math-7B decode geometry (28 layers, 28 q / 4 kv heads, d 128).
    "7b_b64": Workload("7b_b64", 28, 4, 7, 128, "bf16", 64, 8, 512, 4096,
                       sigma=_S7),
    # 7B stepwise best-of-N: prompt 512 + 2048 prior tokens, B=128, N=4.
    "7b_bon4": Workload("7b_bon4", 28, 4, 7, 128, "bf16", 128, 8, 512, 2048,
                        n_cand=4, cand_step=64, sigma=_S7, heavy_frac=0.05),
    # Qwen2.5-Math-72B decode geometry (80 layers, 64 q / 8 kv heads), N=8.
    "72b_bon8": Workload("72b_bon8", 80, 8, 8, 128, "bf16", 64, 8, 1024, 2048,
                         n_cand=8, cand_step=64, sigma=_S7),
    # Throughput sweep: 64 sequences, prior lengths ~ U[512, 16384].
    "7b_s64_b64": Workload("7b_s64_b64", 28, 4, 7, 128, "bf16", 64, 8, 0, 0,
                           n_seq=64, sigma=_S7),
    "7b_s64_b128": Workload("7b_s64_b128", 28, 4, 7, 128, "bf16", 128, 8, 0,
                            0, n_seq=64, sigma=_S7),
    "7b_s64_b256": Workload("7b_s64_b256", 28, 4, 7, 128, "bf16", 256, 8, 0,
                            0, n_seq=64, sigma=_S7),
    "7b_s64_b512": Workload("7b_s64_b512", 28, 4, 7, 128, "bf16", 512, 8, 0,
                            0, n_seq=64, sigma=_S7),
    # Full-context helper decode at Qwen2.5-Math-1.5B geometry, context 16384.
    "1p5b_full16k": Workload("1p5b_full16k", 28, 2, 6, 128, "bf16", 1 << 30,
                             0, 16384, 0, sigma=_S7),
    # Parity-only: 7B geometry with unscaled N(0,1) q/k so that attention is
    # far from uniform and the selection is exercised.
    "7b_unscaled": Workload("7b_unscaled", 28, 4, 7, 128, "bf16", 64, 8, 512,
                            64, sigma=1.0),
}

PRIOR_LEN_RANGE = (512, 16384)


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float32 values to the element type; returns float32 holding
    exactly representable values."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    if dtype == "f32":
        return x
    if dtype != "bf16":
        raise ValueError(dtype)
    t = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32)
    return t.numpy()


def _rng(seed: int, *tags: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(
        [int(seed)] + [int(t) for t in tags])))


_TAG_PROMPT, _TAG_STEP, _TAG_HEAVY, _TAG_LEN, _TAG_PICK = 1, 2, 3, 4, 5


def _heavy_mask(w: Workload, rng: np.random.Generator, shape, n_axis: int):
    """Boolean mask of the keys scaled by heavy_scale."""
    if w.heavy_frac <= 0:
        return None
    if w.heavy_exact:
        # exact count floor(frac * n) per (layer, head) along axis n_axis
        n = shape[n_axis]
        cnt = int(math.floor(w.heavy_frac * n))
        lead = shape[:n_axis]
        m = np.zeros(shape[:n_axis + 1], bool)
        for idx in np.ndindex(*lead):
            sel = rng.permutation(n)[:cnt]
            m[idx + (sel,)] = True
        return m
    return rng.random(shape[:n_axis + 1]) < w.heavy_frac


def prompt(w: Workload, seed: int, seq: int, n: int, n_layers: Optional[int] = None):
    """Prompt keys/values [L][H][n][d] (float32, element-type exact)."""
    L = w.n_layers if n_layers is None else n_layers
    shape = (L, w.n_kv_heads, n, w.head_dim)
    rng = _rng(seed, _TAG_PROMPT, seq)
    k = rng.standard_normal(shape, dtype=np.float32) * np.float32(w.sigma)
    v = rng.standard_normal(shape, dtype=np.float32) * np.float32(w.sigma)
    hm = _heavy_mask(w, _rng(seed, _TAG_HEAVY, seq), shape, 2)
    if hm is not None:
        k[hm] *= np.float32(w.heavy_scale)
    return round_to(k, w.dtype), round_to(v, w.dtype)


def step_inputs(w: Workload, seed: int, step: int, n_seq: int,
                n_layers: Optional[int] = None, cand: int = 0):
    """One decode step: q [S][L][Hq][d], k_new/v_new [S][L][H][d]."""
    L = w.n_layers if n_layers is None else n_layers
    rng = _rng(seed, _TAG_STEP, step, cand)
    q = rng.standard_normal((n_seq, L, w.n_q_heads, w.head_dim),
                            dtype=np.float32) * np.float32(w.sigma)
    kshape = (n_seq, L, w.n_kv_heads, w.head_dim)
    k = rng.standard_normal(kshape, dtype=np.float32) * np.float32(w.sigma)
    v = rng.standard_normal(kshape, dtype=np.float32) * np.float32(w.sigma)
    if w.heavy_frac > 0 and not w.heavy_exact:
        hm = _rng(seed, _TAG_HEAVY, 1 << 20, step, cand).random(kshape[:3]) \
            < w.heavy_frac
        k[hm] *= np.float32(w.heavy_scale)
    return (round_to(q, w.dtype), round_to(k, w.dtype), round_to(v, w.dtype))


def prior_lengths(seed: int, n_seq: int, lo: int = PRIOR_LEN_RANGE[0],
                  hi: int = PRIOR_LEN_RANGE[1]) -> np.ndarray:
    """Per-sequence prior context lengths ~ U[lo, hi] (inclusive)."""
    return _rng(seed, _TAG_LEN).integers(lo, hi + 1, size=n_seq).astype(np.int32)


def candidate_pick(seed: int, step: int, n_seq: int, n_cand: int) -> np.ndarray:
    """Seeded stand-in for the PRM argmax of Eq. 2: the committed candidate."""
    return _rng(seed, _TAG_PICK, step).integers(0, n_cand, size=n_seq).astype(np.int32)


# Next-token logits of candidate rows (the degeneration detector's input).
# The paper's models are Qwen2.5-Math; their output layer has 152,064 logits
# (the tokenizer's vocabulary padded), which fixes the row length.
VOCAB = 152064
_TAG_LOGITS = 6


def candidate_logits(seed: int, step: int, rows: int, vocab: int = VOCAB,
                     sigma=3.0, boost=0.0, dtype: str = "bf16") -> np.ndarray:
    """Synthetic logits [rows][vocab] for one generated position (float32,
    element-type exact): N(0,1) * sigma[row], plus boost[row] on one token
    per row drawn uniformly.  sigma and boost are scalars or per-row arrays.

    The spread sets where a row sits against the detector's threshold: a
    wide spread concentrates the distribution on few tokens (a coherent,
    confident candidate), a narrow one spreads it over many (an incoherent
    one).  These Gaussian rows stand in for the Qwen2.5-Math logits of the
    paper's candidates."""
    rng = _rng(seed, _TAG_LOGITS, step)
    x = rng.standard_normal((rows, vocab), dtype=np.float32)
    x *= np.asarray(sigma, np.float32).reshape(-1, 1) if np.ndim(sigma) else \
        np.float32(sigma)
    b = np.broadcast_to(np.asarray(boost, np.float32), (rows,))
    if np.any(b != 0):
        hot = rng.integers(0, vocab, size=rows)
        x[np.arange(rows), hot] += b
    return round_to(x, dtype)
