"""Analytic memory / compute model of evicted decoding, and the algorithmic
byte counts of the decode-step kernels.

Part 1 restates the paper's App. D ("Overhead Derivation"):
  Eq. 8   m_kv = 2 L h_kv d_h b                  (KV bytes per token)
  Eq. 9   M_full(l) = m_kv l,  M_evict = m_kv B'  (B' = B + w)
  Eq. 10  M_full / M_evict = l / B'
  Eq. 11  M_KVR = N (m_kv^base B' + m_kv^help l),  M_full-BoN = N m_kv^base l
  Eq. 12  C(l) = 2P + 4 L d l                     (FLOP per decoded token)
  Eq. 13  C_evict = 2P + (1 + alpha) 4 L d B'
  Eq. 14  l* = (1 + alpha) B'
  Eq. 15  rho = C^help(l) / C^base_evict
with the Qwen2.5-Math constants of Table 4.

Part 2 counts the bytes a decode-step kernel must move at minimum (each byte
of input read once, each byte of output written once); the benchmark divides
these by the measured kernel time to get the achieved HBM bandwidth.
"""
from __future__ import annotations

import dataclasses

KiB = 1024
GiB = 1024 ** 3


@dataclasses.dataclass(frozen=True)
class ModelConsts:
    """Table 4: layers L, model dim d, KV heads h_kv, head dim d_h, FFN dim,
    parameter count P."""
    L: int
    d: int
    h_kv: int
    d_h: int
    d_ffn: int
    P: float


TABLE4 = {
    "7b": ModelConsts(28, 3584, 4, 128, 18944, 7.62e9),
    "72b": ModelConsts(80, 8192, 8, 128, 29568, 72.7e9),
    "1.5b": ModelConsts(28, 1536, 2, 128, 8960, 1.54e9),
}


def m_kv(m: ModelConsts, b: int = 2) -> int:
    """Eq. 8: bytes of K and V per cached token, all layers and KV heads."""
    return 2 * m.L * m.h_kv * m.d_h * b


def mem_full(m: ModelConsts, ell: int, b: int = 2) -> int:
    """Eq. 9: full-KV bytes per sequence at context ell."""
    return m_kv(m, b) * ell


def mem_evict(m: ModelConsts, B_phys: int, b: int = 2) -> int:
    """Eq. 9: evicted bytes per sequence, bounded by B' rows."""
    return m_kv(m, b) * B_phys


def mem_kvr(base: ModelConsts, helper: ModelConsts, N: int, ell: int,
            B_phys: int, b: int = 2) -> int:
    """Eq. 11: N evicted base candidates plus N full-context helper ones."""
    return N * (m_kv(base, b) * B_phys + m_kv(helper, b) * ell)


def mem_full_bon(base: ModelConsts, N: int, ell: int, b: int = 2) -> int:
    """Eq. 11: N full-KV base candidates."""
    return N * m_kv(base, b) * ell


def c_dense(m: ModelConsts) -> float:
    """Eq. 12: context-independent FLOP per token (2 per parameter)."""
    return 2.0 * m.P


def c_attn(m: ModelConsts, ell: float) -> float:
    """Eq. 12: QK^T plus value aggregation over ell cached tokens across the
    full query width d, two FLOP per multiply-add, all layers."""
    return 4.0 * m.L * m.d * ell


def c_evict(m: ModelConsts, B_phys: int, alpha: float) -> float:
    """Eq. 13: evicted per-token cost, flat in the context length."""
    return c_dense(m) + (1.0 + alpha) * c_attn(m, B_phys)


def crossover(B_phys: int, alpha: float) -> float:
    """Eq. 14: context beyond which evicted decode is cheaper per token."""
    return (1.0 + alpha) * B_phys


def helper_ratio(base: ModelConsts, helper: ModelConsts, ell: int,
                 B_phys: int, alpha: float) -> float:
    """Eq. 15: helper per-token cost relative to one evicted base candidate."""
    return (c_dense(helper) + c_attn(helper, ell)) / c_evict(base, B_phys, alpha)


# ---------------------------------------------------------------------------
# Part 2: algorithmic bytes of the decode-step kernels
# ---------------------------------------------------------------------------

STATE_BYTES = 16  # per unit: live length and next position, read and written


def step_unit_bytes(m: int, d: int, G: int, elem: int, out_elem: int,
                    budget: int, window: int, evict: bool = True,
                    moved: int = 0) -> int:
    """Minimum bytes of one fused decode step of one (sequence, layer, KV head)
    unit holding m rows before the step (n = m + 1 after the append).

    Reads every live K/V row, the new k/v, the G query rows, every live row's
    score and position; writes the G output rows, the retained rows' scores
    and the new row (K, V, position) into its slot.  `moved` counts surviving
    rows that sit beyond the retained length and are copied into freed slots
    (0 in the steady state, where the new row fills the single freed slot).
    """
    n = m + 1
    keep = min(n, budget + window) if evict else n
    b = 0
    b += 2 * m * d * elem          # K and V of the live rows
    b += 2 * d * elem              # k_new, v_new
    b += 2 * d * elem              # new row written into its slot
    b += G * d * elem              # q
    b += G * d * out_elem          # out
    b += 4 * m + 4 * keep          # scores: read live, write retained
    b += 4 * m + 4                 # positions: read live, write the new one
    b += moved * (2 * d * elem + 8) * 2
    b += STATE_BYTES
    return b


def attend_full_unit_bytes(m: int, d: int, G: int, elem: int,
                           out_elem: int) -> int:
    """Minimum bytes of one full-context decode step (no scores, no eviction)
    of one unit holding m rows before the append."""
    return (2 * m * d * elem + 2 * d * elem + 2 * d * elem + G * d * elem
            + G * d * out_elem + 4 + STATE_BYTES)
