"""Thin Python binding of libkvr (include/kvr.h) over ctypes.

Argument marshalling only: every step of the decode path runs in the CUDA
kernels of libkvr.so.  Functions keep the C names; torch tensors are passed by
their data pointers, and the stream defaults to torch's current CUDA stream.
Importing this module fails loudly if libkvr.so has not been built.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libkvr.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        f"libkvr.so not found at {LIB_PATH}: build it with "
        "`python -c 'import __graft_entry__ as g; g.build()'` (there is no "
        "fallback implementation)")

lib = ctypes.CDLL(LIB_PATH)

KVR_OK, KVR_EINVAL, KVR_ENOMEM, KVR_ECAPACITY, KVR_ECUDA, KVR_EDEVICE, \
    KVR_ESTATE = range(7)
STATUS_NAMES = {0: "KVR_OK", 1: "KVR_EINVAL", 2: "KVR_ENOMEM",
                3: "KVR_ECAPACITY", 4: "KVR_ECUDA", 5: "KVR_EDEVICE",
                6: "KVR_ESTATE"}
KVR_BF16, KVR_F32 = 0, 1
DTYPES = {"bf16": KVR_BF16, "f32": KVR_F32}
TORCH_DTYPES = {"bf16": torch.bfloat16, "f32": torch.float32}


class KvrError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class kvr_cache_desc(ctypes.Structure):
    _fields_ = [("n_seq", ctypes.c_int), ("n_layers", ctypes.c_int),
                ("n_kv_heads", ctypes.c_int), ("group", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("capacity", ctypes.c_int),
                ("kv_dtype", ctypes.c_int), ("out_dtype", ctypes.c_int),
                ("softmax_scale", ctypes.c_float)]


_P = ctypes.c_void_p
_I = ctypes.c_int
_S = ctypes.c_int

_SIGS = {
    "kvr_cache_required_bytes": (ctypes.c_size_t, [ctypes.POINTER(kvr_cache_desc)]),
    "kvr_cache_create": (_S, [ctypes.POINTER(kvr_cache_desc), _P, ctypes.c_size_t,
                              _P, ctypes.POINTER(_P)]),
    "kvr_cache_destroy": (None, [_P]),
    "kvr_cache_load": (_S, [_P, _I, _P, _P, _I, _I, _P]),
    "kvr_decode_attend_score": (_S, [_P, _I, _I, _P, _P, _P, _P, _P]),
    "kvr_decode_attend_score_noalloc": (_S, [_P, _I, _I, _P, _P, _P, _P, _P]),
    "kvr_evict_compact": (_S, [_P, _I, _I, _I, _I, _P]),
    "kvr_decode_step": (_S, [_P, _I, _I, _P, _P, _P, _P, _I, _I, _P]),
    "kvr_decode_step_rkv": (_S, [_P, _I, _I, _P, _P, _P, _P, _I, _I,
                                 ctypes.c_float, _P]),
    "kvr_decode_step_host": (_S, [_P, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P,
                                  _I, _I, _P]),
    "kvr_absorb_chunk": (_S, [_P, _I, _I, _I, _P, _P, _P, _P, _I, _I, _I, _P]),
    "kvr_cache_copy_sequences": (_S, [_P, _P, _P, _P, _I, _P]),
    "kvr_evict_compact_rkv": (_S, [_P, _I, _I, _I, _I, ctypes.c_float, _P]),
    "kvr_cache_export": (_S, [_P, _I, _P, _P, _P, _P, _P, _P, _P]),
    "kvr_cache_import": (_S, [_P, _I, _P, _P, _P, _P, _P, _P, _P]),
    "kvr_cache_lengths": (_S, [_P, _P]),
    "kvr_cache_launch_count": (_S, [_P, _P]),
    "kvr_cache_set_fused": (_S, [_P, _I]),
    "kvr_cache_set_wait_limit": (_S, [_P, ctypes.c_uint64]),
    "kvr_cache_set_hold_first_unit": (_S, [_P, _I]),
    "kvr_cache_set_fused_tuning": (_S, [_P, _I, _I]),
    "kvr_cache_set_chunk_tuning": (_S, [_P, _I, _I]),
    "kvr_fork_set_kernel": (_S, [_P, _I]),
    "kvr_fork_last_kernel": (_I, [_P]),
    "kvr_cache_set_absorb_kernel": (_S, [_P, _I]),
    "kvr_cache_last_absorb_kernel": (_I, [_P]),
    "kvr_cache_scores": (_S, [_P, _P, _P, _P, _P]),
    "kvr_sync_status": (_S, [_P, _P]),
    "kvr_last_error": (ctypes.c_char_p, []),
}
for _name, (_res, _args) in _SIGS.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args


def kvr_last_error() -> str:
    return lib.kvr_last_error().decode()


def _check(status: int, where: str):
    if status != KVR_OK:
        raise KvrError(status, where, kvr_last_error())


def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        if not t.is_contiguous():
            raise ValueError("tensors passed to libkvr must be contiguous")
        return ctypes.c_void_p(t.data_ptr())
    if isinstance(t, np.ndarray):
        if not t.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays passed to libkvr must be C-contiguous")
        return t.ctypes.data_as(ctypes.c_void_p)
    return ctypes.c_void_p(int(t))


def make_desc(n_seq, n_layers, n_kv_heads, group, head_dim, capacity,
              kv_dtype="bf16", out_dtype="bf16", softmax_scale=0.0):
    return kvr_cache_desc(n_seq, n_layers, n_kv_heads, group, head_dim,
                          capacity, DTYPES[kv_dtype], DTYPES[out_dtype],
                          float(softmax_scale))


def kvr_cache_required_bytes(desc: kvr_cache_desc) -> int:
    return int(lib.kvr_cache_required_bytes(ctypes.byref(desc)))


def kvr_cache_create(desc, dev_buf, nbytes, stream=None):
    h = ctypes.c_void_p()
    _check(lib.kvr_cache_create(ctypes.byref(desc), _ptr(dev_buf), nbytes,
                                _stream(stream), ctypes.byref(h)),
           "kvr_cache_create")
    return h


def kvr_cache_destroy(h):
    lib.kvr_cache_destroy(h)


def kvr_cache_load(h, seq, k, v, n_rows, first_pos=0, stream=None):
    _check(lib.kvr_cache_load(h, seq, _ptr(k), _ptr(v), n_rows, first_pos,
                              _stream(stream)), "kvr_cache_load")


def kvr_decode_attend_score(h, layer_begin, layer_end, q, k_new, v_new, out,
                            stream=None):
    _check(lib.kvr_decode_attend_score(h, layer_begin, layer_end, _ptr(q),
                                       _ptr(k_new), _ptr(v_new), _ptr(out),
                                       _stream(stream)),
           "kvr_decode_attend_score")


def kvr_decode_attend_score_noalloc(h, layer_begin, layer_end, q, k_new,
                                    v_new, out, stream=None):
    _check(lib.kvr_decode_attend_score_noalloc(h, layer_begin, layer_end,
                                               _ptr(q), _ptr(k_new),
                                               _ptr(v_new), _ptr(out),
                                               _stream(stream)),
           "kvr_decode_attend_score_noalloc")


def kvr_evict_compact(h, layer_begin, layer_end, budget, window, stream=None):
    _check(lib.kvr_evict_compact(h, layer_begin, layer_end, budget, window,
                                 _stream(stream)), "kvr_evict_compact")


def kvr_decode_step(h, layer_begin, layer_end, q, k_new, v_new, out, budget,
                    window, stream=None):
    _check(lib.kvr_decode_step(h, layer_begin, layer_end, _ptr(q), _ptr(k_new),
                               _ptr(v_new), _ptr(out), budget, window,
                               _stream(stream)), "kvr_decode_step")


def kvr_decode_step_rkv(h, layer_begin, layer_end, q, k_new, v_new, out,
                        budget, window, lam, stream=None):
    _check(lib.kvr_decode_step_rkv(h, layer_begin, layer_end, _ptr(q),
                                   _ptr(k_new), _ptr(v_new), _ptr(out), budget,
                                   window, float(lam), _stream(stream)),
           "kvr_decode_step_rkv")


def kvr_decode_step_host(h, layer_begin, layer_end, q_host, k_new_host,
                         v_new_host, out_host, q_dev, k_new_dev, v_new_dev,
                         out_dev, budget, window, stream=None):
    _check(lib.kvr_decode_step_host(
        h, layer_begin, layer_end, _ptr(q_host), _ptr(k_new_host),
        _ptr(v_new_host), _ptr(out_host), _ptr(q_dev), _ptr(k_new_dev),
        _ptr(v_new_dev), _ptr(out_dev), budget, window, _stream(stream)),
        "kvr_decode_step_host")


def kvr_absorb_chunk(h, layer_begin, layer_end, chunk, q, k_new, v_new, out,
                     budget, window, evict=True, stream=None):
    _check(lib.kvr_absorb_chunk(h, layer_begin, layer_end, chunk, _ptr(q),
                                _ptr(k_new), _ptr(v_new), _ptr(out), budget,
                                window, 1 if evict else 0, _stream(stream)),
           "kvr_absorb_chunk")


def kvr_evict_compact_rkv(h, layer_begin, layer_end, budget, window, lam,
                          stream=None):
    _check(lib.kvr_evict_compact_rkv(h, layer_begin, layer_end, budget, window,
                                     float(lam), _stream(stream)),
           "kvr_evict_compact_rkv")


def kvr_cache_copy_sequences(dst, dst_seqs, src, src_seqs, stream=None):
    d = np.ascontiguousarray(dst_seqs, dtype=np.int32)
    s = np.ascontiguousarray(src_seqs, dtype=np.int32)
    if d.shape != s.shape or d.ndim != 1:
        raise ValueError("dst_seqs and src_seqs must be 1-D of one length")
    _check(lib.kvr_cache_copy_sequences(dst, _ptr(d), src, _ptr(s), len(d),
                                        _stream(stream)),
           "kvr_cache_copy_sequences")


def kvr_cache_import(h, seq, host_k, host_v, host_score, host_pos, host_len,
                     host_next_pos, stream=None):
    _check(lib.kvr_cache_import(h, seq, _ptr(host_k), _ptr(host_v),
                                _ptr(host_score), _ptr(host_pos),
                                _ptr(host_len), _ptr(host_next_pos),
                                _stream(stream)), "kvr_cache_import")


def kvr_cache_export(h, seq, host_k, host_v, host_score, host_pos, host_len,
                     host_next_pos, stream=None):
    _check(lib.kvr_cache_export(h, seq, _ptr(host_k), _ptr(host_v),
                                _ptr(host_score), _ptr(host_pos),
                                _ptr(host_len), _ptr(host_next_pos),
                                _stream(stream)), "kvr_cache_export")


def kvr_cache_lengths(h, host_len):
    _check(lib.kvr_cache_lengths(h, _ptr(host_len)), "kvr_cache_lengths")


def kvr_cache_launch_count(h) -> int:
    n = ctypes.c_uint64()
    _check(lib.kvr_cache_launch_count(h, ctypes.byref(n)),
           "kvr_cache_launch_count")
    return int(n.value)


def kvr_cache_set_fused(h, enable: bool):
    _check(lib.kvr_cache_set_fused(h, 1 if enable else 0), "kvr_cache_set_fused")


def kvr_cache_set_fused_tuning(h, groups: int, group_warps: int = 0):
    _check(lib.kvr_cache_set_fused_tuning(h, groups, group_warps),
           "kvr_cache_set_fused_tuning")


def kvr_fork_set_kernel(h, kernel: int):
    _check(lib.kvr_fork_set_kernel(h, kernel), "kvr_fork_set_kernel")


def kvr_fork_last_kernel(h) -> int:
    return int(lib.kvr_fork_last_kernel(h))


def kvr_cache_set_chunk_tuning(h, groups: int, stages: int = 0):
    _check(lib.kvr_cache_set_chunk_tuning(h, groups, stages),
           "kvr_cache_set_chunk_tuning")


def kvr_sync_status(h, stream=None):
    _check(lib.kvr_sync_status(h, _stream(stream)), "kvr_sync_status")


class Cache:
    """Owner of one kvr_cache handle and the torch buffer it lives in."""

    def __init__(self, n_seq, n_layers, n_kv_heads, group, head_dim, capacity,
                 kv_dtype="bf16", out_dtype="bf16", softmax_scale=0.0,
                 device="cuda", stream=None, buf=None):
        """buf: an optional caller-owned uint8 device tensor of at least
        kvr_cache_required_bytes (256-byte aligned); by default one is
        allocated."""
        self.desc = make_desc(n_seq, n_layers, n_kv_heads, group, head_dim,
                              capacity, kv_dtype, out_dtype, softmax_scale)
        self.S, self.L, self.H, self.G, self.d = (n_seq, n_layers, n_kv_heads,
                                                  group, head_dim)
        self.cap = capacity
        self.kv_dtype, self.out_dtype = kv_dtype, out_dtype
        self.nbytes = kvr_cache_required_bytes(self.desc)
        if self.nbytes == 0:
            raise KvrError(KVR_EINVAL, "Cache", "invalid descriptor")
        if buf is None:
            buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        elif buf.numel() < self.nbytes or buf.dtype != torch.uint8:
            raise ValueError("buf must be uint8 with at least "
                             f"{self.nbytes} bytes")
        self.buf = buf
        self.handle = kvr_cache_create(self.desc, self.buf, self.nbytes, stream)

    def __del__(self):
        h = getattr(self, "handle", None)
        if h:
            kvr_cache_destroy(h)
            self.handle = None

    @property
    def kv_torch_dtype(self):
        return TORCH_DTYPES[self.kv_dtype]

    @property
    def out_torch_dtype(self):
        return TORCH_DTYPES[self.out_dtype]

    def load(self, seq, k, v, first_pos=0, stream=None):
        k = k.contiguous()
        v = v.contiguous()
        kvr_cache_load(self.handle, seq, k, v, k.shape[2], first_pos, stream)

    def _layers(self, layers):
        return (0, self.L) if layers is None else layers

    def new_out(self, nl):
        return torch.empty(self.S, nl, self.H * self.G, self.d,
                           dtype=self.out_torch_dtype, device=self.buf.device)

    def attend_score(self, q, k_new, v_new, out=None, layers=None, stream=None):
        lb, le = self._layers(layers)
        out = self.new_out(le - lb) if out is None else out
        kvr_decode_attend_score(self.handle, lb, le, q, k_new, v_new, out,
                                stream)
        return out

    def evict(self, budget, window, layers=None, stream=None):
        lb, le = self._layers(layers)
        kvr_evict_compact(self.handle, lb, le, budget, window, stream)

    def step(self, q, k_new, v_new, budget, window, out=None, layers=None,
             stream=None):
        lb, le = self._layers(layers)
        out = self.new_out(le - lb) if out is None else out
        kvr_decode_step(self.handle, lb, le, q, k_new, v_new, out, budget,
                        window, stream)
        return out

    def step_rkv(self, q, k_new, v_new, budget, window, lam=0.1, out=None,
                 layers=None, stream=None):
        """A decode step with the R-KV eviction (kvr_decode_step_rkv)."""
        lb, le = self._layers(layers)
        out = self.new_out(le - lb) if out is None else out
        kvr_decode_step_rkv(self.handle, lb, le, q, k_new, v_new, out, budget,
                            window, lam, stream)
        return out

    def absorb(self, q, k_new, v_new, budget=0, window=0, evict=True,
               out=None, layers=None, stream=None):
        """q [S][nl][c][H*G][d], k_new/v_new [S][nl][c][H][d] -> out
        [S][nl][c][H*G][d] (kvr_absorb_chunk)."""
        lb, le = self._layers(layers)
        c = q.shape[2]
        if out is None:
            out = torch.empty(self.S, le - lb, c, self.H * self.G, self.d,
                              dtype=self.out_torch_dtype, device=self.buf.device)
        kvr_absorb_chunk(self.handle, lb, le, c, q, k_new, v_new, out, budget,
                         window, evict, stream)
        return out

    def evict_rkv(self, budget, window, lam=0.1, layers=None, stream=None):
        """Eviction with the R-KV score (App. C), mix weight lam."""
        lb, le = self._layers(layers)
        kvr_evict_compact_rkv(self.handle, lb, le, budget, window, lam, stream)

    def copy_from(self, src: "Cache", src_seqs, dst_seqs, stream=None):
        """Sequence dst_seqs[i] takes the whole state of src's sequence
        src_seqs[i] (App. C: forking a candidate by copy, or committing the
        chosen one)."""
        kvr_cache_copy_sequences(self.handle, dst_seqs, src.handle, src_seqs,
                                 stream)

    def lengths(self):
        a = np.zeros((self.S, self.L), np.int32)
        kvr_cache_lengths(self.handle, a)
        return a

    def export(self, seq, kv=True, stream=None):
        """Host copy of one sequence: dict of numpy arrays (K/V as float32)."""
        rows = (self.L, self.H, self.cap)
        score = np.zeros(rows, np.float32)
        pos = np.zeros(rows, np.int32)
        ln = np.zeros(rows[:2], np.int32)
        npos = np.zeros(rows[:2], np.int32)
        hk = hv = None
        if kv:
            hk = torch.empty(*rows, self.d, dtype=self.kv_torch_dtype).contiguous()
            hv = torch.empty_like(hk)
        kvr_cache_export(self.handle, seq, hk, hv, score, pos, ln, npos, stream)
        res = {"score": score, "pos": pos, "len": ln, "next_pos": npos}
        if kv:
            res["K"] = hk.float().numpy()
            res["V"] = hv.float().numpy()
        return res

    def import_state(self, seq, state, stream=None):
        """Replace sequence seq with a state dict in the form export(seq,
        kv=True) returns (kvr_cache_import); K/V are cast to kv_dtype."""
        hk, hv = (torch.from_numpy(np.ascontiguousarray(state[x], np.float32))
                  .to(self.kv_torch_dtype).contiguous() for x in ("K", "V"))
        arr = {x: np.ascontiguousarray(state[x], t) for x, t in (
            ("score", np.float32), ("pos", np.int32), ("len", np.int32),
            ("next_pos", np.int32))}
        kvr_cache_import(self.handle, seq, hk, hv, arr["score"], arr["pos"],
                         arr["len"], arr["next_pos"], stream)

    def scores_view(self):
        """(score, pos, state) as device tensors viewing the cache buffer (no
        copy): score and pos [S][L][H][row_stride], state [S][L][H][4]."""
        sp, pp, stp = _P(), _P(), _P()
        stride = ctypes.c_int64()
        _check(lib.kvr_cache_scores(self.handle, ctypes.byref(sp), ctypes.byref(pp),
                                    ctypes.byref(stp), ctypes.byref(stride)),
               "kvr_cache_scores")
        base = self.buf.data_ptr()
        rows = self.S * self.L * self.H * stride.value

        def view(ptr, n, dtype):
            off = ptr.value - base
            return self.buf[off:off + 4 * n].view(dtype)

        shape = (self.S, self.L, self.H, stride.value)
        return (view(sp, rows, torch.float32).view(shape),
                view(pp, rows, torch.int32).view(shape),
                view(stp, self.S * self.L * self.H * 4, torch.int32).view(
                    self.S, self.L, self.H, 4))

    def set_absorb_kernel(self, kernel: int):
        """kvr_absorb_chunk's one-launch kernel: 0 tcgen05, 1 mma.sync."""
        _check(lib.kvr_cache_set_absorb_kernel(self.handle, kernel),
               "kvr_cache_set_absorb_kernel")

    def last_absorb_kernel(self) -> int:
        """How the last absorb ran (kvr_cache_last_absorb_kernel): 0 tcgen05,
        1 mma.sync, 2 token by token, -1 before the first."""
        return int(lib.kvr_cache_last_absorb_kernel(self.handle))

    def set_fused(self, enable: bool):
        kvr_cache_set_fused(self.handle, enable)

    def set_wait_limit(self, ns: int):
        """Bound of the step kernels' waits on copies (0: the 2 s default)."""
        _check(lib.kvr_cache_set_wait_limit(self.handle, int(ns)),
               "kvr_cache_set_wait_limit")

    def set_hold_first_unit(self, enable: bool):
        """Testing hook: the step kernels' first unit is never loaded, so
        its bounded wait runs out (kvr_cache_set_hold_first_unit)."""
        _check(lib.kvr_cache_set_hold_first_unit(self.handle, 1 if enable
                                                 else 0),
               "kvr_cache_set_hold_first_unit")

    def set_chunk_tuning(self, groups: int, stages: int = 0):
        """groups -1 keeps the chunked kernel off (older per-unit kernels)."""
        kvr_cache_set_chunk_tuning(self.handle, groups, stages)

    def launch_count(self):
        return kvr_cache_launch_count(self.handle)

    def sync_status(self, stream=None):
        kvr_sync_status(self.handle, stream)


# ---- candidates -------------------------------------------------------------

for _name, (_res, _args) in {
    "kvr_fork_required_bytes": (ctypes.c_size_t, [_P, _I, _I]),
    "kvr_fork_candidates": (_S, [_P, _I, _I, _P, ctypes.c_size_t, _P,
                                 ctypes.POINTER(_P)]),
    "kvr_fork_decode_attend_score": (_S, [_P, _I, _I, _P, _P, _P, _P, _P]),
    "kvr_fork_commit": (_S, [_P, _P, _I, _I, _P]),
    "kvr_fork_export": (_S, [_P, _I, _I, _P, _P, _P, _P, _P, _P, _P]),
    "kvr_fork_destroy": (None, [_P]),
}.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args


def kvr_fork_required_bytes(parent, n_cand, tail_cap) -> int:
    return int(lib.kvr_fork_required_bytes(parent, n_cand, tail_cap))


def kvr_fork_candidates(parent, n_cand, tail_cap, dev_buf, nbytes, stream=None):
    h = ctypes.c_void_p()
    _check(lib.kvr_fork_candidates(parent, n_cand, tail_cap, _ptr(dev_buf),
                                   nbytes, _stream(stream), ctypes.byref(h)),
           "kvr_fork_candidates")
    return h


def kvr_fork_decode_attend_score(fork, layer_begin, layer_end, q, k_new, v_new,
                                 out, stream=None):
    _check(lib.kvr_fork_decode_attend_score(fork, layer_begin, layer_end,
                                            _ptr(q), _ptr(k_new), _ptr(v_new),
                                            _ptr(out), _stream(stream)),
           "kvr_fork_decode_attend_score")


def kvr_fork_commit(fork, chosen, budget, window, stream=None):
    chosen = np.ascontiguousarray(chosen, dtype=np.int32)
    _check(lib.kvr_fork_commit(fork, _ptr(chosen), budget, window,
                               _stream(stream)), "kvr_fork_commit")


def kvr_fork_export(fork, cand, seq, prefix_score, tail_k, tail_v, tail_score,
                    tail_pos, tail_len, stream=None):
    _check(lib.kvr_fork_export(fork, cand, seq, _ptr(prefix_score), _ptr(tail_k),
                               _ptr(tail_v), _ptr(tail_score), _ptr(tail_pos),
                               _ptr(tail_len), _stream(stream)),
           "kvr_fork_export")


def kvr_fork_destroy(fork):
    lib.kvr_fork_destroy(fork)


class Fork:
    """N candidates of a Cache sharing its live rows (owner of the buffer)."""

    def __init__(self, cache: Cache, n_cand: int, tail_cap: int, stream=None,
                 kernel: int = 0, buf=None):
        """kernel: 0 the library's choice, 1 candidate-batched, 2 chunked,
        3 one CTA per unit, 4 generic, 5 candidate-batched on 5th-generation
        tensor cores (kvr_fork_set_kernel).  buf: an
        optional caller-owned uint8 device tensor of at least
        kvr_fork_required_bytes."""
        self.cache, self.N, self.tcap = cache, n_cand, tail_cap
        self.nbytes = kvr_fork_required_bytes(cache.handle, n_cand, tail_cap)
        if self.nbytes == 0:
            raise KvrError(KVR_EINVAL, "Fork", "invalid fork arguments")
        if buf is None:
            buf = torch.empty(self.nbytes, dtype=torch.uint8,
                              device=cache.buf.device)
        elif buf.numel() < self.nbytes or buf.dtype != torch.uint8:
            raise ValueError("buf must be uint8 with at least "
                             f"{self.nbytes} bytes")
        self.buf = buf
        self.handle = kvr_fork_candidates(cache.handle, n_cand, tail_cap,
                                          self.buf, self.nbytes, stream)
        if kernel:
            kvr_fork_set_kernel(self.handle, kernel)

    def __del__(self):
        h = getattr(self, "handle", None)
        if h:
            kvr_fork_destroy(h)
            self.handle = None

    def attend_score(self, q, k_new, v_new, out=None, layers=None, stream=None):
        c = self.cache
        lb, le = (0, c.L) if layers is None else layers
        if out is None:
            out = torch.empty(self.N, c.S, le - lb, c.H * c.G, c.d,
                              dtype=c.out_torch_dtype, device=c.buf.device)
        kvr_fork_decode_attend_score(self.handle, lb, le, q, k_new, v_new, out,
                                     stream)
        return out

    def commit(self, chosen, budget, window, stream=None):
        kvr_fork_commit(self.handle, chosen, budget, window, stream)

    def last_kernel(self) -> int:
        """The kernel that ran the last candidate step (kvr_fork_last_kernel)."""
        return kvr_fork_last_kernel(self.handle)

    def export(self, cand, seq, kv=False, stream=None):
        c = self.cache
        ps = np.zeros((c.L, c.H, c.cap), np.float32)
        ts = np.zeros((c.L, c.H, self.tcap), np.float32)
        tp = np.zeros((c.L, c.H, self.tcap), np.int32)
        tl = np.zeros((c.L, c.H), np.int32)
        tk = tv = None
        if kv:
            tk = torch.empty(c.L, c.H, self.tcap, c.d, dtype=c.kv_torch_dtype)
            tv = torch.empty_like(tk)
        kvr_fork_export(self.handle, cand, seq, ps, tk, tv, ts, tp, tl, stream)
        res = {"prefix_score": ps, "tail_score": ts, "tail_pos": tp,
               "tail_len": tl}
        if kv:
            res["tail_K"] = tk.float().numpy()
            res["tail_V"] = tv.float().numpy()
        return res


# ---- full-context decode ----------------------------------------------------

for _name, (_res, _args) in {
    "kvr_decode_attend_workspace_bytes": (ctypes.c_size_t, [_P, _I, _I, _I]),
    "kvr_decode_attend": (_S, [_P, _I, _I, _P, _P, _P, _P, _I, _P,
                               ctypes.c_size_t, _P]),
}.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args


def kvr_decode_attend_workspace_bytes(h, layer_begin, layer_end, n_splits=0):
    return int(lib.kvr_decode_attend_workspace_bytes(h, layer_begin, layer_end,
                                                     n_splits))


def kvr_decode_attend(h, layer_begin, layer_end, q, k_new, v_new, out,
                      n_splits, workspace, workspace_bytes, stream=None):
    _check(lib.kvr_decode_attend(h, layer_begin, layer_end, _ptr(q),
                                 _ptr(k_new), _ptr(v_new), _ptr(out), n_splits,
                                 _ptr(workspace), workspace_bytes,
                                 _stream(stream)), "kvr_decode_attend")


def attend_full(cache: Cache, q, k_new, v_new, out=None, layers=None,
                n_splits=0, workspace=None, stream=None):
    """Full-context decode step on `cache` (no scores, no eviction)."""
    lb, le = (0, cache.L) if layers is None else layers
    out = cache.new_out(le - lb) if out is None else out
    need = kvr_decode_attend_workspace_bytes(cache.handle, lb, le, n_splits)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8,
                                device=cache.buf.device)
    kvr_decode_attend(cache.handle, lb, le, q, k_new, v_new, out, n_splits,
                      workspace, workspace.numel(), stream)
    return out


# ---- degeneration detector: the entropy test --------------------------------

class kvr_entropy_desc(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int), ("vocab", ctypes.c_int),
                ("window", ctypes.c_int), ("guard", ctypes.c_int),
                ("tau", ctypes.c_float), ("temperature", ctypes.c_float),
                ("logits_dtype", ctypes.c_int)]


for _name, (_res, _args) in {
    "kvr_entropy_required_bytes": (ctypes.c_size_t,
                                   [ctypes.POINTER(kvr_entropy_desc)]),
    "kvr_entropy_create": (_S, [ctypes.POINTER(kvr_entropy_desc), _P,
                                ctypes.c_size_t, _P, ctypes.POINTER(_P)]),
    "kvr_entropy_reset": (_S, [_P, _I, _I, _P]),
    "kvr_entropy_step": (_S, [_P, _P, ctypes.c_int64, _P, _P, _P, _P]),
    "kvr_entropy_export": (_S, [_P, _P, _P, _P, _P]),
    "kvr_entropy_sync_status": (_S, [_P, _P]),
    "kvr_entropy_launch_count": (_S, [_P, _P]),
    "kvr_entropy_set_kernel": (_S, [_P, _I]),
    "kvr_entropy_destroy": (None, [_P]),
}.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args


def kvr_entropy_required_bytes(desc: kvr_entropy_desc) -> int:
    return int(lib.kvr_entropy_required_bytes(ctypes.byref(desc)))


def kvr_entropy_create(desc, dev_buf, nbytes, stream=None):
    h = _P()
    _check(lib.kvr_entropy_create(ctypes.byref(desc), _ptr(dev_buf), nbytes,
                                  _stream(stream), ctypes.byref(h)),
           "kvr_entropy_create")
    return h


def kvr_entropy_reset(h, row_begin, row_end, stream=None):
    _check(lib.kvr_entropy_reset(h, row_begin, row_end, _stream(stream)),
           "kvr_entropy_reset")


def kvr_entropy_step(h, logits, row_stride, entropy=None, mean=None,
                     stopped=None, stream=None):
    _check(lib.kvr_entropy_step(h, _ptr(logits), int(row_stride),
                                _ptr(entropy), _ptr(mean), _ptr(stopped),
                                _stream(stream)), "kvr_entropy_step")


def kvr_entropy_export(h, host_hist, host_count, host_stopped, stream=None):
    _check(lib.kvr_entropy_export(h, _ptr(host_hist), _ptr(host_count),
                                  _ptr(host_stopped), _stream(stream)),
           "kvr_entropy_export")


def kvr_entropy_sync_status(h, stream=None):
    _check(lib.kvr_entropy_sync_status(h, _stream(stream)),
           "kvr_entropy_sync_status")


def kvr_entropy_launch_count(h) -> int:
    n = ctypes.c_uint64()
    _check(lib.kvr_entropy_launch_count(h, ctypes.byref(n)),
           "kvr_entropy_launch_count")
    return n.value


def kvr_entropy_destroy(h):
    lib.kvr_entropy_destroy(h)


class EntropyDetector:
    """Owner of one kvr_entropy handle and the torch buffer it lives in
    (Sec. 3.2 entropy test; App. C tau 7.0, window 12, guard 24)."""

    def __init__(self, rows, vocab, window=12, guard=24, tau=7.0,
                 temperature=1.0, logits_dtype="bf16", device="cuda",
                 stream=None):
        self.desc = kvr_entropy_desc(rows, vocab, window, guard, float(tau),
                                     float(temperature), DTYPES[logits_dtype])
        self.rows, self.vocab, self.window = rows, vocab, window
        self.logits_dtype = logits_dtype
        self.nbytes = kvr_entropy_required_bytes(self.desc)
        if self.nbytes == 0:
            raise KvrError(KVR_EINVAL, "EntropyDetector", "invalid descriptor")
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        self.handle = kvr_entropy_create(self.desc, self.buf, self.nbytes,
                                         stream)

    def __del__(self):
        h = getattr(self, "handle", None)
        if h:
            kvr_entropy_destroy(h)
            self.handle = None

    def reset(self, begin=0, end=None, stream=None):
        kvr_entropy_reset(self.handle, begin, self.rows if end is None else end,
                          stream)

    def step(self, logits, entropy=None, mean=None, stopped=None, stream=None):
        """One generated token: logits [rows][>= vocab] (row stride taken
        from the tensor).  Returns (entropy, mean, stopped) device tensors."""
        if logits.dim() != 2 or logits.shape[0] != self.rows or \
                logits.shape[1] < self.vocab or logits.stride(1) != 1:
            raise ValueError("logits must be [rows][>= vocab] with unit "
                             "column stride")
        if logits.dtype != TORCH_DTYPES[self.logits_dtype]:
            raise ValueError("logits dtype does not match the descriptor")
        dev = logits.device
        entropy = torch.empty(self.rows, dtype=torch.float32, device=dev) \
            if entropy is None else entropy
        mean = torch.empty(self.rows, dtype=torch.float32, device=dev) \
            if mean is None else mean
        stopped = torch.empty(self.rows, dtype=torch.int32, device=dev) \
            if stopped is None else stopped
        _check(lib.kvr_entropy_step(self.handle,
                                    ctypes.c_void_p(logits.data_ptr()),
                                    int(logits.stride(0)), _ptr(entropy),
                                    _ptr(mean), _ptr(stopped),
                                    _stream(stream)), "kvr_entropy_step")
        return entropy, mean, stopped

    def export(self, stream=None):
        hist = np.zeros((self.rows, self.window), np.float32)
        count = np.zeros(self.rows, np.int32)
        stopped = np.zeros(self.rows, np.int32)
        kvr_entropy_export(self.handle, hist, count, stopped, stream)
        return hist, count, stopped

    def set_kernel(self, kernel: int):
        """0: the library's choice, 1: persistent streaming kernel, 2: one CTA
        per piece of a row."""
        _check(lib.kvr_entropy_set_kernel(self.handle, kernel),
               "kvr_entropy_set_kernel")

    def launch_count(self):
        return kvr_entropy_launch_count(self.handle)

    def sync_status(self, stream=None):
        kvr_entropy_sync_status(self.handle, stream)
