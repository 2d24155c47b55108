"""CPU oracle for the token-selection path (fp64, plain loops, written in C).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's ``cpu_baseline`` / reference leg may import this package. The CUDA
product path never does, and this package imports nothing from it.

The arithmetic lives in ``litevlm_oracle.c`` (its header states the definition
and every reading of the paper it takes). This module only compiles that file
with gcc and marshals numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "litevlm_oracle.c")
_SRC_THREADS = os.path.join(_HERE, "litevlm_oracle_threads.c")  # all-cores score for the CPU baseline
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liblitevlm_oracle.so")
_lock = threading.Lock()
_lib = None

DTYPE_CODES = {"f32": 0, "bf16": 1, "e4m3": 2}


def build(src: str = _SRC, out: str = _LIB, extra_flags=()) -> str:
    """Compile the oracle with gcc (no fused multiply-add contraction). The
    default build also links the all-cores score (litevlm_oracle_threads.c)."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    srcs = [src] + ([_SRC_THREADS] if src == _SRC else [])
    cmd = ["gcc", "-std=c99", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-pthread",
           *extra_flags, "-o", tmp, *srcs, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def load(path: Optional[str] = None):
    """ctypes handle of the oracle library, built on first use."""
    global _lib
    if path is not None:
        return _bind(ctypes.CDLL(path))
    with _lock:
        if _lib is None:
            if (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < max(os.path.getmtime(_SRC),
                                                                          os.path.getmtime(_SRC_THREADS)):
                build()
            _lib = _bind(ctypes.CDLL(_LIB))
    return _lib


def _bind(lib):
    P = ctypes.c_void_p
    i32, i64, f64, f32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double, ctypes.c_float
    lib.litevlm_oracle_decode.argtypes = [i32, P, i64]
    lib.litevlm_oracle_decode.restype = f64
    lib.litevlm_oracle_score.argtypes = [i32, P, P, i32, i32, i32, i32, P, P, f64, f64, P, P, P, P]
    lib.litevlm_oracle_score.restype = ctypes.c_int
    lib.litevlm_oracle_keep_count.argtypes = [i32, f32]
    lib.litevlm_oracle_keep_count.restype = i64
    lib.litevlm_oracle_topk.argtypes = [i32, P, P, P, f32, P, P]
    lib.litevlm_oracle_topk.restype = ctypes.c_int
    lib.litevlm_oracle_compact.argtypes = [i64, P, P, P, i64]
    lib.litevlm_oracle_compact.restype = ctypes.c_int
    lib.litevlm_oracle_score_full.argtypes = [i32, P, P, P, i32, i32, i32, i32, P, P, P, P, f64, f64, P, P, P]
    lib.litevlm_oracle_score_full.restype = ctypes.c_int
    lib.litevlm_oracle_splice.argtypes = [i32, P, P, P, P, P, P, P, P, i64, P, P, P]
    lib.litevlm_oracle_splice.restype = ctypes.c_int
    lib.litevlm_oracle_select_views.argtypes = [i32, i32, P, P, P, ctypes.c_float, ctypes.c_float, ctypes.c_float,
                                                 i32, P, P, P, P]
    lib.litevlm_oracle_select_views.restype = ctypes.c_int
    lib.litevlm_oracle_project.argtypes = [i64, i32, i32, P, P, f64, P, P, i32, P, f64, P]
    lib.litevlm_oracle_project.restype = ctypes.c_int
    if hasattr(lib, "litevlm_oracle_score_threads"):
        lib.litevlm_oracle_score_threads.argtypes = [i32, P, P, i32, i32, i32, i32, P, P, f64, f64, P, i32]
        lib.litevlm_oracle_score_threads.restype = ctypes.c_int
    return lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


class OracleError(RuntimeError):
    pass


def decode(dtype: str, raw: np.ndarray, lib=None) -> np.ndarray:
    """Element-wise decode of f32 / bf16 bits / e4m3 codes to float64."""
    lib = lib or load()
    raw = np.ascontiguousarray(raw)
    flat = raw.reshape(-1)
    code = DTYPE_CODES[dtype]
    return np.array([lib.litevlm_oracle_decode(code, _ptr(flat), i) for i in range(flat.size)],
                    dtype=np.float64).reshape(raw.shape)


def score(q: np.ndarray, k: np.ndarray, seq_offsets, text_offsets, hq: int, hkv: int, head_dim: int,
          dtype: str = "bf16", q_scale: float = 1.0, k_scale: float = 1.0, lib=None, details: bool = False):
    """Per-visual-token importance scores (fp32), and with details=True also the
    unrounded fp64 scores, per-(b,h,i) softmax row sums and log-sum-exp values."""
    lib = lib or load()
    so = np.ascontiguousarray(seq_offsets, dtype=np.int32)
    to = np.ascontiguousarray(text_offsets, dtype=np.int32)
    batch = so.size - 1
    n_tot, t_tot = int(so[-1]), int(to[-1])
    q = np.ascontiguousarray(q)
    k = np.ascontiguousarray(k)
    out = np.zeros(n_tot, dtype=np.float32)
    s64 = np.zeros(n_tot, dtype=np.float64) if details else None
    rows = np.zeros(hq * t_tot, dtype=np.float64) if details else None
    lse = np.zeros(hq * t_tot, dtype=np.float64) if details else None
    rc = lib.litevlm_oracle_score(batch, _ptr(so), _ptr(to), hq, hkv, head_dim, DTYPE_CODES[dtype],
                                  _ptr(q), _ptr(k), float(q_scale), float(k_scale),
                                  _ptr(out), _ptr(s64), _ptr(rows), _ptr(lse))
    if rc != 0:
        raise OracleError(f"litevlm_oracle_score returned {rc}")
    if details:
        return out, s64, rows, lse
    return out


def score_threads(q: np.ndarray, k: np.ndarray, seq_offsets, text_offsets, hq: int, hkv: int, head_dim: int,
                  dtype: str = "bf16", q_scale: float = 1.0, k_scale: float = 1.0, threads: int = 1, lib=None):
    """The scores of ``score`` computed on `threads` POSIX threads, bit for bit
    the same (the serial summation order is kept)."""
    lib = lib or load()
    so = np.ascontiguousarray(seq_offsets, dtype=np.int32)
    to = np.ascontiguousarray(text_offsets, dtype=np.int32)
    q = np.ascontiguousarray(q)
    k = np.ascontiguousarray(k)
    out = np.zeros(int(so[-1]), dtype=np.float32)
    rc = lib.litevlm_oracle_score_threads(so.size - 1, _ptr(so), _ptr(to), hq, hkv, head_dim, DTYPE_CODES[dtype],
                                          _ptr(q), _ptr(k), float(q_scale), float(k_scale), _ptr(out), int(threads))
    if rc != 0:
        raise OracleError(f"litevlm_oracle_score_threads returned {rc}")
    return out


def score_full(q: np.ndarray, k: np.ndarray, k_sys: np.ndarray, k_txt: np.ndarray, seq_offsets, text_offsets,
               sys_offsets, hq: int, hkv: int, head_dim: int, dtype: str = "bf16", q_scale: float = 1.0,
               k_scale: float = 1.0, lib=None, details: bool = False):
    """Scores with the softmax over the full causal key set (system, visual,
    text keys up to the query); details=True also returns the fp64 scores and
    the visual attention share per (b, h, i)."""
    lib = lib or load()
    so, to, yo = (np.ascontiguousarray(a, dtype=np.int32) for a in (seq_offsets, text_offsets, sys_offsets))
    batch = so.size - 1
    n_tot, t_tot = int(so[-1]), int(to[-1])
    arrs = [np.ascontiguousarray(a) for a in (q, k, k_sys, k_txt)]
    out = np.zeros(n_tot, dtype=np.float32)
    s64 = np.zeros(n_tot, dtype=np.float64)
    share = np.zeros(max(1, hq * t_tot), dtype=np.float64)
    rc = lib.litevlm_oracle_score_full(batch, _ptr(so), _ptr(to), _ptr(yo), hq, hkv, head_dim, DTYPE_CODES[dtype],
                                       _ptr(arrs[0]), _ptr(arrs[1]), _ptr(arrs[2]), _ptr(arrs[3]), float(q_scale),
                                       float(k_scale), _ptr(out), _ptr(s64), _ptr(share))
    if rc != 0:
        raise OracleError(f"litevlm_oracle_score_full returned {rc}")
    if details:
        return out, s64, share[:hq * t_tot]
    return out


def keep_count(n: int, keep_ratio: float, lib=None) -> int:
    lib = lib or load()
    return int(lib.litevlm_oracle_keep_count(int(n), float(keep_ratio)))


def topk(seq_offsets, scores: np.ndarray, keep_k=None, keep_ratio: float = 0.0, lib=None):
    """(kept_idx int32 [sum k_b], out_offsets int32 [B+1])."""
    lib = lib or load()
    so = np.ascontiguousarray(seq_offsets, dtype=np.int32)
    batch = so.size - 1
    scores = np.ascontiguousarray(scores, dtype=np.float32)
    kk = None if keep_k is None else np.ascontiguousarray(keep_k, dtype=np.int32)
    if kk is not None:
        total = int(kk.sum())
    else:
        total = sum(keep_count(int(so[b + 1] - so[b]), keep_ratio, lib) for b in range(batch))
    kept = np.zeros(max(total, 1), dtype=np.int32)
    out_off = np.zeros(batch + 1, dtype=np.int32)
    rc = lib.litevlm_oracle_topk(batch, _ptr(so), _ptr(scores), _ptr(kk), float(keep_ratio),
                                 _ptr(kept), _ptr(out_off))
    if rc != 0:
        raise OracleError(f"litevlm_oracle_topk returned {rc}")
    return kept[:total], out_off


def compact(kept_idx: np.ndarray, src: np.ndarray, lib=None) -> np.ndarray:
    """Rows src[kept_idx] copied byte for byte (src is [rows, ...], any dtype)."""
    lib = lib or load()
    src = np.ascontiguousarray(src)
    kept = np.ascontiguousarray(kept_idx, dtype=np.int32)
    row_bytes = src.dtype.itemsize * (int(np.prod(src.shape[1:])) if src.ndim > 1 else 1)
    dst = np.zeros((kept.size,) + src.shape[1:], dtype=src.dtype)
    rc = lib.litevlm_oracle_compact(kept.size, _ptr(kept), _ptr(src), _ptr(dst), row_bytes)
    if rc != 0:
        raise OracleError(f"litevlm_oracle_compact returned {rc}")
    return dst


def splice(sys_offsets, seq_offsets, kept_offsets, kept_idx, text_offsets, sys_rows: np.ndarray,
           vis_rows: np.ndarray, txt_rows: np.ndarray, lib=None):
    """Prefill sequence [system; kept visual; text] per request with original
    position ids. Rows are [n, row_bytes] uint8 (or any dtype, copied as bytes).
    Returns (out_rows, out_offsets, position_ids)."""
    lib = lib or load()
    so, vo, ko, to = (np.ascontiguousarray(a, dtype=np.int32) for a in
                      (sys_offsets, seq_offsets, kept_offsets, text_offsets))
    batch = len(so) - 1
    ki = np.ascontiguousarray(kept_idx, dtype=np.int32)
    rows = [np.ascontiguousarray(r).view(np.uint8).reshape(r.shape[0], -1) for r in (sys_rows, vis_rows, txt_rows)]
    rb = max(r.shape[1] for r in rows)
    total = int(so[-1] + ko[-1] + to[-1])
    out = np.zeros((max(total, 1), rb), np.uint8)
    off = np.zeros(batch + 1, np.int32)
    pos = np.zeros(max(total, 1), np.int32)
    rc = lib.litevlm_oracle_splice(batch, _ptr(so), _ptr(vo), _ptr(ko), _ptr(ki), _ptr(to), _ptr(rows[0]),
                                   _ptr(rows[1]), _ptr(rows[2]), rb, _ptr(out), _ptr(off), _ptr(pos))
    if rc != 0:
        raise OracleError(f"splice failed ({rc})")
    return out[:total], off, pos[:total]


def select_views(lexical: np.ndarray, logits: np.ndarray, tokens_per_view, w_lex: float, w_logit: float,
                 threshold: float, min_views: int = 0, lib=None):
    """Patch-selection gating. lexical, logits: float32 [B, V]. Returns
    (view_mask uint8 [B, V], view_offsets [B+1], selected_views, seq_offsets [B+1])."""
    lib = lib or load()
    lx = np.ascontiguousarray(lexical, dtype=np.float32)
    lg = np.ascontiguousarray(logits, dtype=np.float32)
    batch, nv = lx.shape
    tpv = np.ascontiguousarray(tokens_per_view, dtype=np.int32)
    mask = np.zeros((batch, nv), np.uint8)
    vo = np.zeros(batch + 1, np.int32)
    sv = np.zeros(max(1, batch * nv), np.int32)
    so = np.zeros(batch + 1, np.int32)
    rc = lib.litevlm_oracle_select_views(batch, nv, _ptr(lx), _ptr(lg), _ptr(tpv), float(w_lex), float(w_logit),
                                         float(threshold), int(min_views), _ptr(mask), _ptr(vo), _ptr(sv), _ptr(so))
    if rc != 0:
        raise OracleError(f"litevlm_oracle_select_views returned {rc}")
    return mask, vo, sv[:int(vo[-1])], so


def project(x_bf16: np.ndarray, gamma, eps: float, w_bf16: np.ndarray, bias=None, head_dim: int = 0,
            positions=None, rope_base: float = 10000.0, lib=None) -> np.ndarray:
    """RoPE(W . RMSNorm(x) + bias) in fp64. x_bf16 [rows, H] and w_bf16 [O, H]
    as uint16 bf16 bits; gamma [H], bias [O] float32; positions int32 [rows].
    Returns float64 [rows, O]."""
    lib = lib or load()
    x = np.ascontiguousarray(x_bf16, dtype=np.uint16)
    w = np.ascontiguousarray(w_bf16, dtype=np.uint16)
    rows, hidden = x.shape
    out_f = w.shape[0]
    g = np.ascontiguousarray(gamma, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    pos = np.ascontiguousarray(np.zeros(rows, np.int32) if positions is None else positions, dtype=np.int32)
    y = np.zeros((rows, out_f), np.float64)
    rc = lib.litevlm_oracle_project(rows, hidden, out_f, _ptr(x), _ptr(g), float(eps), _ptr(w), _ptr(b), head_dim,
                                    _ptr(pos), float(rope_base), _ptr(y))
    if rc != 0:
        raise OracleError(f"litevlm_oracle_project returned {rc}")
    return y


def select(w_inputs: dict, hq: int, hkv: int, head_dim: int, dtype: str, keep_k=None, keep_ratio=0.0,
           gather=("hidden",), lib=None, threads: int = 1):
    """The whole path on one batch: scores, kept indices, offsets and gathered
    rows. threads > 1 computes the scores on that many threads (same bits)."""
    args = (w_inputs["q"], w_inputs["k"], w_inputs["seq_offsets"], w_inputs["text_offsets"], hq, hkv, head_dim,
            dtype, w_inputs.get("q_scale", 1.0), w_inputs.get("k_scale", 1.0))
    s = score(*args, lib=lib) if threads <= 1 else score_threads(*args, threads=threads, lib=lib)
    kept, off = topk(w_inputs["seq_offsets"], s, keep_k=keep_k, keep_ratio=keep_ratio, lib=lib)
    rows = {name: compact(kept, w_inputs[name], lib=lib) for name in gather}
    return s, kept, off, rows
