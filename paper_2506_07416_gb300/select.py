"""Thin ctypes binding of the C-ABI in include/litevlm_select.h.

Argument marshalling only: torch tensors give device pointers and the current
CUDA stream; every step of the path runs in liblitevlm_select.so. There is no
CPU fallback: if the library is missing the import of this module fails.

Names follow the C functions: create / destroy / score / topk / compact /
check_device (litevlm_select_*), plus ``Selector``, a small object that owns
a handle and allocates outputs with torch.
"""
from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
# LITEVLM_LIB may name another build of the library (e.g. the debug variant,
# liblitevlm_select_debug.so); by default the release build in the package
LIB_PATH = os.environ.get("LITEVLM_LIB") or os.path.join(_PKG, "liblitevlm_select.so")

STATUS = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "WORKSPACE", 4: "CUDA", 5: "TIMEOUT",
          6: "DEVICE_BOUNDS"}
DTYPES = {"bf16": 0, "e4m3": 1}


class LitevlmError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status
        self.name = STATUS.get(status, str(status))


class Config(ctypes.Structure):
    _fields_ = [("max_batch", ctypes.c_int32), ("max_total_visual", ctypes.c_int64),
                ("max_total_text", ctypes.c_int64), ("num_q_heads", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("qk_dtype", ctypes.c_int32),
                ("flags", ctypes.c_int32)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; run __graft_entry__.build() (needs nvcc)")
    lib = ctypes.CDLL(LIB_PATH)
    P, i32, i64, f32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
    lib.litevlm_select_create.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(P)]
    lib.litevlm_select_destroy.argtypes = [P]
    lib.litevlm_select_last_error.argtypes = [P]
    lib.litevlm_select_last_error.restype = ctypes.c_char_p
    lib.litevlm_select_last_launches.argtypes = [P]
    lib.litevlm_select_last_launches.restype = ctypes.c_int32
    lib.litevlm_status_string.argtypes = [ctypes.c_int]
    lib.litevlm_status_string.restype = ctypes.c_char_p
    lib.litevlm_select_score.argtypes = [P, i32, P, P, P, P, P, P, f32, f32, P, P]
    lib.litevlm_select_score_full_keys.argtypes = [P, i32, P, P, P, P, P, P, P, P, P, P, f32, f32, P, P]
    lib.litevlm_select_views.argtypes = [P, i32, i32, P, P, P, f32, f32, f32, i32, P, P, P, P, P, P]
    lib.litevlm_select_fold_norm.argtypes = [P, i32, i32, P, P, P, P]
    lib.litevlm_select_rope_table.argtypes = [P, i32, i32, f32, P, P]
    lib.litevlm_select_project.argtypes = [P, i64, i32, i32, P, P, P, f32, i32, P, P, i32, f32, P, P]
    lib.litevlm_select_topk.argtypes = [P, i32, P, P, P, P, P, f32, P, P, P, P]
    lib.litevlm_select_compact.argtypes = [P, i64, P, i64, i32, P, P, P, P]
    lib.litevlm_select_score_topk.argtypes = [P, i32, P, P, P, P, P, P, f32, f32, P, P, P, f32, P, P, P, P]
    lib.litevlm_select_check_device.argtypes = [P, P]
    lib.litevlm_select_host_view.argtypes = [P, P, ctypes.POINTER(P)]
    lib.litevlm_select_score_plan.argtypes = [P, i32, P, P, P]
    lib.litevlm_select_splice.argtypes = [P, i32, P, P, P, P, P, P, P, P, P, P, P, P, i64, P, P, P, P, P]
    lib.litevlm_select_score_noalloc.argtypes = [i32, i32, i32, i32, i32, P, P, P, P, P, P, f32, f32, P, P, P]
    lib.litevlm_select_keep_offsets.argtypes = [i32, P, P, f32, P]
    lib.litevlm_select_set_wait_budget.argtypes = [P, i64]
    lib.litevlm_select_set_debug_flags.argtypes = [P, i32]
    for fn in ("create", "destroy", "score", "score_full_keys", "topk", "compact", "check_device", "score_plan",
               "score_noalloc", "splice", "views", "fold_norm", "rope_table", "project", "score_topk", "host_view",
               "keep_offsets", "set_wait_budget", "set_debug_flags"):
        getattr(lib, "litevlm_select_" + fn).restype = ctypes.c_int
    return lib


LIB = _load()

# every symbol declared in include/litevlm_select.h
EXPORTS = ["litevlm_select_create", "litevlm_select_destroy", "litevlm_select_last_error",
           "litevlm_status_string", "litevlm_select_score", "litevlm_select_topk", "litevlm_select_compact",
           "litevlm_select_check_device", "litevlm_select_score_plan", "litevlm_select_score_noalloc",
           "litevlm_select_splice", "litevlm_select_score_full_keys", "litevlm_select_views",
           "litevlm_select_fold_norm", "litevlm_select_rope_table", "litevlm_select_project",
           "litevlm_select_last_launches", "litevlm_select_score_topk", "litevlm_select_host_view",
           "litevlm_select_keep_offsets", "litevlm_select_set_wait_budget", "litevlm_select_set_debug_flags"]
FLAGS = {"auto": 0, "reread": 1, "resident": 2, "resident_1buf": 8, "resident_2buf": 16, "resident_flat": 64}
# LITEVLM_FLAG_SCORE_SPLIT_QUERIES: resident plans for T > 64 run each head's text rows as two pseudo-heads
QUERY_SPLIT = {"whole": 0, "split": 128}
KERNELS = {1: "score_tc (K re-read per pass)", 2: "score_res (logits resident in TMEM, one head at a time)",
           3: "score_res (logits resident in TMEM, two heads overlapped)",
           4: "score_res (logits resident in TMEM, one head at a time, flattened (request, head) schedule over "
              "every cluster that fits at once)"}
KERNELS.update({k + 3: v + ", each head's text rows as two pseudo-heads" for k, v in list(KERNELS.items())[1:]})


def _check(rc: int, handle) -> None:
    if rc != 0:
        msg = LIB.litevlm_select_last_error(handle)
        raise LitevlmError(rc, (msg or b"").decode())


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _host_i32(a) -> Optional[np.ndarray]:
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        return np.ascontiguousarray(a, dtype=np.int32)
    try:
        import torch
        if isinstance(a, torch.Tensor):
            return np.ascontiguousarray(a.detach().cpu().numpy(), dtype=np.int32)
    except ImportError:
        pass
    return np.ascontiguousarray(np.asarray(a), dtype=np.int32)


def _stream_ptr(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ----------------------------------------------------------------------------
# C functions, one to one
# ----------------------------------------------------------------------------

QUERY_LAST_TOKEN = 32


def create(max_batch: int, max_total_visual: int, max_total_text: int, num_q_heads: int, num_kv_heads: int,
           head_dim: int, qk_dtype: str = "bf16", score_kernel: str = "auto", query: str = "all",
           query_split: str = "whole") -> int:
    """query: "all" (every text token is a query) or "last" (only the last one).
    query_split: "whole", or "split" (resident plans for T > 64 run each head's
    text rows as two pseudo-heads)."""
    cfg = Config(max_batch, max_total_visual, max_total_text, num_q_heads, num_kv_heads, head_dim,
                 DTYPES[qk_dtype], FLAGS[score_kernel] | QUERY_SPLIT[query_split] |
                 (QUERY_LAST_TOKEN if query == "last" else 0))
    h = ctypes.c_void_p()
    _check(LIB.litevlm_select_create(ctypes.byref(cfg), ctypes.byref(h)), None)
    return h.value


def destroy(handle: int) -> None:
    _check(LIB.litevlm_select_destroy(handle), handle)


def score(handle: int, batch: int, q_text, text_offsets_d, text_offsets_h, k_vis, seq_offsets_d, seq_offsets_h,
          q_scale: float, k_scale: float, scores, stream=None) -> None:
    to_h, so_h = _host_i32(text_offsets_h), _host_i32(seq_offsets_h)
    _check(LIB.litevlm_select_score(handle, batch, _ptr(q_text), _ptr(text_offsets_d), _ptr(to_h), _ptr(k_vis),
                                    _ptr(seq_offsets_d), _ptr(so_h), q_scale, k_scale, _ptr(scores),
                                    _stream_ptr(stream)), handle)


def score_full_keys(handle: int, batch: int, q_text, text_offsets_d, text_offsets_h, k_vis, seq_offsets_d,
                    seq_offsets_h, k_sys, sys_offsets_d, sys_offsets_h, k_text, q_scale: float, k_scale: float,
                    scores, stream=None) -> None:
    to_h, so_h, yo_h = _host_i32(text_offsets_h), _host_i32(seq_offsets_h), _host_i32(sys_offsets_h)
    _check(LIB.litevlm_select_score_full_keys(handle, batch, _ptr(q_text), _ptr(text_offsets_d), _ptr(to_h),
                                              _ptr(k_vis), _ptr(seq_offsets_d), _ptr(so_h), _ptr(k_sys),
                                              _ptr(sys_offsets_d), _ptr(yo_h), _ptr(k_text), q_scale, k_scale,
                                              _ptr(scores), _stream_ptr(stream)), handle)


def views(handle: int, batch: int, num_views: int, lexical, logits, tokens_per_view_h, w_lex: float, w_logit: float,
          threshold: float, min_views: int, view_mask, view_offsets, selected_views, seq_offsets,
          seq_offsets_h: Optional[np.ndarray] = None, stream=None) -> None:
    tpv = _host_i32(tokens_per_view_h)
    _check(LIB.litevlm_select_views(handle, batch, num_views, _ptr(lexical), _ptr(logits), _ptr(tpv), w_lex, w_logit,
                                    threshold, min_views, _ptr(view_mask), _ptr(view_offsets), _ptr(selected_views),
                                    _ptr(seq_offsets), _ptr(seq_offsets_h), _stream_ptr(stream)), handle)


def score_topk(handle: int, batch: int, q_text, text_offsets_d, text_offsets_h, k_vis, seq_offsets_d, seq_offsets_h,
               q_scale: float, k_scale: float, scores, keep_k_d, keep_k_h, keep_ratio: float, kept_idx,
               out_offsets_d, out_offsets_h, stream=None) -> None:
    to_h, so_h, kk_h = _host_i32(text_offsets_h), _host_i32(seq_offsets_h), _host_i32(keep_k_h)
    _check(LIB.litevlm_select_score_topk(handle, batch, _ptr(q_text), _ptr(text_offsets_d), _ptr(to_h),
                                         _ptr(k_vis), _ptr(seq_offsets_d), _ptr(so_h), q_scale, k_scale,
                                         _ptr(scores), _ptr(keep_k_d), _ptr(kk_h), keep_ratio, _ptr(kept_idx),
                                         _ptr(out_offsets_d), _ptr(out_offsets_h), _stream_ptr(stream)), handle)


def fold_norm(handle: int, out_features: int, hidden: int, w, gamma, w_folded, stream=None) -> None:
    _check(LIB.litevlm_select_fold_norm(handle, out_features, hidden, _ptr(w), _ptr(gamma), _ptr(w_folded),
                                        _stream_ptr(stream)), handle)


def rope_table(handle: int, max_positions: int, head_dim: int, rope_base: float, table, stream=None) -> None:
    _check(LIB.litevlm_select_rope_table(handle, max_positions, head_dim, rope_base, _ptr(table),
                                         _stream_ptr(stream)), handle)


def project(handle: int, rows: int, hidden: int, out_features: int, x, w_folded, bias, eps: float, head_dim: int,
            positions, table, max_positions: int, y, stream=None, out_scale: float = 0.0) -> None:
    _check(LIB.litevlm_select_project(handle, rows, hidden, out_features, _ptr(x), _ptr(w_folded), _ptr(bias), eps,
                                      head_dim, _ptr(positions), _ptr(table), max_positions, out_scale, _ptr(y),
                                      _stream_ptr(stream)), handle)


def topk(handle: int, batch: int, scores, seq_offsets_d, seq_offsets_h, keep_k_d, keep_k_h, keep_ratio: float,
         kept_idx, out_offsets_d, out_offsets_h: Optional[np.ndarray] = None, stream=None) -> None:
    so_h, kk_h = _host_i32(seq_offsets_h), _host_i32(keep_k_h)
    _check(LIB.litevlm_select_topk(handle, batch, _ptr(scores), _ptr(seq_offsets_d), _ptr(so_h), _ptr(keep_k_d),
                                   _ptr(kk_h), keep_ratio, _ptr(kept_idx), _ptr(out_offsets_d),
                                   _ptr(out_offsets_h), _stream_ptr(stream)), handle)


def compact(handle: int, total_kept: int, kept_idx, src_rows: int, srcs: Sequence, dsts: Sequence,
            row_bytes: Sequence[int], stream=None) -> None:
    n = len(srcs)
    src_arr = (ctypes.c_void_p * n)(*[_ptr(s) for s in srcs])
    dst_arr = (ctypes.c_void_p * n)(*[_ptr(d) for d in dsts])
    rb_arr = (ctypes.c_int64 * n)(*[int(r) for r in row_bytes])
    _check(LIB.litevlm_select_compact(handle, total_kept, _ptr(kept_idx), src_rows, n, src_arr, dst_arr, rb_arr,
                                      _stream_ptr(stream)), handle)


def splice(handle: int, batch: int, sys_rows, sys_offsets_d, sys_offsets_h, vis_rows, seq_offsets_d, seq_offsets_h,
           kept_idx, kept_offsets_d, kept_offsets_h, txt_rows, text_offsets_d, text_offsets_h, row_bytes: int,
           out_rows, out_offsets_d, position_ids, out_offsets_h: Optional[np.ndarray] = None, stream=None) -> None:
    so, vo, ko, to = (_host_i32(a) for a in (sys_offsets_h, seq_offsets_h, kept_offsets_h, text_offsets_h))
    _check(LIB.litevlm_select_splice(handle, batch, _ptr(sys_rows), _ptr(sys_offsets_d), _ptr(so), _ptr(vis_rows),
                                     _ptr(seq_offsets_d), _ptr(vo), _ptr(kept_idx), _ptr(kept_offsets_d), _ptr(ko),
                                     _ptr(txt_rows), _ptr(text_offsets_d), _ptr(to), int(row_bytes), _ptr(out_rows),
                                     _ptr(out_offsets_d), _ptr(out_offsets_h), _ptr(position_ids),
                                     _stream_ptr(stream)), handle)


def host_view(handle: int, host_ptr: int) -> int:
    """litevlm_select_host_view: the device address of pinned host memory."""
    out = ctypes.c_void_p()
    _check(LIB.litevlm_select_host_view(handle, host_ptr, ctypes.byref(out)), handle)
    return int(out.value)


def check_device(handle: int, stream=None) -> None:
    _check(LIB.litevlm_select_check_device(handle, _stream_ptr(stream)), handle)


def keep_offsets(seq_offsets_h, keep_k_h=None, keep_ratio: float = 0.0) -> np.ndarray:
    """litevlm_select_keep_offsets: prefix of the kept-token counts k_b (host only)."""
    so = _host_i32(seq_offsets_h)
    kk = _host_i32(keep_k_h)
    out = np.zeros(len(so), np.int32)
    _check(LIB.litevlm_select_keep_offsets(len(so) - 1, _ptr(so), _ptr(kk), keep_ratio, _ptr(out)), None)
    return out


def set_wait_budget(handle: int, cycles: int) -> None:
    """litevlm_select_set_wait_budget: clock cycles each device-side wait may take (0: default)."""
    _check(LIB.litevlm_select_set_wait_budget(handle, int(cycles)), handle)


DEBUG_STALL_SCORE = 1


def set_debug_flags(handle: int, flags: int) -> None:
    """litevlm_select_set_debug_flags: switches for tests of the failure path (0: off)."""
    _check(LIB.litevlm_select_set_debug_flags(handle, int(flags)), handle)


def score_noalloc(num_q_heads: int, num_kv_heads: int, head_dim: int, qk_dtype: str, batch: int, q_text,
                  text_offsets_d, text_offsets_h, k_vis, seq_offsets_d, seq_offsets_h, q_scale: float,
                  k_scale: float, scores, err_d, stream=None) -> None:
    """litevlm_select_score_noalloc: no handle, scratch in the library's static device arrays."""
    to_h, so_h = _host_i32(text_offsets_h), _host_i32(seq_offsets_h)
    _check(LIB.litevlm_select_score_noalloc(num_q_heads, num_kv_heads, head_dim, DTYPES[qk_dtype], batch,
                                            _ptr(q_text), _ptr(text_offsets_d), _ptr(to_h), _ptr(k_vis),
                                            _ptr(seq_offsets_d), _ptr(so_h), q_scale, k_scale, _ptr(scores),
                                            _ptr(err_d), _stream_ptr(stream)), None)


def score_plan(handle: int, batch: int, text_offsets_h, seq_offsets_h):
    """(kernel, cluster, tiles_per_cta, groups) litevlm_select_score would launch."""
    to_h, so_h = _host_i32(text_offsets_h), _host_i32(seq_offsets_h)
    out = np.zeros(4, np.int32)
    _check(LIB.litevlm_select_score_plan(handle, batch, _ptr(to_h), _ptr(so_h), _ptr(out)), handle)
    return tuple(int(v) for v in out)


# ----------------------------------------------------------------------------
# convenience object (allocates outputs with torch; still marshalling only)
# ----------------------------------------------------------------------------

class Selector:
    """Owns one handle. Tensors are torch CUDA tensors laid out as in the C header."""

    def __init__(self, max_batch: int, max_total_visual: int, max_total_text: int, num_q_heads: int,
                 num_kv_heads: int, head_dim: int, qk_dtype: str = "bf16", score_kernel: str = "auto",
                 query: str = "all", query_split: str = "whole"):
        self.handle = create(max_batch, max_total_visual, max_total_text, num_q_heads, num_kv_heads, head_dim,
                             qk_dtype, score_kernel, query, query_split)
        self.qk_dtype = qk_dtype

    def close(self) -> None:
        if self.handle:
            destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def score(self, q, text_offsets, k, seq_offsets, q_scale=1.0, k_scale=1.0, out=None, text_offsets_h=None,
              seq_offsets_h=None, stream=None):
        import torch
        so_h = _host_i32(seq_offsets if seq_offsets_h is None else seq_offsets_h)
        to_h = _host_i32(text_offsets if text_offsets_h is None else text_offsets_h)
        if out is None:
            out = torch.empty(int(so_h[-1]), dtype=torch.float32, device=k.device)
        score(self.handle, len(so_h) - 1, q, text_offsets, to_h, k, seq_offsets, so_h, q_scale, k_scale, out,
              stream)
        return out

    def score_full_keys(self, q, text_offsets, k, seq_offsets, k_sys, sys_offsets, k_text, q_scale=1.0,
                        k_scale=1.0, out=None, text_offsets_h=None, seq_offsets_h=None, sys_offsets_h=None,
                        stream=None):
        """Scores with the softmax over [system; visual; causal text] keys."""
        import torch
        so_h = _host_i32(seq_offsets if seq_offsets_h is None else seq_offsets_h)
        to_h = _host_i32(text_offsets if text_offsets_h is None else text_offsets_h)
        yo_h = _host_i32(sys_offsets if sys_offsets_h is None else sys_offsets_h)
        if out is None:
            out = torch.empty(int(so_h[-1]), dtype=torch.float32, device=k.device)
        score_full_keys(self.handle, len(so_h) - 1, q, text_offsets, to_h, k, seq_offsets, so_h, k_sys, sys_offsets,
                        yo_h, k_text, q_scale, k_scale, out, stream)
        return out

    def select_views(self, lexical, logits, tokens_per_view, w_lex: float, w_logit: float, threshold: float,
                     min_views: int = 0, stream=None):
        """Patch-selection gating on float32 CUDA tensors [B, V]. Returns
        (view_mask, view_offsets, selected_views, seq_offsets device tensors,
        seq_offsets host numpy; the call synchronises to fill the latter)."""
        import torch
        batch, nv = lexical.shape
        dev = lexical.device
        mask = torch.empty((max(batch, 1), nv), dtype=torch.uint8, device=dev)
        vo = torch.empty(batch + 1, dtype=torch.int32, device=dev)
        sv = torch.empty(max(batch * nv, 1), dtype=torch.int32, device=dev)
        so = torch.empty(batch + 1, dtype=torch.int32, device=dev)
        so_h = np.zeros(batch + 1, np.int32)
        views(self.handle, batch, nv, lexical, logits, tokens_per_view, w_lex, w_logit, threshold, min_views, mask,
              vo, sv, so, so_h, stream)
        return mask[:batch], vo, sv, so, so_h

    def score_topk(self, q, text_offsets, k, seq_offsets, q_scale=1.0, k_scale=1.0, keep_k=None,
                   keep_ratio: float = 0.0, text_offsets_h=None, seq_offsets_h=None, stream=None, out=None,
                   kept_idx=None, out_offsets=None):
        """Scores and top-k in one call. Returns (scores, kept_idx, out_offsets
        device, out_offsets host numpy); out / kept_idx / out_offsets are
        optional caller buffers."""
        import torch
        so_h = _host_i32(seq_offsets if seq_offsets_h is None else seq_offsets_h)
        to_h = _host_i32(text_offsets if text_offsets_h is None else text_offsets_h)
        batch = len(so_h) - 1
        kk_h = _host_i32(keep_k)
        kk_d = None
        if kk_h is not None:
            kk_d = keep_k if isinstance(keep_k, torch.Tensor) and keep_k.is_cuda else \
                torch.from_numpy(kk_h).to(k.device)
        total = int(keep_offsets(so_h, kk_h, keep_ratio)[-1])
        scores = out if out is not None else torch.empty(max(1, int(so_h[-1])), dtype=torch.float32, device=k.device)
        kept = kept_idx if kept_idx is not None else torch.empty(max(total, 1), dtype=torch.int32, device=k.device)
        off_d = out_offsets if out_offsets is not None else torch.empty(batch + 1, dtype=torch.int32, device=k.device)
        off_h = np.zeros(batch + 1, np.int32)
        score_topk(self.handle, batch, q, text_offsets, to_h, k, seq_offsets, so_h, q_scale, k_scale, scores, kk_d,
                   kk_h, keep_ratio, kept, off_d, off_h, stream)
        self._keep_alive = kk_d
        return scores[:int(so_h[-1])], kept[:int(off_h[-1])], off_d, off_h

    def fold_norm(self, w, gamma, stream=None):
        """bf16 W * gamma (per input column) for project()."""
        import torch
        out = torch.empty_like(w)
        fold_norm(self.handle, w.shape[0], w.shape[1], w, gamma, out, stream)
        return out

    def rope_table(self, max_positions: int, head_dim: int, rope_base: float, device="cuda", stream=None):
        import torch
        t = torch.empty((max_positions, head_dim // 2, 2), dtype=torch.float32, device=device)
        rope_table(self.handle, max_positions, head_dim, rope_base, t, stream)
        return t

    def project(self, x, w_folded, bias=None, eps: float = 1e-6, head_dim: int = 0, positions=None, table=None,
                out=None, stream=None, out_scale: float = 0.0):
        """y = RoPE(RMS-scale(x) . w_folded^T + bias): bf16 [rows, out_features],
        or uint8 e4m3 codes of y / out_scale when out_scale > 0."""
        import torch
        rows, hidden = x.shape
        out_f = w_folded.shape[0]
        if out is None:
            out = torch.empty((rows, out_f), dtype=torch.uint8 if out_scale > 0 else torch.bfloat16,
                              device=x.device)
        project(self.handle, rows, hidden, out_f, x, w_folded, bias, eps, head_dim, positions, table,
                0 if table is None else table.shape[0], out, stream, out_scale)
        return out

    def topk(self, scores, seq_offsets, keep_k=None, keep_ratio: float = 0.0, seq_offsets_h=None, kept_idx=None,
             out_offsets=None, stream=None):
        """Returns (kept_idx, out_offsets device tensor, out_offsets host numpy)."""
        import torch
        so_h = _host_i32(seq_offsets if seq_offsets_h is None else seq_offsets_h)
        batch = len(so_h) - 1
        kk_h = _host_i32(keep_k)
        kk_d = None
        if kk_h is not None:
            kk_d = keep_k if isinstance(keep_k, torch.Tensor) and keep_k.is_cuda else \
                torch.from_numpy(kk_h).to(scores.device)
        off_h = np.zeros(batch + 1, dtype=np.int32)
        total = int(keep_offsets(so_h, kk_h, keep_ratio)[-1])
        if kept_idx is None:
            kept_idx = torch.empty(max(total, 1), dtype=torch.int32, device=scores.device)
        if out_offsets is None:
            out_offsets = torch.empty(batch + 1, dtype=torch.int32, device=scores.device)
        topk(self.handle, batch, scores, seq_offsets, so_h, kk_d, kk_h, keep_ratio, kept_idx, out_offsets, off_h,
             stream)
        self._keep_alive = kk_d
        return kept_idx[:int(off_h[-1])], out_offsets, off_h

    def compact(self, kept_idx, total_kept: int, srcs: Sequence, dsts: Optional[List] = None, stream=None):
        """Gathers the kept rows of each source into the device. A source in
        pinned host memory is read through its device view, so only its kept
        rows cross the host link."""
        import torch
        rows = [s.shape[0] for s in srcs]
        if dsts is None:
            dsts = [torch.empty((max(total_kept, 0),) + tuple(s.shape[1:]), dtype=s.dtype, device=kept_idx.device)
                    for s in srcs]
        rb = [s[0].numel() * s.element_size() if s.shape[0] else 1 for s in srcs]
        src_ptrs = [self.host_view(s) if s.device.type == "cpu" else s for s in srcs]
        compact(self.handle, total_kept, kept_idx, min(rows) if rows else 0, src_ptrs, dsts, rb, stream)
        return dsts

    def host_view(self, t) -> int:
        """Device address of a pinned host tensor (or host pointer)."""
        return host_view(self.handle, _ptr(t))

    def splice(self, sys_rows, sys_offsets, vis_rows, seq_offsets, kept_idx, kept_offsets, txt_rows, text_offsets,
               stream=None):
        """[system; kept visual; text] rows per request and their original
        position ids. Rows are 2-D torch CUDA tensors with equal row sizes;
        offsets are int32 CUDA tensors. Returns (rows, out_offsets, out_offsets
        host numpy, position_ids)."""
        import torch
        so, vo, ko, to = (_host_i32(a) for a in (sys_offsets, seq_offsets, kept_offsets, text_offsets))
        batch = len(so) - 1
        total = int(so[-1] + ko[-1] + to[-1])
        ref = next(r for r in (sys_rows, vis_rows, txt_rows) if r is not None)
        rb = ref[0].numel() * ref.element_size() if ref.shape[0] else ref.element_size() * int(np.prod(ref.shape[1:]))
        out = torch.empty((max(total, 1),) + tuple(ref.shape[1:]), dtype=ref.dtype, device=ref.device)
        pos = torch.empty(max(total, 1), dtype=torch.int32, device=ref.device)
        off_d = torch.empty(batch + 1, dtype=torch.int32, device=ref.device)
        off_h = np.zeros(batch + 1, np.int32)
        splice(self.handle, batch, sys_rows, sys_offsets, so, vis_rows, seq_offsets, vo, kept_idx, kept_offsets, ko,
               txt_rows, text_offsets, to, rb, out, off_d, pos, off_h, stream)
        return out[:total], off_d, off_h, pos[:total]

    def check_device(self, stream=None) -> None:
        check_device(self.handle, stream)

    def set_wait_budget(self, cycles: int) -> None:
        set_wait_budget(self.handle, cycles)

    def set_debug_flags(self, flags: int) -> None:
        set_debug_flags(self.handle, flags)

    def score_plan(self, text_offsets_h, seq_offsets_h):
        so = _host_i32(seq_offsets_h)
        return score_plan(self.handle, len(so) - 1, text_offsets_h, so)
