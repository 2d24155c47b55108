"""Helpers for the GPU tests: move seeded host inputs to the device and compare
GPU results with the oracle under the tolerances of the parity bar."""
from __future__ import annotations

import numpy as np

# Relative tolerance per element: |gpu - oracle| <= rtol * |oracle| + 1e-30.
RTOL = {"bf16": 2e-3, "e4m3": 3e-2}


def to_device(x: dict, w, device="cuda") -> dict:
    import torch
    out = {}
    for name in ("q", "k", "v", "hidden"):
        if name not in x:
            continue
        a = x[name]
        if a.dtype == np.uint16:
            out[name] = torch.from_numpy(a.view(np.int16).copy()).view(torch.bfloat16).to(device)
        else:
            out[name] = torch.from_numpy(a.copy()).to(device)
    for name in ("seq_offsets", "text_offsets"):
        out[name] = torch.from_numpy(np.ascontiguousarray(x[name], dtype=np.int32)).to(device)
    out["q_scale"] = x.get("q_scale", 1.0)
    out["k_scale"] = x.get("k_scale", 1.0)
    return out


def to_host(xd: dict) -> dict:
    """Device inputs back to the host layout the oracle reads (bf16 as uint16 bits)."""
    import torch
    out = {}
    for name, t in xd.items():
        if isinstance(t, torch.Tensor):
            if t.dtype == torch.bfloat16:
                out[name] = t.view(torch.int16).cpu().numpy().view(np.uint16)
            else:
                out[name] = t.cpu().numpy()
        else:
            out[name] = t
    return out


def rel_err(g: np.ndarray, o: np.ndarray) -> float:
    g = np.asarray(g, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    if g.size == 0:
        return 0.0
    return float(np.max(np.abs(g - o) / (np.abs(o) + 1e-30)))


def assert_scores_close(g, o, dtype: str):
    err = rel_err(g, o)
    assert err <= RTOL[dtype], f"max relative error {err:.3e} > {RTOL[dtype]}"
    return err


def sub_offsets(offsets: np.ndarray, requests) -> np.ndarray:
    lens = np.diff(np.asarray(offsets, dtype=np.int64))[list(requests)]
    return np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)


def gather_rows(a: np.ndarray, offsets: np.ndarray, requests) -> np.ndarray:
    return np.concatenate([a[offsets[b]:offsets[b + 1]] for b in requests], axis=0)
