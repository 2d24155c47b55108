"""Seeded synthetic inputs for the token-selection path.

This module only draws random tensors with the shapes of the paper's
multi-camera workloads (Table 1 and the Training section: 448x448 tiles, 256
visual tokens per tile, up to 12 tiles from 6 cameras, about 142 text tokens).
It holds none of the selection arithmetic, so both the CPU oracle and the CUDA
path can take their inputs from here without sharing any computation.

Two back-ends produce the same shapes:
  * ``make_numpy``: numpy PCG64, platform-deterministic; used for the sizes the
    oracle finishes in seconds.
  * ``make_torch``: a seeded torch generator on a device; used for the full
    bench sizes (gigabytes of K and hidden rows), where a numpy draw would be
    too slow. Its values differ from ``make_numpy`` for the same seed; the full
    size parity tests copy the torch inputs back to the host for the oracle.

Layouts (row-major, contiguous):
  q       [sum_b T_b, Hq,  d]   text-query rows of every request
  k, v    [sum_b N_b, Hkv, d]   visual-token key/value rows
  hidden  [sum_b N_b, hidden]   visual-token hidden states
  seq_offsets / text_offsets    int32 prefix arrays of length B+1
bf16 tensors are carried as uint16 bit patterns on the numpy side and e4m3
tensors as uint8 codes with one float32 scale per tensor (absmax / 448).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace
from typing import Dict, List, Optional, Sequence

import numpy as np

E4M3_MAX = 448.0


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    n_vis: Sequence[int]
    n_txt: Sequence[int]
    hq: int
    hkv: int
    head_dim: int
    hidden: int
    dtype: str  # "bf16" or "e4m3" for q/k; hidden and v are always bf16
    keep_k: Optional[Sequence[int]] = None
    keep_ratio: Optional[float] = None
    gather: Sequence[str] = ("hidden",)
    sigma: float = 1.0  # std of q/k entries
    salient_frac: float = 0.0
    salient_count: int = 0
    salient_gain: float = 3.0
    k_lognormal_sigma: float = 0.0
    seed: int = 0
    description: str = ""

    @property
    def total_vis(self) -> int:
        return int(sum(self.n_vis))

    @property
    def total_txt(self) -> int:
        return int(sum(self.n_txt))

    def seq_offsets(self) -> np.ndarray:
        return _offsets(self.n_vis)

    def text_offsets(self) -> np.ndarray:
        return _offsets(self.n_txt)

    def row_bytes(self) -> Dict[str, int]:
        return {"hidden": self.hidden * 2, "k": self.hkv * self.head_dim * (2 if self.dtype == "bf16" else 1),
                "v": self.hkv * self.head_dim * 2}


def _offsets(lens: Sequence[int]) -> np.ndarray:
    off = np.zeros(len(lens) + 1, dtype=np.int32)
    off[1:] = np.cumsum(np.asarray(lens, dtype=np.int64))
    return off


def workload(name: str, **overrides) -> Workload:
    """The five synthetic workloads, named by what they are.

    tiny        1 request, 2 views x 64 = 128 visual + 16 text tokens, 4 heads x 64,
                hidden 256, 8 salient tokens, keep 32
    single      1 request, 6 views x 256 = 1536 visual + 64 text tokens, 16 heads x 128,
                hidden 2048, 5% salient tokens, keep ratio 0.3
    highres     1 request, 6 views x 1024 = 6144 visual + 128 text tokens, 28 query /
                4 KV heads x 128, hidden 3584, lognormal K norms (sigma 0.5), keep 0.25,
                gathers hidden + K + V
    fp8_ragged  32 requests, 1..6 views x 576 visual, 32..128 text tokens, 32 heads x 128,
                e4m3 q/k with per-tensor scales, hidden 4096, keep 20% per request
    sweep       128 requests x (3456 visual + 64 text), 32 heads x 128, hidden 4096,
                keep ratio 0.1 / 0.2 / 0.3 / 0.5
    """
    if name == "tiny":
        w = Workload("tiny", 1, [128], [16], 4, 4, 64, 256, "bf16", keep_k=[32],
                     sigma=1.0, salient_count=8, seed=0,
                     description="1 x (128 visual + 16 text), 4 heads x 64, keep 32")
    elif name == "single":
        w = Workload("single", 1, [1536], [64], 16, 16, 128, 2048, "bf16", keep_ratio=0.3,
                     sigma=1.0 / math.sqrt(128), salient_frac=0.05, seed=1,
                     description="1 x (6 views x 256 = 1536 visual + 64 text), 16 heads x 128, keep 30%")
    elif name == "highres":
        w = Workload("highres", 1, [6144], [128], 28, 4, 128, 3584, "bf16", keep_ratio=0.25,
                     gather=("hidden", "k", "v"), sigma=1.0 / math.sqrt(128),
                     k_lognormal_sigma=0.5, seed=2,
                     description="1 x (6 views x 1024 = 6144 visual + 128 text), 28/4 GQA heads x 128, keep 25%")
    elif name == "fp8_ragged":
        rng = np.random.Generator(np.random.PCG64(3))
        views = rng.integers(1, 7, size=32)
        txt = rng.integers(32, 129, size=32)
        n_vis = [int(576 * v) for v in views]
        w = Workload("fp8_ragged", 32, n_vis, [int(t) for t in txt], 32, 32, 128, 4096, "e4m3",
                     keep_k=[int(math.floor(0.2 * n)) for n in n_vis],
                     sigma=1.0 / math.sqrt(128), seed=3,
                     description="32 x (1..6 views x 576 visual + 32..128 text), 32 heads x 128, e4m3, keep 20%")
    elif name == "sweep":
        w = Workload("sweep", 128, [3456] * 128, [64] * 128, 32, 32, 128, 4096, "bf16", keep_ratio=0.3,
                     sigma=1.0 / math.sqrt(128), seed=4,
                     description="128 x (6 views x 576 = 3456 visual + 64 text), 32 heads x 128, keep 10/20/30/50%")
    else:
        raise KeyError(f"unknown workload {name!r}")
    return replace(w, **overrides) if overrides else w


def sub_batch(w: Workload, requests: Sequence[int]) -> Workload:
    """The same workload restricted to a subset of requests (shapes only)."""
    kk = None if w.keep_k is None else [w.keep_k[r] for r in requests]
    return replace(w, batch=len(requests), n_vis=[w.n_vis[r] for r in requests],
                   n_txt=[w.n_txt[r] for r in requests], keep_k=kk)


# ----------------------------------------------------------------------------
# numpy back-end
# ----------------------------------------------------------------------------

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float values to bfloat16 (round to nearest even), as uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def f32_to_e4m3(x: np.ndarray):
    """Per-tensor scaled e4m3 codes (uint8) and the float32 scale absmax/448."""
    import torch  # conversion to float8 goes through torch's rounding
    x = np.asarray(x, dtype=np.float32)
    amax = float(np.max(np.abs(x))) if x.size else 1.0
    scale = np.float32(amax / E4M3_MAX if amax > 0 else 1.0)
    t = torch.from_numpy(x / scale).to(torch.float8_e4m3fn)
    return t.view(torch.uint8).numpy().copy(), float(scale)


def _salient_rows(rng, w: Workload, q_f: np.ndarray, k_f: np.ndarray) -> List[np.ndarray]:
    """Overwrite a few K rows per request with a copy of the request's mean
    query direction, scaled to salient_gain times the typical row norm.
    Returns the chosen local positions per request."""
    so, to = w.seq_offsets(), w.text_offsets()
    g = w.hq // w.hkv
    chosen = []
    for b in range(w.batch):
        n = int(so[b + 1] - so[b])
        n_sal = w.salient_count if w.salient_count else int(w.salient_frac * n)
        if n == 0 or n_sal == 0:
            chosen.append(np.zeros(0, np.int64))
            continue
        pos = rng.permutation(n)[:n_sal]
        chosen.append(np.sort(pos))
        qb = q_f[to[b]:to[b + 1]]  # [T, Hq, d]
        for kv in range(w.hkv):
            u = qb[:, kv * g:(kv + 1) * g, :].sum(axis=(0, 1)).astype(np.float64)
            nrm = np.linalg.norm(u)
            if nrm == 0:
                continue
            k_f[so[b] + pos, kv, :] = (w.salient_gain * w.sigma * math.sqrt(w.head_dim) * u / nrm)
    return chosen


def make_numpy(w: Workload, seed: Optional[int] = None, fp32: bool = False) -> Dict[str, object]:
    """Host inputs. With fp32=True, q/k are also returned unrounded as float32
    ("q_f32", "k_f32"), for oracle checks on the exact fp32 draw."""
    rng = np.random.Generator(np.random.PCG64(w.seed if seed is None else seed))
    T, N, d = w.total_txt, w.total_vis, w.head_dim
    q_f = (rng.standard_normal((T, w.hq, d)) * w.sigma).astype(np.float32)
    k_f = (rng.standard_normal((N, w.hkv, d)) * w.sigma).astype(np.float32)
    if w.k_lognormal_sigma > 0:
        k_f *= np.exp(w.k_lognormal_sigma * rng.standard_normal((N, 1, 1))).astype(np.float32)
    salient = _salient_rows(rng, w, q_f, k_f) if (w.salient_count or w.salient_frac) else []
    out: Dict[str, object] = {"seq_offsets": w.seq_offsets(), "text_offsets": w.text_offsets(),
                              "salient": salient}
    if w.dtype == "bf16":
        out["q"], out["k"] = f32_to_bf16_bits(q_f), f32_to_bf16_bits(k_f)
        out["q_scale"] = out["k_scale"] = 1.0
    elif w.dtype == "e4m3":
        out["q"], out["q_scale"] = f32_to_e4m3(q_f)
        out["k"], out["k_scale"] = f32_to_e4m3(k_f)
    else:
        raise ValueError(w.dtype)
    if fp32:
        out["q_f32"], out["k_f32"] = q_f, k_f
    if "v" in w.gather:
        out["v"] = f32_to_bf16_bits(rng.standard_normal((N, w.hkv, d)).astype(np.float32))
    out["hidden"] = f32_to_bf16_bits(rng.standard_normal((N, w.hidden)).astype(np.float32))
    return out


# ----------------------------------------------------------------------------
# torch back-end (device-side draw for the full sizes)
# ----------------------------------------------------------------------------

def make_torch(w: Workload, device, seed: Optional[int] = None, chunk_rows: int = 1 << 16):
    """Device inputs as torch tensors (bf16 / uint8 e4m3 codes, int32 offsets)."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed if seed is None else seed)
    T, N, d = w.total_txt, w.total_vis, w.head_dim

    def normal(rows, cols, scale, dtype):
        out = torch.empty((rows, cols), dtype=dtype, device=device)
        for r0 in range(0, rows, chunk_rows):
            r1 = min(rows, r0 + chunk_rows)
            out[r0:r1] = (torch.randn((r1 - r0, cols), generator=gen, device=device) * scale).to(dtype)
        return out

    q_f = normal(T, w.hq * d, w.sigma, torch.float32).view(T, w.hq, d)
    k_f = normal(N, w.hkv * d, w.sigma, torch.float32).view(N, w.hkv, d)
    if w.k_lognormal_sigma > 0:
        k_f *= torch.exp(w.k_lognormal_sigma * torch.randn((N, 1, 1), generator=gen, device=device))
    if w.salient_count or w.salient_frac:
        so, to = w.seq_offsets(), w.text_offsets()
        g = w.hq // w.hkv
        for b in range(w.batch):
            n = int(so[b + 1] - so[b])
            n_sal = w.salient_count if w.salient_count else int(w.salient_frac * n)
            if n == 0 or n_sal == 0:
                continue
            pos = torch.randperm(n, generator=gen, device=device)[:n_sal] + int(so[b])
            qb = q_f[int(to[b]):int(to[b + 1])].view(-1, w.hkv, g, d).sum(dim=(0, 2))  # [Hkv, d]
            u = qb / qb.norm(dim=-1, keepdim=True).clamp_min(1e-30)
            k_f[pos] = (w.salient_gain * w.sigma * math.sqrt(d) * u).unsqueeze(0)
    out = {"seq_offsets": torch.from_numpy(w.seq_offsets()).to(device),
           "text_offsets": torch.from_numpy(w.text_offsets()).to(device)}
    if w.dtype == "bf16":
        out["q"], out["k"] = q_f.to(torch.bfloat16), k_f.to(torch.bfloat16)
        out["q_scale"] = out["k_scale"] = 1.0
    else:
        for name, x in (("q", q_f), ("k", k_f)):
            amax = float(x.abs().max()) if x.numel() else 1.0
            scale = float(np.float32(amax / E4M3_MAX if amax > 0 else 1.0))
            out[name] = (x / scale).to(torch.float8_e4m3fn).view(torch.uint8)
            out[name + "_scale"] = scale
    del q_f, k_f
    if "v" in w.gather:
        out["v"] = normal(N, w.hkv * d, 1.0, torch.bfloat16).view(N, w.hkv, d)
    out["hidden"] = normal(N, w.hidden, 1.0, torch.bfloat16)
    return out


# ----------------------------------------------------------------------------
# keys of the system prompt and the text tokens (full-key-set scores)
# ----------------------------------------------------------------------------

def context_keys_numpy(w: Workload, sys_lens: Sequence[int], k_scale: float = 1.0, seed: Optional[int] = None,
                       sink_gain: float = 0.0, q_f32: Optional[np.ndarray] = None) -> Dict[str, object]:
    """Key rows of the system prompt ([sum S_b, Hkv, d]) and of the text tokens
    ([sum T_b, Hkv, d]), drawn like the visual keys (normal, std sigma) and
    encoded like them (bf16 bits, or e4m3 codes under the visual keys' scale
    k_scale, clipped to +-448). sink_gain > 0 makes each request's first system
    key an attention sink: each KV head's row points along the request's mean
    query direction u of that head group (q_f32, the unrounded queries), scaled
    so that the mean logit q.k / sqrt(d) of the group's queries is sink_gain."""
    rng = np.random.Generator(np.random.PCG64((w.seed + 1000003) if seed is None else seed))
    so = _offsets(sys_lens)
    S, T, d = int(so[-1]), w.total_txt, w.head_dim
    ks = (rng.standard_normal((S, w.hkv, d)) * w.sigma).astype(np.float32)
    kt = (rng.standard_normal((T, w.hkv, d)) * w.sigma).astype(np.float32)
    if sink_gain > 0 and S > 0:
        to, g = w.text_offsets(), w.hq // w.hkv
        for b in range(len(sys_lens)):
            if sys_lens[b] == 0 or to[b + 1] == to[b]:
                continue
            for kv in range(w.hkv):
                qg = q_f32[to[b]:to[b + 1], kv * g:(kv + 1) * g, :].astype(np.float64)
                u = qg.sum(axis=(0, 1))
                nrm = np.linalg.norm(u)
                if nrm == 0:
                    continue
                u /= nrm
                proj = float(np.mean(qg @ u))  # mean q.u > 0
                ks[so[b], kv] = (sink_gain * math.sqrt(d) / proj * u).astype(np.float32)
    out: Dict[str, object] = {"sys_offsets": so}
    for name, x in (("k_sys", ks), ("k_txt", kt)):
        if w.dtype == "bf16":
            out[name] = f32_to_bf16_bits(x)
        else:
            import torch
            y = np.clip(x / np.float32(k_scale), -E4M3_MAX, E4M3_MAX).astype(np.float32)
            out[name] = torch.from_numpy(y).to(torch.float8_e4m3fn).view(torch.uint8).numpy().copy()
    return out


def context_keys_torch(w: Workload, sys_lens: Sequence[int], device, k_scale: float = 1.0,
                       seed: Optional[int] = None):
    """The same shapes drawn on a device (values differ from the numpy draw)."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed((w.seed + 1000003) if seed is None else seed)
    so = _offsets(sys_lens)
    S, T, d = int(so[-1]), w.total_txt, w.head_dim
    out = {"sys_offsets": torch.from_numpy(so).to(device)}
    for name, rows in (("k_sys", S), ("k_txt", T)):
        x = torch.randn((max(rows, 0), w.hkv, d), generator=gen, device=device) * w.sigma
        if w.dtype == "bf16":
            out[name] = x.to(torch.bfloat16)
        else:
            out[name] = (x / k_scale).clamp(-E4M3_MAX, E4M3_MAX).to(torch.float8_e4m3fn).view(torch.uint8)
    return out


# ----------------------------------------------------------------------------
# patch-selection gating inputs
# ----------------------------------------------------------------------------

def view_gating_numpy(batch: int, num_views: int = 6, seed: int = 5, lexical_p: float = 0.25,
                      logit_sigma: float = 2.0, quantum: float = 0.0):
    """Per-view lexical-mapping scores (1 with probability lexical_p, else 0)
    and module logits (normal, std logit_sigma; rounded to multiples of quantum
    when quantum > 0, which produces ties), float32 [batch, num_views]. The
    paper's setting has 6 cameras of 2 tiles x 256 tokens (12 tiles)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    lex = (rng.random((batch, num_views)) < lexical_p).astype(np.float32)
    lg = rng.standard_normal((batch, num_views)) * logit_sigma
    if quantum > 0:
        lg = np.round(lg / quantum) * quantum
    return lex, lg.astype(np.float32)


# ----------------------------------------------------------------------------
# layer-0 projection inputs (random weights of the decoder layer's shapes)
# ----------------------------------------------------------------------------

def projection_numpy(rows: int, hidden: int, out_features: int, seed: int = 6, bias: bool = False,
                     max_position: int = 4096):
    """Hidden rows x ~ N(0, 1) (bf16 bits), RMSNorm weight gamma ~ U(0.5, 1.5),
    projection weight W ~ N(0, 1/hidden) (bf16 bits, [out, in]), optional bias
    ~ N(0, 0.1), and positions drawn uniformly below max_position."""
    rng = np.random.Generator(np.random.PCG64(seed))
    x = f32_to_bf16_bits(rng.standard_normal((rows, hidden)).astype(np.float32))
    gamma = rng.uniform(0.5, 1.5, hidden).astype(np.float32)
    w = f32_to_bf16_bits((rng.standard_normal((out_features, hidden)) / math.sqrt(hidden)).astype(np.float32))
    b = (rng.standard_normal(out_features) * 0.1).astype(np.float32) if bias else None
    pos = rng.integers(0, max_position, rows).astype(np.int32)
    return x, gamma, w, b, pos
