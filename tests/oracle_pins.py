"""Pins of the CPU oracle to facts that do not come from the oracle itself.

Each ``pin_*`` function takes a loaded oracle library and raises AssertionError
when the oracle disagrees with the fact it checks. ``test_oracle_pins.py`` runs
them on the real oracle; ``test_oracle_mutations.py`` runs them on copies of the
oracle with a planted mistake and expects at least one to fail for every mistake.

Sources of truth used here (none of them is the oracle's own formula):
  * a hand-worked example (2 heads, 4 visual tokens) with closed-form scores;
  * closed forms: identical keys give uniform scores 1/N;
  * a special case that is a library routine: one head and one query give
    scipy.special.softmax of the scaled logits;
  * invariants: softmax rows sum to 1, a request's scores sum to 1, permuting
    visual tokens permutes the scores, replicating grouped K heads (GQA -> MHA)
    leaves the scores unchanged, salient keys aligned with the queries rank first;
  * brute force: top-k against Python's sorted() on small inputs with ties, -0, NaN;
  * the paper's Table 1 token counts (ratio meaning and rounding);
  * torch's own bf16 and float8_e4m3fn decoders;
  * numpy fancy indexing for the gather.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

import oracle
from paper_2506_07416_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _bf16(x) -> np.ndarray:
    return inputs.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def _bf16_value(bits: np.ndarray) -> np.ndarray:
    return inputs.bf16_bits_to_f32(bits).astype(np.float64)


# ---------------------------------------------------------------------------
# element decoders
# ---------------------------------------------------------------------------

def pin_bf16_decode(lib):
    import torch
    codes = np.arange(0, 1 << 16, 97, dtype=np.uint16)  # strided sweep over every exponent
    codes = np.concatenate([codes, np.array([0x0000, 0x8000, 0x3F80, 0xBF80, 0x7F80, 0xFF80, 0x0001, 0x7F7F],
                                            dtype=np.uint16)])
    got = oracle.decode("bf16", codes, lib=lib)
    ref = torch.from_numpy(codes.view(np.int16).copy()).view(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(got, ref)


def pin_e4m3_decode(lib):
    import torch
    codes = np.arange(256, dtype=np.uint8)
    got = oracle.decode("e4m3", codes, lib=lib)
    ref = torch.from_numpy(codes.copy()).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    np.testing.assert_array_equal(got, ref)
    assert got[0x7E] == 448.0 and got[0x01] == 2.0 ** -9 and np.isnan(got[0x7F])


# ---------------------------------------------------------------------------
# scores
# ---------------------------------------------------------------------------

def worked_example():
    """2 query/key heads, d = 4 (logit scale 1/2), 2 text and 4 visual tokens.

    Head 0: q0 = [2,0,0,0], q1 = [0,2,0,0]; k0 = [1,0,0,0], k1 = [0,1,0,0],
    k2 = k3 = 0, so the logit rows are [1,0,0,0] and [0,1,0,0].
    Head 1: both queries are zero, so every softmax entry is 1/4 whatever the keys.
    score0 = score1 = (e/(e+3) + 1/(e+3) + 1/2) / 4 and score2 = score3 = (2/(e+3) + 1/2) / 4.
    """
    q = np.zeros((2, 2, 4), np.float32)
    q[0, 0, 0] = 2.0
    q[1, 0, 1] = 2.0
    k = np.zeros((4, 2, 4), np.float32)
    k[0, 0, 0] = 1.0
    k[1, 0, 1] = 1.0
    k[:, 1, :] = np.array([[0.5, -1.0, 2.0, 0.25], [3.0, 0.0, -0.5, 1.0],
                           [-2.0, 1.5, 0.75, 0.0], [1.0, 1.0, 1.0, -1.0]], np.float32)
    e = math.e
    hi = (e / (e + 3) + 1 / (e + 3) + 0.5) / 4
    lo = (2 / (e + 3) + 0.5) / 4
    return q, k, np.array([hi, hi, lo, lo])


def pin_worked_example(lib):
    q, k, expect = worked_example()
    so, to = np.array([0, 4], np.int32), np.array([0, 2], np.int32)
    # the same example with the two heads swapped must give the same scores
    qs, ks = q[:, ::-1, :].copy(), k[:, ::-1, :].copy()
    for dtype, qq, kk in (("f32", q, k), ("bf16", _bf16(q), _bf16(k)), ("f32", qs, ks)):
        s, s64, rows, _ = oracle.score(qq, kk, so, to, 2, 2, 4, dtype, lib=lib, details=True)
        np.testing.assert_allclose(s64, expect, rtol=1e-14, atol=0)
        np.testing.assert_array_equal(s, expect.astype(np.float32))
        np.testing.assert_allclose(rows, 1.0, rtol=0, atol=1e-14)
        assert abs(s64.sum() - 1.0) < 1e-14
        kept, off = oracle.topk(so, s, keep_k=[1], lib=lib)
        assert kept.tolist() == [0] and off.tolist() == [0, 1]
        kept, off = oracle.topk(so, s, keep_k=[3], lib=lib)
        assert kept.tolist() == [0, 1, 2] and off.tolist() == [0, 3]


def pin_uniform_keys(lib):
    """Identical key rows: every logit of a row is equal, so every score is 1/N
    and the top-k is the first k indices (the tie-break)."""
    rng = np.random.Generator(np.random.PCG64(11))
    n, t, hq, hkv, d = 37, 5, 6, 3, 8
    q = rng.standard_normal((t, hq, d)).astype(np.float32)
    k = np.broadcast_to(rng.standard_normal((1, hkv, d)).astype(np.float32), (n, hkv, d)).copy()
    so, to = np.array([0, n], np.int32), np.array([0, t], np.int32)
    s, s64, _, _ = oracle.score(q, k, so, to, hq, hkv, d, "f32", lib=lib, details=True)
    np.testing.assert_allclose(s64, 1.0 / n, rtol=1e-13)
    assert np.all(s == s[0])
    kept, _ = oracle.topk(so, s, keep_k=[9], lib=lib)
    assert kept.tolist() == list(range(9))


def pin_single_query_is_softmax(lib):
    """One head and one query: the score vector is softmax(q.K^T / sqrt(d))."""
    from scipy.special import softmax
    rng = np.random.Generator(np.random.PCG64(12))
    n, d = 50, 16
    q = _bf16(rng.standard_normal((1, 1, d)) * 0.7)
    k = _bf16(rng.standard_normal((n, 1, d)) * 0.7)
    so, to = np.array([0, n], np.int32), np.array([0, 1], np.int32)
    _, s64, _, lse = oracle.score(q, k, so, to, 1, 1, d, "bf16", lib=lib, details=True)
    logits = _bf16_value(k)[:, 0, :] @ _bf16_value(q)[0, 0, :] / math.sqrt(d)
    np.testing.assert_allclose(s64, softmax(logits), rtol=1e-12, atol=0)
    from scipy.special import logsumexp
    np.testing.assert_allclose(lse, [logsumexp(logits)], rtol=1e-13)


def _ragged(seed, hq, hkv, d, n_vis, n_txt, sigma=0.6):
    rng = np.random.Generator(np.random.PCG64(seed))
    q = rng.standard_normal((sum(n_txt), hq, d)).astype(np.float32) * sigma
    k = rng.standard_normal((sum(n_vis), hkv, d)).astype(np.float32) * sigma
    so = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int32)
    to = np.concatenate([[0], np.cumsum(n_txt)]).astype(np.int32)
    return q, k, so, to


def pin_row_and_total_sums(lib):
    q, k, so, to = _ragged(13, 4, 2, 16, [20, 0, 33, 7], [3, 2, 5, 1])
    _, s64, rows, _ = oracle.score(q, k, so, to, 4, 2, 16, "f32", lib=lib, details=True)
    row_req = np.repeat(np.arange(4), 4 * np.diff(to))
    np.testing.assert_allclose(rows[row_req != 1], 1.0, rtol=0, atol=1e-13)
    for b in range(4):
        if so[b + 1] > so[b]:
            assert abs(s64[so[b]:so[b + 1]].sum() - 1.0) < 1e-13


def pin_batch_equals_single_requests(lib):
    """Requests are independent: scoring a ragged batch gives, for each request,
    the scores of that request scored alone."""
    hq, hkv, d = 4, 2, 16
    n_vis, n_txt = [13, 0, 40, 9], [3, 2, 5, 1]
    q, k, so, to = _ragged(22, hq, hkv, d, n_vis, n_txt)
    _, whole, _, _ = oracle.score(q, k, so, to, hq, hkv, d, "f32", lib=lib, details=True)
    for b in range(len(n_vis)):
        if n_vis[b] == 0:
            continue
        qb, kb = q[to[b]:to[b + 1]], k[so[b]:so[b + 1]]
        _, alone, _, _ = oracle.score(qb, kb, [0, n_vis[b]], [0, n_txt[b]], hq, hkv, d, "f32", lib=lib,
                                      details=True)
        np.testing.assert_array_equal(whole[so[b]:so[b + 1]], alone)


def pin_permutation_equivariance(lib):
    q, k, so, to = _ragged(14, 4, 4, 16, [41], [6])
    perm = np.random.Generator(np.random.PCG64(15)).permutation(41)
    _, a, _, _ = oracle.score(q, k, so, to, 4, 4, 16, "f32", lib=lib, details=True)
    _, b, _, _ = oracle.score(q, k[perm], so, to, 4, 4, 16, "f32", lib=lib, details=True)
    np.testing.assert_allclose(b, a[perm], rtol=1e-12)


def pin_gqa_replication(lib):
    """Query head h reads key head floor(h / G): replicating each key head G
    times in order (GQA -> MHA) must not change the scores."""
    hq, hkv, d = 6, 2, 16
    q, k, so, to = _ragged(16, hq, hkv, d, [29, 18], [4, 3])
    _, a, _, _ = oracle.score(q, k, so, to, hq, hkv, d, "f32", lib=lib, details=True)
    k_rep = np.repeat(k, hq // hkv, axis=1)
    _, b, _, _ = oracle.score(q, k_rep, so, to, hq, hq, d, "f32", lib=lib, details=True)
    np.testing.assert_allclose(a, b, rtol=1e-12)


def pin_scale_placement(lib):
    """The per-tensor scales multiply the logits: (2q, k) with scales 1 equals
    (q, k) with q_scale 2, and likewise for k (powers of two are exact)."""
    q, k, so, to = _ragged(17, 2, 2, 8, [23], [3])
    _, a, _, _ = oracle.score(2 * q, k, so, to, 2, 2, 8, "f32", lib=lib, details=True)
    _, b, _, _ = oracle.score(q, k, so, to, 2, 2, 8, "f32", q_scale=2.0, lib=lib, details=True)
    _, c, _, _ = oracle.score(q, 2 * k, so, to, 2, 2, 8, "f32", lib=lib, details=True)
    _, e, _, _ = oracle.score(q, k, so, to, 2, 2, 8, "f32", k_scale=2.0, lib=lib, details=True)
    np.testing.assert_allclose(b, a, rtol=1e-13)
    np.testing.assert_allclose(e, c, rtol=1e-13)
    np.testing.assert_allclose(a, c, rtol=1e-13)


def pin_e4m3_scores(lib):
    """e4m3 codes with scales score like the decoded values in f32 (e4m3 values
    and power-of-two scales are exact in f32)."""
    import torch
    q, k, so, to = _ragged(18, 2, 1, 16, [31], [4], sigma=2.0)
    q8 = torch.from_numpy(q).to(torch.float8_e4m3fn)
    k8 = torch.from_numpy(k).to(torch.float8_e4m3fn)
    qv, kv = q8.to(torch.float32).numpy(), k8.to(torch.float32).numpy()
    _, a, _, _ = oracle.score(q8.view(torch.uint8).numpy(), k8.view(torch.uint8).numpy(), so, to, 2, 1, 16,
                              "e4m3", q_scale=0.5, k_scale=0.25, lib=lib, details=True)
    _, b, _, _ = oracle.score(qv * 0.5, kv * 0.25, so, to, 2, 1, 16, "f32", lib=lib, details=True)
    np.testing.assert_allclose(a, b, rtol=1e-13)


def pin_salient_tokens_rank_first(lib):
    """Keys aligned with the mean query direction get the largest logits, so
    the tiny workload's 8 salient tokens are the top 8 (sign of the logit)."""
    w = inputs.workload("tiny")
    x = inputs.make_numpy(w)
    s = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, "bf16", lib=lib)
    pos = x["salient"][0]
    top = np.sort(np.argsort(-s.astype(np.float64), kind="stable")[:w.salient_count])
    assert top.tolist() == pos.tolist()


# ---------------------------------------------------------------------------
# top-k
# ---------------------------------------------------------------------------

def brute_topk(scores: np.ndarray, k: int):
    def key(j):
        v = float(scores[j])
        return (1, 0.0, j) if math.isnan(v) else (0, -v, j)
    return sorted(sorted(range(len(scores)), key=key)[:k])


def pin_topk_bruteforce(lib):
    rng = np.random.Generator(np.random.PCG64(19))
    specials = np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 1e-38, -1e-38], np.float32)
    for trial in range(300):
        n = int(rng.integers(1, 65))
        pool = rng.choice(rng.standard_normal(max(1, n // 3)).astype(np.float32), size=n)
        m = rng.random(n) < 0.2
        pool[m] = rng.choice(specials, size=int(m.sum()))
        k = int(rng.integers(0, n + 1))
        so = np.array([0, n], np.int32)
        kept, off = oracle.topk(so, pool, keep_k=[k], lib=lib)
        assert kept.tolist() == brute_topk(pool, k), (trial, pool.tolist(), k)
        assert off.tolist() == [0, k]


def pin_topk_batch_and_ratio(lib):
    rng = np.random.Generator(np.random.PCG64(20))
    n_vis = [10, 0, 25, 1, 64]
    so = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int32)
    s = np.round(rng.standard_normal(so[-1]), 1).astype(np.float32)  # many ties
    for r in (0.0, 0.1, 0.3, 0.5, 0.999, 1.0):
        kept, off = oracle.topk(so, s, keep_ratio=r, lib=lib)
        ks = [int(math.floor(float(np.float32(r)) * n)) for n in n_vis]
        assert np.diff(off).tolist() == ks
        exp = []
        for b in range(len(n_vis)):
            exp += [so[b] + j for j in brute_topk(s[so[b]:so[b + 1]], ks[b])]
        assert kept.tolist() == exp


def pin_table1_token_counts(lib):
    """Table 1: r is the kept fraction of visual tokens and k rounds down."""
    with open(os.path.join(GOLDEN, "table1_token_counts.json")) as f:
        g = json.load(f)
    for row in g["rows"]:
        n = int(round(row["tiles"] * g["visual_tokens_per_tile"]))
        kept = oracle.keep_count(n, row["r"], lib=lib)
        assert kept + g["text_tokens"] == row["input_tokens"], row


def pin_compact(lib):
    rng = np.random.Generator(np.random.PCG64(21))
    src = rng.integers(0, 256, size=(40, 24), dtype=np.uint8)
    idx = np.sort(rng.choice(40, size=17, replace=False)).astype(np.int32)
    np.testing.assert_array_equal(oracle.compact(idx, src, lib=lib), src[idx])
    hid = _bf16(rng.standard_normal((40, 8)))
    np.testing.assert_array_equal(oracle.compact(idx, hid, lib=lib), hid[idx])


# ---------------------------------------------------------------------------
# full causal key set in the softmax normaliser
# ---------------------------------------------------------------------------

def pin_full_keys_worked_example(lib):
    """The worked example with one system key and the two text tokens' keys in
    the normaliser. Head 0's system and text keys are zero (logit 0); head 1's
    queries are zero, so all its logits are 0 whatever the keys. Row i of a head
    sees 1 system key, the 4 visual keys and i + 1 text keys:
      head 0: row 0 [e,1,1,1] / (e+5), row 1 [1,e,1,1] / (e+6)
      head 1: row 0 1/6 each, row 1 1/7 each."""
    q, k, _ = worked_example()
    rng = np.random.Generator(np.random.PCG64(29))
    k_sys = np.zeros((1, 2, 4), np.float32)
    k_txt = np.zeros((2, 2, 4), np.float32)
    k_sys[:, 1, :] = rng.standard_normal((1, 4))
    k_txt[:, 1, :] = rng.standard_normal((2, 4))
    e = math.e
    common = 1 / 6 + 1 / 7
    expect = np.array([(e / (e + 5) + 1 / (e + 6) + common) / 4, (1 / (e + 5) + e / (e + 6) + common) / 4,
                       (1 / (e + 5) + 1 / (e + 6) + common) / 4, (1 / (e + 5) + 1 / (e + 6) + common) / 4])
    s, s64, share = oracle.score_full(q, k, k_sys, k_txt, [0, 4], [0, 2], [0, 1], 2, 2, 4, "f32", lib=lib,
                                      details=True)
    np.testing.assert_allclose(s64, expect, rtol=1e-14, atol=0)
    np.testing.assert_allclose(share, [(e + 3) / (e + 5), (e + 3) / (e + 6), 4 / 6, 4 / 7], rtol=1e-14)


def pin_full_keys_equal_duplicated_visual_keys(lib):
    """With one text token per request, extra keys that copy visual keys act as
    duplicated visual tokens: the full-key scores of the original visual tokens
    equal the visual-only oracle's scores on the visual keys plus those copies."""
    rng = np.random.Generator(np.random.PCG64(31))
    hq, hkv, d = 4, 2, 16
    N, S = [9, 5], [2, 1]
    so, yo = (np.concatenate([[0], np.cumsum(x)]).astype(np.int32) for x in (N, S))
    to = np.array([0, 1, 2], np.int32)
    q = rng.standard_normal((2, hq, d)).astype(np.float32)
    k = rng.standard_normal((int(so[-1]), hkv, d)).astype(np.float32)
    # system keys: request 0 copies its tokens 3 and 4, request 1 its token 2;
    # text keys: each request copies one of its tokens
    k_sys = np.stack([k[so[0] + 3], k[so[0] + 4], k[so[1] + 2]]).astype(np.float32)
    k_txt = np.stack([k[so[0] + 7], k[so[1] + 1]]).astype(np.float32)
    s = oracle.score_full(q, k, k_sys, k_txt, so, to, yo, hq, hkv, d, "f32", lib=lib)
    ext0 = np.concatenate([k[so[0]:so[1]], k_sys[:2], k_txt[:1]])
    ext1 = np.concatenate([k[so[1]:so[2]], k_sys[2:], k_txt[1:]])
    eo = np.array([0, len(ext0), len(ext0) + len(ext1)], np.int32)
    ref = oracle.score(q, np.concatenate([ext0, ext1]), eo, to, hq, hkv, d, "f32", lib=lib)
    np.testing.assert_allclose(s[so[0]:so[1]], ref[eo[0]:eo[0] + N[0]], rtol=2e-7)
    np.testing.assert_allclose(s[so[1]:so[2]], ref[eo[1]:eo[1] + N[1]], rtol=2e-7)
    assert s[so[0]:so[1]].sum() < 1.0 and s[so[1]:so[2]].sum() < 1.0


# ---------------------------------------------------------------------------
# prefill splice (system rows, kept visual rows, text rows; original positions)
# ---------------------------------------------------------------------------

def pin_splice_worked_example(lib):
    """Two requests worked by hand. Request 0: 2 system rows, visual tokens 0..2
    of which 0 and 2 are kept, 1 text row: rows s0 s1 v0 v2 t0 at positions
    0 1 2 4 5 (the pruned token 1 leaves a gap). Request 1: 1 system row, visual
    tokens 3..4 of which 4 (local 1) is kept, 2 text rows: s2 v4 t1 t2 at 0 2 3 4."""
    sys_rows = np.array([[10], [11], [12]], np.uint8)
    vis_rows = np.array([[20], [21], [22], [23], [24]], np.uint8)
    txt_rows = np.array([[30], [31], [32]], np.uint8)
    out, off, pos = oracle.splice([0, 2, 3], [0, 3, 5], [0, 2, 3], [0, 2, 4], [0, 1, 3], sys_rows, vis_rows, txt_rows,
                                  lib=lib)
    assert out.ravel().tolist() == [10, 11, 20, 22, 30, 12, 24, 31, 32]
    assert off.tolist() == [0, 5, 9]
    assert pos.tolist() == [0, 1, 2, 4, 5, 0, 2, 3, 4]


def pin_splice_invariants(lib):
    """Keeping every visual token gives the unpruned sequence with positions
    0..L-1; keeping none gives [system; text] with text at S + N + t; rows are
    byte copies of their sources and positions increase within a request."""
    rng = np.random.Generator(np.random.PCG64(23))
    S, N, T = [3, 0, 5], [7, 4, 0], [2, 6, 1]
    so, vo, to = (np.concatenate([[0], np.cumsum(x)]).astype(np.int32) for x in (S, N, T))
    sys_rows = rng.integers(0, 256, size=(so[-1], 40), dtype=np.uint8)
    vis_rows = rng.integers(0, 256, size=(vo[-1], 40), dtype=np.uint8)
    txt_rows = rng.integers(0, 256, size=(to[-1], 40), dtype=np.uint8)
    out, off, pos = oracle.splice(so, vo, vo, np.arange(vo[-1], dtype=np.int32), to, sys_rows, vis_rows, txt_rows, lib=lib)
    for b in range(3):
        seq = np.concatenate([sys_rows[so[b]:so[b + 1]], vis_rows[vo[b]:vo[b + 1]], txt_rows[to[b]:to[b + 1]]])
        np.testing.assert_array_equal(out[off[b]:off[b + 1]], seq)
        assert pos[off[b]:off[b + 1]].tolist() == list(range(S[b] + N[b] + T[b]))
    out, off, pos = oracle.splice(so, vo, np.zeros(4, np.int32), np.zeros(0, np.int32), to, sys_rows, vis_rows,
                                  txt_rows, lib=lib)
    for b in range(3):
        assert pos[off[b]:off[b + 1]].tolist() == list(range(S[b])) + [S[b] + N[b] + t for t in range(T[b])]
    keep = [np.sort(rng.choice(n, size=n // 2, replace=False)) for n in N]
    ko = np.concatenate([[0], np.cumsum([len(k) for k in keep])]).astype(np.int32)
    ki = np.concatenate([vo[b] + keep[b] for b in range(3)]).astype(np.int32)
    out, off, pos = oracle.splice(so, vo, ko, ki, to, sys_rows, vis_rows, txt_rows, lib=lib)
    for b in range(3):
        p = pos[off[b]:off[b + 1]]
        assert np.all(np.diff(p) > 0)
        np.testing.assert_array_equal(out[off[b] + S[b]:off[b] + S[b] + len(keep[b])], vis_rows[vo[b] + keep[b]])
        assert p[S[b]:S[b] + len(keep[b])].tolist() == [S[b] + j for j in keep[b]]


# ---------------------------------------------------------------------------
# patch-selection gating
# ---------------------------------------------------------------------------

def pin_views_worked_example(lib):
    """Hand-worked gating of three requests over four views (w_lex 2, w_logit 1,
    threshold 0.5, min_views 1; tokens per view 512, 512, 256, 128):
      request 0: s = [2.2, -1, 3, 0.5]  -> views 0, 2 (0.5 is not above 0.5)   768 tokens
      request 1: s = [-5, -2, -3, -2]   -> none pass; the best is -2 at views 1
                                           and 3, the lower index wins: view 1   512 tokens
      request 2: s = [NaN, 0, -1, -7]   -> none pass; NaN ranks lowest: view 1  512 tokens"""
    lex = np.array([[1, 0, 0, 1], [0, 0, 0, 0], [0, 0, 0, 0]], np.float32)
    lg = np.array([[0.2, -1, 3, -1.5], [-5, -2, -3, -2], [np.nan, 0, -1, -7]], np.float32)
    mask, vo, sv, so = oracle.select_views(lex, lg, [512, 512, 256, 128], 2.0, 1.0, 0.5, 1, lib=lib)
    assert mask.tolist() == [[1, 0, 1, 0], [0, 1, 0, 0], [0, 1, 0, 0]], mask
    assert vo.tolist() == [0, 2, 3, 4] and sv.tolist() == [0, 2, 1, 1]
    assert so.tolist() == [0, 768, 1280, 1792]
    # min_views 0: an empty selection is allowed
    mask0, vo0, sv0, so0 = oracle.select_views(lex, lg, [512, 512, 256, 128], 2.0, 1.0, 0.5, 0, lib=lib)
    assert mask0.tolist() == [[1, 0, 1, 0], [0, 0, 0, 0], [0, 0, 0, 0]] and so0.tolist() == [0, 768, 768, 768]


def pin_views_properties(lib):
    """On random inputs: a threshold below every score keeps every view and
    N_b = sum of tokens_per_view; one above every score keeps none (min_views
    0) or exactly the min_views best (every kept score >= every dropped one);
    raising the threshold never adds a view; offsets are prefix sums."""
    rng = np.random.Generator(np.random.PCG64(37))
    B, V = 50, 6
    lex = (rng.random((B, V)) < 0.3).astype(np.float32)
    lg = rng.standard_normal((B, V)).astype(np.float32) * 2
    tpv = np.array([256, 512, 256, 576, 256, 128], np.int32)
    m, vo, sv, so = oracle.select_views(lex, lg, tpv, 1.5, 0.7, -1e30, 0, lib=lib)
    assert m.all() and np.array_equal(np.diff(so), np.full(B, tpv.sum())) and np.array_equal(np.diff(vo), np.full(B, V))
    m, vo, sv, so = oracle.select_views(lex, lg, tpv, 1.5, 0.7, 1e30, 0, lib=lib)
    assert not m.any() and so[-1] == 0 and vo[-1] == 0
    for k in (1, 2, 3):
        m, vo, sv, so = oracle.select_views(lex, lg, tpv, 1.5, 0.7, 1e30, k, lib=lib)
        assert np.array_equal(m.sum(axis=1), np.full(B, k))
        s = np.float32(1.5) * lex + np.float32(0.7) * lg
        for b in range(B):
            assert s[b][m[b] == 1].min() >= s[b][m[b] == 0].max()
    prev = None
    for t in (-2.0, -0.5, 0.0, 0.7, 1.5, 3.0):
        m, vo, sv, so = oracle.select_views(lex, lg, tpv, 1.5, 0.7, t, 0, lib=lib)
        if prev is not None:
            assert np.all(m <= prev)
        prev = m
        assert np.array_equal(np.diff(so), (m * tpv[None, :]).sum(axis=1))
        assert np.array_equal(np.diff(vo), m.sum(axis=1))
        assert sv.tolist() == [v for b in range(B) for v in range(V) if m[b, v]]


# ---------------------------------------------------------------------------
# layer-0 projection (RMSNorm -> W -> RoPE)
# ---------------------------------------------------------------------------

def _bf(a):
    return inputs.f32_to_bf16_bits(np.asarray(a, np.float32))


def pin_project_worked_example(lib):
    """Hand-worked rows, H = O = head_dim = 4, eps = 0 unless stated:
      x = [3,4,0,0], W = I, p = 1, base 1e4: rms 2.5 -> [1.2,1.6,0,0]; pairs (0,2),
        (1,3) with theta = 1, 0.01 -> [1.2 cos 1, 1.6 cos .01, 1.2 sin 1, 1.6 sin .01]
      x = [0,0,0,5], p = 2: -> [0, -2 sin .02, 0, 2 cos .02]
      no RoPE, gamma = [2,1,1,1], bias = [1,0,0,0], x = [3,4,0,0]: [3.4, 1.6, 0, 0]
      eps = 3, x = [1,1,1,1], W = I: every output 1/sqrt(1 + 3) = 0.5
      W with one 1 at [0][1], x = [1,3,1,1]: rms sqrt(3) -> y = [sqrt 3, 0, 0, 0]"""
    eye = _bf(np.eye(4))
    one = np.ones(4, np.float32)
    y = oracle.project(_bf([[3, 4, 0, 0], [0, 0, 0, 5]]), one, 0.0, eye, None, 4, [1, 2], 1e4, lib=lib)
    np.testing.assert_allclose(y[0], [1.2 * math.cos(1), 1.6 * math.cos(0.01), 1.2 * math.sin(1),
                                      1.6 * math.sin(0.01)], rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(y[1], [0, -2 * math.sin(0.02), 0, 2 * math.cos(0.02)], rtol=1e-14, atol=1e-15)
    y = oracle.project(_bf([[3, 4, 0, 0]]), [2, 1, 1, 1], 0.0, eye, [1, 0, 0, 0], 0, None, lib=lib)
    np.testing.assert_allclose(y[0], [3.4, 1.6, 0, 0], rtol=1e-14, atol=1e-15)
    y = oracle.project(_bf([[1, 1, 1, 1]]), one, 3.0, eye, None, 0, None, lib=lib)
    np.testing.assert_allclose(y[0], [0.5] * 4, rtol=1e-14)
    w = np.zeros((4, 4), np.float32)
    w[0, 1] = 1.0
    y = oracle.project(_bf([[1, 3, 1, 1]]), one, 0.0, _bf(w), None, 0, None, lib=lib)
    np.testing.assert_allclose(y[0], [math.sqrt(3), 0, 0, 0], rtol=1e-14, atol=1e-15)


def pin_project_properties(lib):
    """Random rows and weights (H 48, two heads of 16): RoPE keeps each head's
    norm, and rotated query . key depends only on the position difference;
    scaling x by a power of two leaves y unchanged (eps 0); doubling gamma
    doubles y; with W = I, gamma 1 and no bias or RoPE every row has mean
    square 1 (a mean over H, not a sum)."""
    rng = np.random.Generator(np.random.PCG64(41))
    H, O, d = 48, 32, 16
    x = _bf(rng.standard_normal((6, H)))
    w = _bf(rng.standard_normal((O, H)) / math.sqrt(H))
    g = rng.uniform(0.5, 1.5, H).astype(np.float32)
    base = oracle.project(x, g, 0.0, w, None, 0, None, lib=lib)
    pos = np.array([0, 3, 17, 100, 2048, 5], np.int32)
    rot = oracle.project(x, g, 0.0, w, None, d, pos, 1e4, lib=lib)
    for h in range(O // d):
        np.testing.assert_allclose(np.linalg.norm(rot[:, h * d:(h + 1) * d], axis=1),
                                   np.linalg.norm(base[:, h * d:(h + 1) * d], axis=1), rtol=1e-12)
    shift = oracle.project(x, g, 0.0, w, None, d, pos + 37, 1e4, lib=lib)
    for i, j in ((0, 1), (2, 5), (3, 4)):
        for h in range(O // d):
            sl = slice(h * d, (h + 1) * d)
            assert abs(rot[i, sl] @ rot[j, sl] - shift[i, sl] @ shift[j, sl]) < 1e-10
    xs = inputs.f32_to_bf16_bits(inputs.bf16_bits_to_f32(x) * 8.0)
    np.testing.assert_allclose(oracle.project(xs, g, 0.0, w, None, 0, None, lib=lib), base, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(oracle.project(x, 2 * g, 0.0, w, None, 0, None, lib=lib), 2 * base, rtol=1e-12,
                               atol=1e-14)
    y = oracle.project(x, np.ones(H, np.float32), 0.0, _bf(np.eye(H)), None, 0, None, lib=lib)
    np.testing.assert_allclose(np.mean(y * y, axis=1), 1.0, rtol=1e-12)


ALL_PINS = [pin_bf16_decode, pin_e4m3_decode, pin_worked_example, pin_uniform_keys, pin_single_query_is_softmax,
            pin_row_and_total_sums, pin_batch_equals_single_requests, pin_permutation_equivariance, pin_gqa_replication, pin_scale_placement,
            pin_e4m3_scores, pin_salient_tokens_rank_first, pin_topk_bruteforce, pin_topk_batch_and_ratio,
            pin_table1_token_counts, pin_compact, pin_splice_worked_example, pin_splice_invariants,
            pin_full_keys_worked_example, pin_full_keys_equal_duplicated_visual_keys, pin_views_worked_example,
            pin_views_properties, pin_project_worked_example, pin_project_properties]
