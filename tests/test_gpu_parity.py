"""Parity of the CUDA path (through the C-ABI) with the CPU oracle.

Bar: scores within a relative tolerance of 2e-3 (bf16) / 3e-2 (e4m3) per
element; top-k indices and gathered rows bit-exact when top-k and the gather
are fed the oracle's scores / indices. Small cases span several 128-token
tiles and ragged tails; the full-size workloads run in the launch
configuration the benchmark times and are checked on sampled requests (and by
invariants on all of them)."""
import math

import numpy as np
import pytest

import oracle
from gpu_util import (RTOL, assert_scores_close, gather_rows, rel_err, sub_offsets, to_device, to_host)
from paper_2506_07416_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sel():
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    from paper_2506_07416_gb300 import select
    return select


def _case(name, hq, hkv, d, dtype, n_vis, n_txt, sigma=None, seed=7):
    return inputs.Workload(name, len(n_vis), list(n_vis), list(n_txt), hq, hkv, d, 256, dtype, keep_ratio=0.3,
                           sigma=(1.0 / math.sqrt(d)) if sigma is None else sigma, seed=seed)


SCORE_CASES = [
    inputs.workload("tiny"),
    _case("mha_ragged_tails", 16, 16, 128, "bf16", [1, 127, 128, 129, 700, 0, 1536], [64, 1, 16, 33, 128, 5, 64]),
    _case("gqa_7to1", 28, 4, 128, "bf16", [1000, 2049], [128, 77]),
    _case("d64", 4, 4, 64, "bf16", [300, 5, 64], [16, 3, 1]),
    _case("e4m3_ragged", 8, 8, 128, "e4m3", [576, 1152, 100], [32, 128, 50]),
    _case("many_tiles_one_request", 2, 1, 128, "bf16", [9000], [40]),
    _case("sharp_logits", 4, 4, 128, "bf16", [513], [17], sigma=3.0),
    _case("heads_overlap", 32, 32, 128, "bf16", [1536, 1000, 129], [64, 40, 7]),
]


def _selector(sel, w, max_batch=None, kernel="auto"):
    return sel.Selector(max_batch or max(1, w.batch), max(1, w.total_vis), max(1, w.total_txt), w.hq, w.hkv,
                        w.head_dim, w.dtype, score_kernel=kernel)


def _gpu_scores(sel, s, w, x, xd):
    out = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"],
                  seq_offsets_h=x["seq_offsets"], text_offsets_h=x["text_offsets"])
    s.check_device()
    return out.cpu().numpy()


@pytest.mark.parametrize("kernel", ["reread", "resident", "resident_1buf", "resident_2buf"])
@pytest.mark.parametrize("w", SCORE_CASES, ids=lambda w: w.name)
def test_scores_match_oracle(sel, w, kernel):
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = _selector(sel, w, kernel=kernel)
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    if kernel == "reread":
        assert plan[0] == 1
    elif kernel == "resident_1buf" and max(w.n_txt) <= 64:
        assert plan[0] == 2, plan  # every case with short text fits the resident kernel
    elif kernel == "resident_2buf":
        assert plan[0] in (1, 3, 6), plan  # the re-read kernel where two buffers cannot fit
        if w.name in ("heads_overlap", "tiny", "d64"):
            assert plan[0] == 3, plan
    elif max(w.n_txt) <= 64:
        assert plan[0] in (2, 3), plan
    g = _gpu_scores(sel, s, w, x, xd)
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype,
                     x["q_scale"], x["k_scale"])
    assert_scores_close(g, o, w.dtype)
    # deterministic: a second call gives the same bits
    g2 = _gpu_scores(sel, s, w, x, xd)
    np.testing.assert_array_equal(g, g2)
    so = x["seq_offsets"]
    for b in range(w.batch):
        if so[b + 1] > so[b]:
            assert abs(float(np.sum(g[so[b]:so[b + 1]], dtype=np.float64)) - 1.0) < 1e-4


def test_empty_and_zero_length_requests(sel):
    w = _case("zeros", 4, 2, 128, "bf16", [0, 0, 3, 0], [1, 4, 2, 0])
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = _selector(sel, w)
    g = _gpu_scores(sel, s, w, x, xd)
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, "bf16")
    assert_scores_close(g, o, "bf16")
    # batch 0 is a no-op
    sel.score(s.handle, 0, xd["q"], xd["text_offsets"], np.zeros(1, np.int32), xd["k"], xd["seq_offsets"],
              np.zeros(1, np.int32), 1.0, 1.0, torch.empty(1, device="cuda"))
    s.check_device()


def test_score_argument_errors(sel):
    w = _case("errs", 4, 4, 128, "bf16", [10, 5], [3, 0])
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = _selector(sel, w)
    with pytest.raises(sel.LitevlmError) as e:  # visual tokens without text
        s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], seq_offsets_h=x["seq_offsets"],
                text_offsets_h=x["text_offsets"])
    assert e.value.name == "INVALID_ARG"
    w2 = _case("long_text", 4, 4, 128, "bf16", [10], [129])
    x2 = inputs.make_numpy(w2)
    xd2 = to_device(x2, w2)
    s2 = _selector(sel, w2)
    with pytest.raises(sel.LitevlmError) as e:
        s2.score(xd2["q"], xd2["text_offsets"], xd2["k"], xd2["seq_offsets"], seq_offsets_h=x2["seq_offsets"],
                 text_offsets_h=x2["text_offsets"])
    assert e.value.name == "UNSUPPORTED"
    with pytest.raises(sel.LitevlmError) as e:  # bf16 takes no scales
        s2.score(xd2["q"], xd2["text_offsets"], xd2["k"], xd2["seq_offsets"], q_scale=2.0,
                 seq_offsets_h=x2["seq_offsets"], text_offsets_h=x2["text_offsets"])


# ----------------------------------------------------------------------------- top-k

def _topk_gpu(sel, s, scores_np, so, keep_k=None, ratio=0.0):
    d = torch.from_numpy(np.ascontiguousarray(scores_np, dtype=np.float32)).cuda()
    so_d = torch.from_numpy(np.ascontiguousarray(so, dtype=np.int32)).cuda()
    kept, off_d, off_h = s.topk(d, so_d, keep_k=keep_k, keep_ratio=ratio, seq_offsets_h=so)
    s.check_device()
    return kept.cpu().numpy(), off_d.cpu().numpy(), off_h


@pytest.mark.parametrize("w", SCORE_CASES[:5], ids=lambda w: w.name)
def test_topk_on_oracle_scores_is_bit_exact(sel, w):
    x = inputs.make_numpy(w)
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype,
                     x["q_scale"], x["k_scale"])
    s = _selector(sel, w)
    so = x["seq_offsets"]
    for ratio in (0.0, 0.1, 0.3, 0.5, 0.9, 1.0):
        kept, off_d, off_h = _topk_gpu(sel, s, o, so, ratio=ratio)
        ok, ooff = oracle.topk(so, o, keep_ratio=ratio)
        np.testing.assert_array_equal(kept, ok)
        np.testing.assert_array_equal(off_d, ooff)
        np.testing.assert_array_equal(off_h, ooff)
    keep = [max(0, n // 3 - 1) for n in np.diff(so)]
    kept, off_d, _ = _topk_gpu(sel, s, o, so, keep_k=keep)
    ok, ooff = oracle.topk(so, o, keep_k=keep)
    np.testing.assert_array_equal(kept, ok)
    np.testing.assert_array_equal(off_d, ooff)


def test_topk_ties_nan_signed_zero(sel):
    rng = np.random.Generator(np.random.PCG64(5))
    n_vis = [1, 2, 37, 0, 128, 129, 1000, 4097]
    so = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int32)
    vals = np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 1.0, 0.5, 0.5, -1e-30, 3.4e38], np.float32)
    scores = rng.choice(vals, size=so[-1]).astype(np.float32)
    w = _case("ties", 1, 1, 128, "bf16", n_vis, [1] * len(n_vis))
    s = _selector(sel, w)
    for trial in range(4):
        keep = [int(rng.integers(0, n + 1)) for n in n_vis]
        kept, off_d, _ = _topk_gpu(sel, s, scores, so, keep_k=keep)
        ok, ooff = oracle.topk(so, scores, keep_k=keep)
        np.testing.assert_array_equal(kept, ok)
        np.testing.assert_array_equal(off_d, ooff)
    # all equal: the first k indices
    flat = np.full(so[-1], 0.25, np.float32)
    kept, _, _ = _topk_gpu(sel, s, flat, so, ratio=0.5)
    ok, _ = oracle.topk(so, flat, keep_ratio=0.5)
    np.testing.assert_array_equal(kept, ok)


def test_topk_request_larger_than_shared_memory_stage(sel):
    rng = np.random.Generator(np.random.PCG64(6))
    n_vis = [50000, 300]
    so = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int32)
    scores = np.round(rng.standard_normal(so[-1]), 2).astype(np.float32)  # many ties
    w = _case("big", 1, 1, 128, "bf16", n_vis, [1, 1])
    s = _selector(sel, w)
    keep = [12345, 150]
    kept, off_d, _ = _topk_gpu(sel, s, scores, so, keep_k=keep)
    ok, ooff = oracle.topk(so, scores, keep_k=keep)
    np.testing.assert_array_equal(kept, ok)
    np.testing.assert_array_equal(off_d, ooff)


@pytest.mark.parametrize("max_n", [1024, 1025, 2048, 2049, 4096, 4097, 8192, 8193])
def test_topk_every_kernel_size_class(sel, max_n):
    """Each request-size class of the top-k kernels (keys per thread 2/4/8/16,
    then the shared-memory kernel) on score shapes seen in practice: softmax-
    like values in a narrow range, coarse values with many ties, and specials."""
    rng = np.random.Generator(np.random.PCG64(max_n))
    n_vis = [max_n, 1, 0, int(rng.integers(1, max_n)), max_n - 1, 3]
    so = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int32)
    tot = int(so[-1])
    w = _case("sizes", 1, 1, 128, "bf16", n_vis, [1] * len(n_vis))
    s = _selector(sel, w)
    narrow = (np.float32(1.0 / max_n) * (1 + np.float32(1e-3) * rng.standard_normal(tot))).astype(np.float32)
    coarse = np.round(rng.standard_normal(tot), 1).astype(np.float32)
    special = rng.choice(np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 2.0, 2.0, 1e-30], np.float32), tot)
    for scores in (narrow, coarse, special):
        for trial in range(2):
            keep = [int(rng.integers(0, n + 1)) for n in n_vis]
            kept, off_d, _ = _topk_gpu(sel, s, scores, so, keep_k=keep)
            ok, ooff = oracle.topk(so, scores, keep_k=keep)
            np.testing.assert_array_equal(kept, ok)
            np.testing.assert_array_equal(off_d, ooff)
        kept, off_d, _ = _topk_gpu(sel, s, scores, so, ratio=0.3)
        ok, ooff = oracle.topk(so, scores, keep_ratio=0.3)
        np.testing.assert_array_equal(kept, ok)
        np.testing.assert_array_equal(off_d, ooff)


def test_topk_argument_errors(sel):
    w = _case("e", 1, 1, 128, "bf16", [10], [1])
    s = _selector(sel, w)
    so = np.array([0, 10], np.int32)
    with pytest.raises(sel.LitevlmError):
        _topk_gpu(sel, s, np.zeros(10, np.float32), so, keep_k=[11])
    with pytest.raises(sel.LitevlmError):
        _topk_gpu(sel, s, np.zeros(10, np.float32), so, ratio=1.5)


# ----------------------------------------------------------------------------- gather

def test_compact_bit_exact(sel):
    rng = np.random.Generator(np.random.PCG64(8))
    rows = 777
    w = _case("g", 1, 1, 128, "bf16", [rows], [1])
    s = _selector(sel, w)
    idx = np.sort(rng.choice(rows, size=311, replace=False)).astype(np.int32)
    tensors = [rng.integers(0, 256, size=(rows, 4096), dtype=np.uint8),   # hidden-sized rows
               rng.integers(0, 256, size=(rows, 2048), dtype=np.uint8),   # K rows
               rng.integers(0, 256, size=(rows, 48), dtype=np.uint8),     # short rows
               rng.integers(0, 256, size=(rows, 7184), dtype=np.uint8),   # a 4 KB piece and a partial one
               rng.integers(0, 256, size=(rows, 6), dtype=np.uint8)]      # unaligned rows (byte path)
    for group in (tensors[:4], tensors[4:]):
        srcs = [torch.from_numpy(t).cuda() for t in group]
        dsts = s.compact(torch.from_numpy(idx).cuda(), len(idx), srcs)
        s.check_device()
        for t, d in zip(group, dsts):
            np.testing.assert_array_equal(d.cpu().numpy(), oracle.compact(idx, t))
    assert s.compact(torch.from_numpy(idx).cuda(), 0, [torch.from_numpy(tensors[0]).cuda()])[0].numel() == 0


def test_compact_out_of_range_index_is_reported(sel):
    w = _case("g", 1, 1, 128, "bf16", [8], [1])
    s = _selector(sel, w)
    src = torch.arange(8 * 16, dtype=torch.uint8, device="cuda").view(8, 16)
    idx = torch.tensor([1, 8, 3], dtype=torch.int32, device="cuda")  # 8 is outside [0, 8)
    dst = s.compact(idx, 3, [src])[0]
    with pytest.raises(sel.LitevlmError) as e:
        s.check_device()
    assert e.value.name == "DEVICE_BOUNDS"
    assert torch.equal(dst[0], src[1]) and torch.equal(dst[2], src[3])
    s.check_device()  # the word was cleared


@pytest.mark.parametrize("row_bytes", [4096, 112, 6])
def test_compact_from_pinned_host_memory_bit_exact(sel, row_bytes):
    """Sources in pinned host memory are read through their device view: the
    gathered rows are the source rows byte for byte, next to a device source
    gathered with the same indices."""
    w = _case("g", 1, 1, 128, "bf16", [8], [1])
    s = _selector(sel, w)
    rng = np.random.default_rng(5)
    rows = 3000
    src_np = rng.integers(0, 256, size=(rows, row_bytes), dtype=np.uint8)
    host = torch.from_numpy(src_np).pin_memory()
    dev_src = host.cuda()
    idx_np = np.sort(rng.choice(rows, 907, replace=False)).astype(np.int32)
    idx = torch.from_numpy(idx_np).cuda()
    from_host, from_dev = s.compact(idx, len(idx_np), [host, dev_src])
    s.check_device()
    np.testing.assert_array_equal(from_host.cpu().numpy(), src_np[idx_np])
    np.testing.assert_array_equal(from_dev.cpu().numpy(), src_np[idx_np])


def test_host_view_argument_errors(sel):
    w = _case("g", 1, 1, 128, "bf16", [8], [1])
    s = _selector(sel, w)
    with pytest.raises(sel.LitevlmError) as e:
        s.host_view(0)
    assert e.value.name == "INVALID_ARG"
    host = torch.zeros(64, dtype=torch.uint8).pin_memory()
    assert s.host_view(host) != 0


# ----------------------------------------------------------------------------- whole path

def test_tiny_whole_path(sel):
    w = inputs.workload("tiny")
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = _selector(sel, w)
    g = _gpu_scores(sel, s, w, x, xd)
    o, okept, ooff, orows = oracle.select(x, w.hq, w.hkv, w.head_dim, "bf16", keep_k=w.keep_k)
    assert_scores_close(g, o, "bf16")
    kept, off_d, off_h = s.topk(torch.from_numpy(g).cuda(), xd["seq_offsets"], keep_k=w.keep_k,
                                seq_offsets_h=x["seq_offsets"])
    # the GPU's selection is the exact top-k of the GPU's scores
    gk, _ = oracle.topk(x["seq_offsets"], g, keep_k=w.keep_k)
    np.testing.assert_array_equal(kept.cpu().numpy(), gk)
    # with the oracle's scores it is the oracle's selection
    k2, _, _ = s.topk(torch.from_numpy(o).cuda(), xd["seq_offsets"], keep_k=w.keep_k, seq_offsets_h=x["seq_offsets"])
    np.testing.assert_array_equal(k2.cpu().numpy(), okept)
    rows = s.compact(k2, int(off_h[-1]), [xd["hidden"]])[0]
    s.check_device()
    np.testing.assert_array_equal(rows.view(torch.int16).cpu().numpy().view(np.uint16), orows["hidden"])
    # the 8 salient tokens are among the kept ones
    assert set((x["salient"][0]).tolist()) <= set(gk.tolist())


# ----------------------------------------------------------------------------- full size

def _rows_u8(t):
    """Rows of a device tensor as host bytes, [rows, row_bytes] uint8."""
    t = t.contiguous()
    u = t if t.dtype == torch.uint8 else t.view(torch.uint8)
    return u.reshape(t.shape[0], -1).cpu().numpy()


FULL = [("single", [0]), ("highres", [0]), ("fp8_ragged", None), ("sweep", [0, 77, 127])]


@pytest.mark.parametrize("name,sample", FULL, ids=[f[0] for f in FULL])
def test_full_size_workload(sel, name, sample):
    """Full size, in the launch configuration bench.py times (automatic kernel choice)."""
    w = inputs.workload(name)
    xd = inputs.make_torch(w, "cuda")
    so, to = w.seq_offsets(), w.text_offsets()
    s = _selector(sel, w)
    print(f"{name}: score plan {s.score_plan(to, so)}")
    g_t = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"],
                  seq_offsets_h=so, text_offsets_h=to)
    s.check_device()
    g = g_t.cpu().numpy()
    # invariant on every request: the scores of a request sum to 1
    sums = np.add.reduceat(g.astype(np.float64), so[:-1]) if w.batch > 1 else np.array([g.sum(dtype=np.float64)])
    assert np.max(np.abs(sums - 1.0)) < 1e-4
    if sample is None:  # smallest, largest and a middle request
        order = np.argsort(np.diff(so), kind="stable")
        sample = sorted({int(order[0]), int(order[-1]), int(order[len(order) // 2])})
    # sampled requests against the oracle
    qh = to_host({"q": xd["q"], "k": xd["k"]})
    sq = gather_rows(qh["q"], to, sample)
    sk = gather_rows(qh["k"], so, sample)
    sso, sto = sub_offsets(so, sample), sub_offsets(to, sample)
    o = oracle.score(sq, sk, sso, sto, w.hq, w.hkv, w.head_dim, w.dtype, xd["q_scale"], xd["k_scale"])
    gs = np.concatenate([g[so[b]:so[b + 1]] for b in sample])
    err = assert_scores_close(gs, o, w.dtype)
    print(f"{name}: max rel err {err:.2e} on requests {sample}")
    # top-k fed the oracle's scores: bit-exact on the sampled requests
    ss = _selector(sel, inputs.sub_batch(w, sample))
    ratios = [0.1, 0.2, 0.3, 0.5] if name == "sweep" else [None]
    for r in ratios:
        kk = None if w.keep_k is None else [w.keep_k[b] for b in sample]
        rr = w.keep_ratio if r is None else r
        kept, off_d, _ = _topk_gpu(sel, ss, o, sso, keep_k=kk, ratio=rr or 0.0)
        ok, ooff = oracle.topk(sso, o, keep_k=kk, keep_ratio=rr or 0.0)
        np.testing.assert_array_equal(kept, ok)
        np.testing.assert_array_equal(off_d, ooff)
    # top-k on the GPU scores of every request is the exact top-k of those scores,
    # and the gather moves exactly those rows
    for r in ratios:
        rr = w.keep_ratio if r is None else r
        kept_t, off_d, off_h = s.topk(g_t, xd["seq_offsets"], keep_k=w.keep_k if r is None else None,
                                      keep_ratio=rr or 0.0, seq_offsets_h=so)
        ok, ooff = oracle.topk(so, g, keep_k=w.keep_k if r is None else None, keep_ratio=rr or 0.0)
        np.testing.assert_array_equal(kept_t.cpu().numpy(), ok)
        np.testing.assert_array_equal(off_h, ooff)
        srcs = [xd[n] for n in w.gather]
        outs = s.compact(kept_t, int(off_h[-1]), srcs)
        s.check_device()
        idx = kept_t.long()
        for src, dst in zip(srcs, outs):
            assert torch.equal(dst.view(torch.uint8) if dst.dtype != torch.uint8 else dst,
                               src.index_select(0, idx).view(torch.uint8) if src.dtype != torch.uint8
                               else src.index_select(0, idx))
        # and on the sampled requests, byte for byte against the oracle's gather
        for b in sample:
            kb = ok[ooff[b]:ooff[b + 1]] - so[b]
            for src, dst in zip(srcs, outs):
                want = oracle.compact(kb, _rows_u8(src[so[b]:so[b + 1]]))
                np.testing.assert_array_equal(_rows_u8(dst[off_h[b]:off_h[b + 1]]), want)
    del xd
    torch.cuda.empty_cache()


# ----------------------------------------------------------------------------- prefill splice

def _splice_case(rng, S, N, T, row_bytes, keep_frac=None):
    so, vo, to = (np.concatenate([[0], np.cumsum(x)]).astype(np.int32) for x in (S, N, T))
    keep = []
    for b, n in enumerate(N):
        k = int(rng.integers(0, n + 1)) if keep_frac is None else int(n * keep_frac)
        keep.append(np.sort(rng.choice(n, size=k, replace=False)).astype(np.int32))
    ko = np.concatenate([[0], np.cumsum([len(k) for k in keep])]).astype(np.int32)
    ki = np.concatenate([vo[b] + keep[b] for b in range(len(N))] + [np.zeros(0, np.int32)]).astype(np.int32)
    rows = [rng.integers(0, 256, size=(max(int(o[-1]), 1), row_bytes), dtype=np.uint8) for o in (so, vo, to)]
    return so, vo, ko, ki, to, rows


def _splice_gpu(s, so, vo, ko, ki, to, rows):
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    out, off_d, off_h, pos = s.splice(d(rows[0]), d(so), d(rows[1]), d(vo), d(ki if ki.size else np.zeros(1, np.int32)),
                                      d(ko), d(rows[2]), d(to))
    s.check_device()
    return out.cpu().numpy(), off_d.cpu().numpy(), off_h, pos.cpu().numpy()


@pytest.mark.parametrize("row_bytes", [4096, 112, 6])
def test_splice_bit_exact(sel, row_bytes):
    rng = np.random.Generator(np.random.PCG64(31 + row_bytes))
    S, N, T = [0, 5, 32, 1, 0], [7, 0, 300, 129, 0], [3, 4, 0, 64, 0]
    so, vo, ko, ki, to, rows = _splice_case(rng, S, N, T, row_bytes)
    w = _case("splice", 1, 1, 128, "bf16", N, [1] * len(N))
    s = _selector(sel, w)
    out, off_d, off_h, pos = _splice_gpu(s, so, vo, ko, ki, to, rows)
    o_out, o_off, o_pos = oracle.splice(so, vo, ko, ki, to, rows[0][:so[-1]], rows[1][:vo[-1]], rows[2][:to[-1]])
    np.testing.assert_array_equal(out, o_out)
    np.testing.assert_array_equal(off_d, o_off)
    np.testing.assert_array_equal(off_h, o_off)
    np.testing.assert_array_equal(pos, o_pos)


def test_splice_out_of_range_kept_index_is_reported(sel):
    rng = np.random.Generator(np.random.PCG64(37))
    so, vo, ko, ki, to, rows = _splice_case(rng, [2, 2], [10, 10], [3, 3], 64, keep_frac=0.5)
    ki = ki.copy()
    ki[0] = 15  # a row of the second request listed under the first
    w = _case("splice_bad", 1, 1, 128, "bf16", [10, 10], [1, 1])
    s = _selector(sel, w)
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    s.splice(d(rows[0]), d(so), d(rows[1]), d(vo), d(ki), d(ko), d(rows[2]), d(to))
    with pytest.raises(sel.LitevlmError) as ei:
        s.check_device()
    assert ei.value.name == "DEVICE_BOUNDS"


def test_splice_after_selection_on_the_single_workload(sel):
    """score -> top-k -> splice on the 1536-token request with 32 system and the
    request's 64 text rows (hidden size rows), checked against the oracle's
    splice of the same kept indices."""
    w = inputs.workload("single")
    xd = inputs.make_torch(w, "cuda")
    s = _selector(sel, w)
    so_v, to_t = w.seq_offsets(), w.text_offsets()
    sc = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], seq_offsets_h=so_v, text_offsets_h=to_t)
    kept, ko_d, ko_h = s.topk(sc, xd["seq_offsets"], keep_ratio=w.keep_ratio, seq_offsets_h=so_v)
    g = torch.Generator(device="cuda").manual_seed(41)
    sys_rows = torch.randn((32, w.hidden), generator=g, device="cuda").to(torch.bfloat16)
    txt_rows = torch.randn((int(to_t[-1]), w.hidden), generator=g, device="cuda").to(torch.bfloat16)
    sys_off = torch.tensor([0, 32], dtype=torch.int32, device="cuda")
    out, off_d, off_h, pos = s.splice(sys_rows, sys_off, xd["hidden"], xd["seq_offsets"], kept, ko_d, txt_rows,
                                      xd["text_offsets"])
    s.check_device()
    as_bytes = lambda t: t.contiguous().view(torch.uint8).cpu().numpy().reshape(t.shape[0], -1)
    o_out, o_off, o_pos = oracle.splice([0, 32], so_v, ko_h, kept.cpu().numpy(), to_t, as_bytes(sys_rows),
                                        as_bytes(xd["hidden"]), as_bytes(txt_rows))
    np.testing.assert_array_equal(as_bytes(out), o_out)
    np.testing.assert_array_equal(off_h, o_off)
    np.testing.assert_array_equal(pos.cpu().numpy(), o_pos)
    assert int(off_h[-1]) == 32 + int(ko_h[-1]) + 64


# ----------------------------------------------------------------------------- last-token queries

LAST_TOKEN_CASES = SCORE_CASES[:5] + [_case("long_text_last", 8, 8, 128, "bf16", [700, 129], [200, 3])]


@pytest.mark.parametrize("kernel", ["reread", "resident"])
@pytest.mark.parametrize("w", LAST_TOKEN_CASES, ids=lambda w: w.name)
def test_last_token_queries_match_oracle(sel, w, kernel):
    """Only the last text token of each request is a query: the same score as
    the oracle's on each request's last text row alone."""
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = sel.Selector(max(1, w.batch), max(1, w.total_vis), max(1, w.total_txt), w.hq, w.hkv, w.head_dim, w.dtype,
                     score_kernel=kernel, query="last")
    g = _gpu_scores(sel, s, w, x, xd)
    to = np.asarray(x["text_offsets"])
    last = np.array([to[b + 1] - 1 for b in range(w.batch) if to[b + 1] > to[b]], np.int64)
    lens = [1 if to[b + 1] > to[b] else 0 for b in range(w.batch)]
    to_last = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    o = oracle.score(x["q"][last], x["k"], x["seq_offsets"], to_last, w.hq, w.hkv, w.head_dim, w.dtype,
                     x["q_scale"], x["k_scale"])
    assert_scores_close(g, o, w.dtype)
