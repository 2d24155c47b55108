"""The query split of the TMEM-resident score kernel (plan[0] = 5, 6, 7):
requests with more than 64 text tokens run each query head's text rows as two
pseudo-heads, the first ceil(T/2) rows and the rest, on the 64-row kernel. The
score is a sum over heads and text rows of per-row softmax values, so the split
changes no term, only where it is computed; the denominators stay Hq * T.
Checked against the oracle on ragged and uniform batches (bf16 and e4m3, GQA,
d = 64, odd T, requests of 64 tokens or fewer next to longer ones, the full key
set), for bit-reproducibility and against the one-call score + top-k. The
split is opt-in (LITEVLM_FLAG_SCORE_SPLIT_QUERIES); with last-token queries
there is nothing to split."""
import math

import numpy as np
import pytest

import oracle
from gpu_util import assert_scores_close, to_device
from paper_2506_07416_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sel():
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    from paper_2506_07416_gb300 import select
    return select


def _wl(name, n, t, hq=16, hkv=16, d=128, dtype="bf16", seed=41):
    return inputs.Workload(name, len(n), list(n), list(t), hq, hkv, d, 256, dtype, keep_ratio=0.3,
                           sigma=1.0 / math.sqrt(d), seed=seed)


CASES = [
    # (workload, score kernel option)
    (_wl("ragged_mixed_t", [700, 129, 1536, 300, 1], [128, 65, 100, 64, 77]), "resident"),
    (_wl("ragged_1buf", [1000, 513, 256], [127, 66, 128], seed=42), "resident_1buf"),
    (_wl("ragged_2buf", [384, 256, 500], [128, 90, 71], hq=8, hkv=8, seed=43), "resident_2buf"),
    (_wl("gqa_one_request", [2048], [128], hq=28, hkv=4, seed=44), "resident"),
    (_wl("uniform_flat", [640] * 12, [77] * 12, seed=45), "resident_flat"),
    (_wl("e4m3_ragged", [576, 1152, 100], [32, 128, 71], hq=8, hkv=8, dtype="e4m3", seed=46), "resident"),
    (_wl("e4m3_uniform", [576] * 10, [96] * 10, hq=8, hkv=8, dtype="e4m3", seed=47), "resident_flat"),
    (_wl("d64", [300, 700], [128, 80], hq=4, hkv=4, d=64, seed=48), "resident"),
]


def _score(s, x, xd):
    out = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"],
                  seq_offsets_h=x["seq_offsets"], text_offsets_h=x["text_offsets"])
    s.check_device()
    return out.cpu().numpy()


@pytest.mark.parametrize("w,kern", CASES, ids=lambda c: c.name if hasattr(c, "name") else c)
def test_query_split_matches_oracle(sel, w, kern):
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel=kern,
                     query_split="split")
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] in (5, 6, 7), plan
    if kern == "resident_flat":
        assert plan[0] == 7, plan
    g = _score(s, x, xd)
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype,
                     x["q_scale"], x["k_scale"])
    assert_scores_close(g, o, w.dtype)
    # each request's scores sum to 1 (every text row's softmax does)
    so = x["seq_offsets"]
    for b in range(w.batch):
        if so[b + 1] > so[b]:
            assert abs(float(np.sum(g[so[b]:so[b + 1]], dtype=np.float64)) - 1.0) < 1e-4
    # bit-reproducible, and the one-call score + top-k gives the same bits
    assert np.array_equal(g.view(np.uint32), _score(s, x, xd).view(np.uint32))
    sc, kept, off_d, off_h = s.score_topk(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"],
                                          xd["k_scale"], keep_ratio=0.3, seq_offsets_h=x["seq_offsets"],
                                          text_offsets_h=x["text_offsets"])
    s.check_device()
    assert np.array_equal(g.view(np.uint32), sc.cpu().numpy().view(np.uint32))
    ok, ooff = oracle.topk(x["seq_offsets"], g, keep_ratio=0.3)
    np.testing.assert_array_equal(kept.cpu().numpy(), ok)
    np.testing.assert_array_equal(off_h, ooff)
    s.close()


def test_query_split_with_the_full_key_set(sel):
    w = _wl("full_keys", [900, 400], [128, 70], hq=8, hkv=4, seed=49)
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    n_sys = [7, 3]
    c = inputs.context_keys_numpy(w, n_sys, seed=50)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="resident",
                     query_split="split")
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] in (5, 6, 7), plan
    dev = lambda a: torch.from_numpy(a.view(np.int16).copy()).view(torch.bfloat16).cuda()
    sys_off = np.concatenate([[0], np.cumsum(n_sys)]).astype(np.int32)
    out = s.score_full_keys(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], dev(c["k_sys"]),
                            torch.from_numpy(sys_off).cuda(), dev(c["k_txt"]), seq_offsets_h=x["seq_offsets"],
                            text_offsets_h=x["text_offsets"], sys_offsets_h=sys_off)
    s.check_device()
    o = oracle.score_full(x["q"], x["k"], c["k_sys"], c["k_txt"], x["seq_offsets"], x["text_offsets"], sys_off,
                          w.hq, w.hkv, w.head_dim, w.dtype)
    assert_scores_close(out.cpu().numpy(), o, w.dtype)
    s.close()


def test_no_split_by_default_nor_with_last_token_queries(sel):
    w = _wl("long_text", [1000, 300], [128, 100], seed=51)
    x = inputs.make_numpy(w)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="resident")
    assert s.score_plan(x["text_offsets"], x["seq_offsets"])[0] in (1, 2, 3, 4)
    s.close()
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="resident",
                     query="last", query_split="split")
    assert s.score_plan(x["text_offsets"], x["seq_offsets"])[0] in (1, 2, 3, 4)
    s.close()
