"""The TMEM-resident score kernel's flattened schedule (plan[0] = 4): for
batches whose requests all have the same visual and text token counts, the
batch's (request, head) pairs are split evenly over the clusters that fit on
the GPU at once; a cluster runs its share back to back across request
boundaries, and a request whose heads span two clusters is folded from their
partial rows. Checked against the oracle on uniform batches of several shapes
(bf16 and e4m3, GQA, d = 64, last-token queries, the full causal key set), for
bit-reproducibility, and against the one-call score + top-k."""
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


def _uniform(name, batch, n, t, hq, hkv, d, dtype, seed=21):
    return inputs.Workload(name, batch, [n] * batch, [t] * batch, hq, hkv, d, 256, dtype, keep_ratio=0.3,
                           sigma=1.0 / math.sqrt(d), seed=seed)


CASES = [
    _uniform("many_small", 40, 640, 24, 8, 8, 128, "bf16"),
    _uniform("gqa", 24, 300, 40, 28, 4, 128, "bf16"),
    _uniform("e4m3", 20, 576, 50, 16, 16, 128, "e4m3"),
    _uniform("d64", 30, 200, 8, 4, 4, 64, "bf16"),
    _uniform("ragged_tail_tile", 36, 1000, 64, 16, 16, 128, "bf16"),
]


def _score(s, x, xd):
    out = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"],
                  seq_offsets_h=x["seq_offsets"], text_offsets_h=x["text_offsets"])
    s.check_device()
    return out.cpu().numpy()


@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_flat_schedule_matches_oracle(sel, w):
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="resident_flat")
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] == 4, plan
    assert 1 <= plan[3] <= w.batch * w.hq
    g = _score(s, x, xd)
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype,
                     x["q_scale"], x["k_scale"])
    assert_scores_close(g, o, w.dtype)
    # every request's scores sum to 1
    sums = np.add.reduceat(g.astype(np.float64), x["seq_offsets"][:-1])
    assert np.max(np.abs(sums - 1.0)) < 1e-4
    # deterministic, and the one-call score + top-k gives the same bits
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


def test_flat_schedule_last_token_queries(sel):
    w = _uniform("last_token", 30, 500, 20, 8, 8, 128, "bf16", seed=22)
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="resident_flat",
                     query="last")
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] == 4, plan
    g = _score(s, x, xd)
    to = x["text_offsets"]
    last_rows = np.concatenate([np.arange(to[b + 1] - 1, to[b + 1]) for b in range(w.batch)])
    o = oracle.score(x["q"][last_rows], x["k"], x["seq_offsets"], np.arange(w.batch + 1, dtype=np.int32), w.hq,
                     w.hkv, w.head_dim, w.dtype)
    assert_scores_close(g, o, w.dtype)
    s.close()


def test_flat_schedule_full_key_set(sel):
    w = _uniform("full_keys", 26, 384, 12, 8, 4, 128, "bf16", seed=23)
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    n_sys = [5] * w.batch
    c = inputs.context_keys_numpy(w, n_sys, seed=24)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="resident_flat")
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] == 4, plan
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


def test_flat_flag_falls_back_on_ragged_batches(sel):
    w = inputs.Workload("ragged", 3, [300, 129, 640], [16, 16, 16], 8, 8, 128, 256, "bf16", keep_ratio=0.3,
                        sigma=1.0 / math.sqrt(128), seed=25)
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="resident_flat")
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] == 2, plan  # one buffer, per-request clusters
    g = _score(s, x, xd)
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype)
    assert_scores_close(g, o, w.dtype)
    s.close()


def test_sweep_takes_the_flat_schedule(sel):
    w = inputs.workload("sweep")
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype)
    plan = s.score_plan(w.text_offsets(), w.seq_offsets())
    assert plan[0] == 4 and plan[1] * plan[2] >= 27, plan
    s.close()
