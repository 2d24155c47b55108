"""Parity of litevlm_select_score_full_keys (softmax over the system, visual and
causal text keys) with the oracle's score_full, through the C-ABI.

Same bar as the visual-key scores: relative error per element within 2e-3
(bf16) / 3e-2 (e4m3). The cases cover several 128-token tiles with ragged
tails, requests without system keys or without visual tokens, more than 256
context keys (the statistics kernel's key-tile loop), GQA, d = 64, e4m3 with
the visual keys' scale, an attention-sink system key, and both score kernels."""
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


def _case(name, hq, hkv, d, dtype, n_vis, n_txt, sigma=None, seed=7):
    return inputs.Workload(name, len(n_vis), list(n_vis), list(n_txt), hq, hkv, d, 256, dtype, keep_ratio=0.3,
                           sigma=(1.0 / math.sqrt(d)) if sigma is None else sigma, seed=seed)


# (workload, system-prompt lengths, sink gain)
CASES = [
    (inputs.workload("tiny"), [5], 0.0),
    (_case("mha_ragged_tails", 16, 16, 128, "bf16", [1, 127, 128, 129, 700, 0, 1536], [64, 1, 16, 33, 128, 5, 64]),
     [32, 0, 7, 32, 300, 3, 32], 0.0),
    (_case("gqa_7to1", 28, 4, 128, "bf16", [1000, 2049], [128, 77]), [20, 64], 0.0),
    (_case("d64", 4, 4, 64, "bf16", [300, 5, 64], [16, 3, 1]), [1, 2, 0], 0.0),
    (_case("e4m3_ragged", 8, 8, 128, "e4m3", [576, 1152, 100], [32, 128, 50]), [32, 32, 32], 0.0),
    (_case("heads_overlap", 32, 32, 128, "bf16", [1536, 1000, 129], [64, 40, 7]), [32, 16, 0], 0.0),
    (_case("attention_sink", 8, 8, 128, "bf16", [1536, 576], [64, 20]), [32, 8], 6.0),
]


def _inputs(w, sys_lens, sink):
    x = inputs.make_numpy(w, fp32=True)
    c = inputs.context_keys_numpy(w, sys_lens, k_scale=x["k_scale"], sink_gain=sink, q_f32=x["q_f32"])
    xd = to_device(x, w)
    cd = {}
    for name in ("k_sys", "k_txt"):
        a = c[name]
        if a.shape[0] == 0:
            a = np.zeros((1,) + a.shape[1:], a.dtype)  # a valid, aligned pointer for an empty tensor
        cd[name] = (torch.from_numpy(a.view(np.int16).copy()).view(torch.bfloat16) if a.dtype == np.uint16
                    else torch.from_numpy(a.copy())).cuda()
    cd["sys_offsets"] = torch.from_numpy(c["sys_offsets"]).cuda()
    return x, xd, c, cd


def _gpu(s, x, xd, c, cd):
    out = s.score_full_keys(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], cd["k_sys"], cd["sys_offsets"],
                            cd["k_txt"], xd["q_scale"], xd["k_scale"], seq_offsets_h=x["seq_offsets"],
                            text_offsets_h=x["text_offsets"], sys_offsets_h=c["sys_offsets"])
    s.check_device()
    return out.cpu().numpy()


@pytest.mark.parametrize("kernel", ["reread", "resident", "resident_2buf"])
@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0].name)
def test_full_key_scores_match_oracle(sel, case, kernel):
    w, sys_lens, sink = case
    x, xd, c, cd = _inputs(w, sys_lens, sink)
    s = sel.Selector(max(1, w.batch), max(1, w.total_vis), max(1, w.total_txt), w.hq, w.hkv, w.head_dim, w.dtype,
                     score_kernel=kernel)
    g = _gpu(s, x, xd, c, cd)
    o, _, share = oracle.score_full(x["q"], x["k"], c["k_sys"], c["k_txt"], x["seq_offsets"], x["text_offsets"],
                                    c["sys_offsets"], w.hq, w.hkv, w.head_dim, w.dtype, x["q_scale"], x["k_scale"],
                                    details=True)
    assert_scores_close(g, o, w.dtype)
    np.testing.assert_array_equal(g, _gpu(s, x, xd, c, cd))  # deterministic
    # a request's scores add up to its mean visual attention share (< 1)
    so, to = x["seq_offsets"], x["text_offsets"]
    r0 = 0
    for b in range(w.batch):
        rows = w.hq * int(to[b + 1] - to[b])
        if so[b + 1] > so[b]:
            want = float(np.mean(share[r0:r0 + rows]))
            got = float(np.sum(g[so[b]:so[b + 1]], dtype=np.float64))
            assert abs(got - want) <= 2e-3 * want, (b, got, want)
            assert want < 1.0
        r0 += rows
    if sink > 0:
        assert float(np.sum(g[so[0]:so[1]], dtype=np.float64)) < 0.9  # the sink takes a visible share


def test_full_keys_with_no_context_keys_equals_visual_only(sel):
    """S_b = 0 and T_b = 1: the one query sees the visual keys and itself; with
    its own key pushed far away (logit -> -inf) the scores reduce to the
    visual-key scores of litevlm_select_score."""
    w = _case("self_key_far", 8, 8, 128, "bf16", [700, 129], [1, 1])
    x, xd, c, cd = _inputs(w, [0, 0], 0.0)
    q = x["q"]
    qf = inputs.bf16_bits_to_f32(q).reshape(w.total_txt, w.hq, w.head_dim)
    # text key = -4000 * the unit query direction (G = 1): its logit is about -350, exp() = 0 in fp32
    kt = np.zeros((w.total_txt, w.hkv, w.head_dim), np.float32)
    for t in range(w.total_txt):
        for g in range(w.hkv):
            kt[t, g] = -4000.0 * qf[t, g] / max(np.linalg.norm(qf[t, g]), 1e-6)
    # every head of a group must see the key as far: only true for G = 1
    assert w.hq == w.hkv
    c["k_txt"] = inputs.f32_to_bf16_bits(kt)
    cd["k_txt"] = torch.from_numpy(c["k_txt"].view(np.int16).copy()).view(torch.bfloat16).cuda()
    s = sel.Selector(2, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype)
    g_full = _gpu(s, x, xd, c, cd)
    g_vis = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], seq_offsets_h=x["seq_offsets"],
                    text_offsets_h=x["text_offsets"]).cpu().numpy()
    o = oracle.score_full(x["q"], x["k"], c["k_sys"], c["k_txt"], x["seq_offsets"], x["text_offsets"],
                          c["sys_offsets"], w.hq, w.hkv, w.head_dim, "bf16")
    assert_scores_close(g_full, o, "bf16")
    assert_scores_close(g_full, g_vis, "bf16")


LAST_CASES = [
    (_case("long_text_last", 8, 8, 128, "bf16", [700, 129], [200, 3]), [100, 0]),
    (_case("e4m3_last", 8, 2, 128, "e4m3", [576, 1152], [128, 40]), [32, 300]),
]


@pytest.mark.parametrize("kernel", ["reread", "resident"])
@pytest.mark.parametrize("case", LAST_CASES, ids=lambda c: c[0].name)
def test_full_keys_last_token_query(sel, case, kernel):
    """Last-token queries: the one query sees every system and text key. The
    oracle's equivalent: that row as the only text token, with the request's
    other text keys appended to its system keys (the normaliser is a sum, so
    the order of the keys does not matter)."""
    w, sys_lens = case
    x, xd, c, cd = _inputs(w, sys_lens, 0.0)
    s = sel.Selector(max(1, w.batch), max(1, w.total_vis), max(1, w.total_txt), w.hq, w.hkv, w.head_dim, w.dtype,
                     score_kernel=kernel, query="last")
    g = _gpu(s, x, xd, c, cd)
    to, yo = x["text_offsets"], c["sys_offsets"]
    last = [int(to[b + 1]) - 1 for b in range(w.batch)]
    ks, lens = [], []
    for b in range(w.batch):
        part = np.concatenate([c["k_sys"][yo[b]:yo[b + 1]], c["k_txt"][to[b]:to[b + 1] - 1]])
        ks.append(part)
        lens.append(part.shape[0])
    k_sys2 = np.concatenate(ks)
    yo2 = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    to1 = np.arange(w.batch + 1, dtype=np.int32)
    o = oracle.score_full(x["q"][last], x["k"], k_sys2, c["k_txt"][last], x["seq_offsets"], to1, yo2, w.hq, w.hkv,
                          w.head_dim, w.dtype, x["q_scale"], x["k_scale"])
    assert_scores_close(g, o, w.dtype)


def test_full_keys_argument_errors(sel):
    w = _case("errs", 4, 4, 128, "bf16", [10, 5], [3, 2])
    x, xd, c, cd = _inputs(w, [2, 2], 0.0)
    s = sel.Selector(2, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype)
    with pytest.raises(sel.LitevlmError) as e:
        s.score_full_keys(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], cd["k_sys"], cd["sys_offsets"],
                          0, seq_offsets_h=x["seq_offsets"], text_offsets_h=x["text_offsets"],
                          sys_offsets_h=c["sys_offsets"])
    assert e.value.name == "INVALID_ARG"
    with pytest.raises(sel.LitevlmError) as e:
        s.score_full_keys(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], cd["k_sys"], cd["sys_offsets"],
                          cd["k_txt"], seq_offsets_h=x["seq_offsets"], text_offsets_h=x["text_offsets"],
                          sys_offsets_h=np.array([0, 3, 2], np.int32))
    assert e.value.name == "INVALID_ARG"
    s.check_device()
