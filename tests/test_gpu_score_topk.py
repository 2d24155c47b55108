"""litevlm_select_score_topk (scores and top-k in one call, the head-group
fold moved into the top-k kernel) against the two separate calls on the same
inputs: scores bit-identical (the partials are added in the same order and
divided once, as the score kernel's own fold does), kept indices and offsets
identical, and the kept set equal to the oracle's top-k of those scores. Cases
with head groups (deferred fold), without (one group), e4m3, last-token
queries, and the fallbacks (more than 256 requests, a request beyond 8192
tokens)."""
import math

import numpy as np
import pytest

import oracle
from gpu_util import to_device
from paper_2506_07416_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sel():
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    from paper_2506_07416_gb300 import select
    return select


def _case(name, hq, hkv, d, dtype, n_vis, n_txt, seed=7):
    return inputs.Workload(name, len(n_vis), list(n_vis), list(n_txt), hq, hkv, d, 256, dtype, keep_ratio=0.3,
                           sigma=1.0 / math.sqrt(d), seed=seed)


CASES = [
    (inputs.workload("single"), "auto"),
    (_case("ragged", 16, 16, 128, "bf16", [1, 127, 0, 700, 1536], [64, 1, 5, 33, 64]), "auto"),
    (_case("gqa", 28, 4, 128, "bf16", [1000, 2049], [128, 77]), "auto"),
    (_case("e4m3", 8, 8, 128, "e4m3", [576, 1152, 100], [32, 128, 50]), "auto"),
    (_case("reread", 16, 16, 128, "bf16", [1536, 300], [64, 16]), "reread"),
    (_case("many_requests", 4, 4, 128, "bf16", [64] * 300, [8] * 300), "auto"),
    (_case("long_request", 2, 1, 128, "bf16", [9000, 130], [40, 3]), "auto"),
]


@pytest.mark.parametrize("query", ["all", "last"])
@pytest.mark.parametrize("case", CASES, ids=lambda c: c[0].name)
def test_score_topk_equals_the_two_calls(sel, case, query):
    w, kernel = case
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    so, to = x["seq_offsets"], x["text_offsets"]
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel=kernel,
                     query=query)
    for keep_k, ratio in ((None, 0.3), ([n // 4 for n in w.n_vis], 0.0)):
        ref = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"],
                      seq_offsets_h=so, text_offsets_h=to)
        rk, roff_d, roff_h = s.topk(ref, xd["seq_offsets"], keep_k=keep_k, keep_ratio=ratio, seq_offsets_h=so)
        g, gk, goff_d, goff_h = s.score_topk(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"],
                                             xd["k_scale"], keep_k=keep_k, keep_ratio=ratio, text_offsets_h=to,
                                             seq_offsets_h=so)
        s.check_device()
        assert torch.equal(g, ref[:g.numel()])
        assert torch.equal(gk, rk)
        assert torch.equal(goff_d, roff_d) and np.array_equal(goff_h, roff_h)
        ok, ooff = oracle.topk(so, g.cpu().numpy(), keep_k=keep_k, keep_ratio=ratio)
        np.testing.assert_array_equal(gk.cpu().numpy(), ok)
    s.close()
