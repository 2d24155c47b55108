"""Parity of litevlm_select_views (patch-selection gating) with the oracle,
through the C-ABI. The outputs are integers decided by fp32 scores that both
sides compute the same way (two products and a sum, no contraction), so every
output must be bit-exact: ragged batches over several 1024-request chunks,
1 to 64 views, ties, NaN and infinite logits, a score exactly at the
threshold, and min_views from 0 to V."""
import numpy as np
import pytest

import oracle
from paper_2506_07416_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sel():
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    from paper_2506_07416_gb300 import select
    s = select.Selector(4, 1024, 1024, 4, 4, 128, "bf16")
    yield s
    s.close()


def _check(s, lex, lg, tpv, w_lex, w_logit, thr, min_views):
    mask, vo, sv, so, so_h = s.select_views(torch.from_numpy(lex).cuda(), torch.from_numpy(lg).cuda(), tpv, w_lex,
                                            w_logit, thr, min_views)
    s.check_device()
    om, ovo, osv, oso = oracle.select_views(lex, lg, tpv, w_lex, w_logit, thr, min_views)
    np.testing.assert_array_equal(mask.cpu().numpy(), om)
    np.testing.assert_array_equal(vo.cpu().numpy(), ovo)
    np.testing.assert_array_equal(sv.cpu().numpy()[:int(ovo[-1])], osv)
    np.testing.assert_array_equal(so.cpu().numpy(), oso)
    np.testing.assert_array_equal(so_h, oso)
    return om, oso


@pytest.mark.parametrize("batch,num_views,min_views", [(1, 6, 1), (7, 6, 0), (1000, 6, 1), (3000, 12, 2),
                                                       (5000, 64, 3), (33, 1, 1), (200, 6, 6)])
def test_views_match_oracle(sel, batch, num_views, min_views):
    lex, lg = inputs.view_gating_numpy(batch, num_views, seed=batch + num_views)
    tpv = (np.arange(num_views) % 3 + 1).astype(np.int32) * 256
    _check(sel, lex, lg, tpv, 1.5, 1.0, 1.0, min_views)


def test_views_ties_nan_inf_and_exact_threshold(sel):
    lex, lg = inputs.view_gating_numpy(2000, 6, seed=9, quantum=0.5)  # many equal scores
    lg[::7, 2] = np.nan
    lg[::11, 4] = np.inf
    lg[::13, 1] = -np.inf
    lex[::5, 3] = 1.0
    lg[::5, 3] = -1.5  # 2 * 1 + 1 * (-1.5) = 0.5 = threshold exactly: not selected
    tpv = np.full(6, 512, np.int32)
    for mv in (0, 1, 2, 6):
        m, so = _check(sel, lex, lg, tpv, 2.0, 1.0, 0.5, mv)
        if mv == 0:
            assert not m[::5, 3].any()


def test_views_empty_batch_and_errors(sel):
    z = np.zeros((0, 6), np.float32)
    mask, vo, sv, so, so_h = sel.select_views(torch.from_numpy(z).cuda(), torch.from_numpy(z).cuda(),
                                              np.full(6, 256, np.int32), 1.0, 1.0, 0.0, 0)
    assert vo.cpu().tolist() == [0] and so_h.tolist() == [0]
    from paper_2506_07416_gb300 import select
    lex, lg = inputs.view_gating_numpy(4, 6)
    with pytest.raises(select.LitevlmError) as e:
        sel.select_views(torch.from_numpy(lex).cuda(), torch.from_numpy(lg).cuda(), np.full(6, 256, np.int32),
                         1.0, 1.0, 0.0, 7)
    assert e.value.name == "INVALID_ARG"
    with pytest.raises(select.LitevlmError) as e:
        sel.select_views(torch.from_numpy(lex).cuda(), torch.from_numpy(lg).cuda(), np.full(6, -1, np.int32),
                         1.0, 1.0, 0.0, 0)
    assert e.value.name == "INVALID_ARG"
    sel.check_device()


def test_views_feed_the_score_path(sel):
    """Gating -> N_b -> scores: the selected views' tokens become the visual
    rows of the score call, whose offsets come from the gating output."""
    from paper_2506_07416_gb300 import select
    lex, lg = inputs.view_gating_numpy(5, 6, seed=21)
    tpv = np.full(6, 64, np.int32)
    _, vo, sv, so_d, so_h = sel.select_views(torch.from_numpy(lex).cuda(), torch.from_numpy(lg).cuda(), tpv, 2.0,
                                             1.0, 1.0, 1)
    n_vis = np.diff(so_h).tolist()
    w = inputs.Workload("gated", 5, n_vis, [16] * 5, 4, 4, 128, 256, "bf16", keep_ratio=0.5, sigma=1 / np.sqrt(128),
                        seed=3)
    x = inputs.make_numpy(w)
    s = select.Selector(5, w.total_vis, w.total_txt, 4, 4, 128, "bf16")
    q = torch.from_numpy(x["q"].view(np.int16).copy()).view(torch.bfloat16).cuda()
    k = torch.from_numpy(x["k"].view(np.int16).copy()).view(torch.bfloat16).cuda()
    to = torch.from_numpy(x["text_offsets"]).cuda()
    g = s.score(q, to, k, so_d, seq_offsets_h=so_h, text_offsets_h=x["text_offsets"]).cpu().numpy()
    s.check_device()
    o = oracle.score(x["q"], x["k"], so_h, x["text_offsets"], 4, 4, 128, "bf16")
    from gpu_util import assert_scores_close
    assert_scores_close(g, o, "bf16")
    s.close()
