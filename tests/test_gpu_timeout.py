"""The device-side failure path of the score kernels, made to run on purpose
without faulting, trapping or hanging the GPU.

Every wait of the kernels (mbarrier phases, cluster arrivals) is bounded by the
handle's wait budget. With LITEVLM_DEBUG_STALL_SCORE the TMA producer of either
score kernel first waits on an mbarrier that nothing completes,
before it issues any copy, so that wait runs out of budget; every other wait of
the launch then gives up too, with no copy or contraction in flight. The test
checks that the launch ends by itself, that check_device reports TIMEOUT, and
that the same handle is then exact again: the error word was cleared and the
fold tickets the aborted launch left taken were reset (the request's heads are
split over several CTA groups, so the fold tickets are in use)."""
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


def _score(s, x, xd):
    return s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"],
                   seq_offsets_h=x["seq_offsets"], text_offsets_h=x["text_offsets"])


def test_wait_timeout_is_reported_and_the_handle_recovers(sel):
    w = inputs.workload("single")
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype)
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] in (2, 3) and plan[3] > 1, plan  # resident kernel, heads split over CTA groups

    s.set_wait_budget(20000)  # about 10 us at 2 GHz
    s.set_debug_flags(sel.DEBUG_STALL_SCORE)
    _score(s, x, xd)
    with pytest.raises(sel.LitevlmError) as ei:
        s.check_device()
    assert ei.value.name == "TIMEOUT"

    # back to normal on the same handle: exact against the oracle, and the same
    # bits as a fresh handle (fold tickets at rest again)
    s.set_debug_flags(0)
    s.set_wait_budget(0)
    g = _score(s, x, xd).cpu().numpy()
    s.check_device()
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype)
    assert_scores_close(g, o, w.dtype)
    fresh = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype)
    g2 = _score(fresh, x, xd).cpu().numpy()
    fresh.check_device()
    assert np.array_equal(g.view(np.uint32), g2.view(np.uint32))
    # a second timeout on the same handle is reported again, then cleared again
    s.set_wait_budget(20000)
    s.set_debug_flags(sel.DEBUG_STALL_SCORE)
    _score(s, x, xd)
    with pytest.raises(sel.LitevlmError) as ei:
        s.check_device()
    assert ei.value.name == "TIMEOUT"
    s.set_debug_flags(0)
    s.set_wait_budget(0)
    g3 = _score(s, x, xd).cpu().numpy()
    s.check_device()
    assert np.array_equal(g.view(np.uint32), g3.view(np.uint32))
    fresh.close()
    s.close()


def test_wait_timeout_in_the_reread_kernel(sel):
    """The same failure path in the kernel that streams K twice per head: its
    producer stalls the same way, the launch gives up within the budget, and the
    handle is exact again afterwards (the heads are split over CTA groups, so
    the fold tickets are in use here too)."""
    w = inputs.workload("single")
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="reread")
    plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
    assert plan[0] == 1 and plan[3] > 1, plan  # re-read kernel, heads split over CTA groups

    s.set_wait_budget(20000)
    s.set_debug_flags(sel.DEBUG_STALL_SCORE)
    _score(s, x, xd)
    with pytest.raises(sel.LitevlmError) as ei:
        s.check_device()
    assert ei.value.name == "TIMEOUT"

    s.set_debug_flags(0)
    s.set_wait_budget(0)
    g = _score(s, x, xd).cpu().numpy()
    s.check_device()
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype)
    assert_scores_close(g, o, w.dtype)
    fresh = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel="reread")
    g2 = _score(fresh, x, xd).cpu().numpy()
    fresh.check_device()
    assert np.array_equal(g.view(np.uint32), g2.view(np.uint32))
    fresh.close()
    s.close()


def test_debug_setters_reject_bad_values(sel):
    s = sel.Selector(1, 128, 16, 4, 4, 64, "bf16")
    with pytest.raises(sel.LitevlmError) as ei:
        s.set_debug_flags(2)
    assert ei.value.name == "INVALID_ARG"
    with pytest.raises(sel.LitevlmError) as ei:
        s.set_wait_budget(-1)
    assert ei.value.name == "INVALID_ARG"
    s.close()
