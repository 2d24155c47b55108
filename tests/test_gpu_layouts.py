"""The two shared-memory layouts of the TMEM-resident score kernel at 256-byte
K rows (bf16, d = 128) and up to 64 text rows. The compact layout keeps score
rows for at most 8 tiles per CTA and statistics for at most 320 cluster x slot
columns, which leaves room for a fifth K stage; the full layout has neither
limit. A launch takes the compact layout whenever its plan fits. The shapes
below are picked so that the planner's choices cover both layouts, and every
one is checked against the oracle; the two MMA-issuing threads share the K
ring differently with four and five stages (which thread last used a stage),
so both orders are exercised."""
import math

import numpy as np
import pytest

import oracle
from gpu_util import assert_scores_close, to_device
from paper_2506_07416_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

COMPACT_TILES, COMPACT_COLS = 8, 320


@pytest.fixture(scope="module")
def sel():
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    from paper_2506_07416_gb300 import select
    return select


def _wl(name, n, t, hq=16, hkv=16, seed=31):
    return inputs.Workload(name, len(n), list(n), list(t), hq, hkv, 128, 256, "bf16", keep_ratio=0.3,
                           sigma=1.0 / math.sqrt(128), seed=seed)


CASES = [
    # (workload, score kernel option)
    (_wl("one_large", [6144], [64]), "auto"),
    (_wl("one_large_1buf", [4096], [60], seed=32), "resident_1buf"),
    (_wl("mixed", [3000, 2500, 2048, 1000], [64, 50, 60, 33], seed=33), "auto"),
    (_wl("uniform_small", [900] * 24, [64] * 24, seed=34), "auto"),
    (_wl("gqa_two_buffers", [1024] * 6, [40] * 6, hq=28, hkv=4, seed=35), "resident_2buf"),
    (_wl("odd_tiles", [7 * 128 - 5] * 10, [64] * 10, seed=36), "resident_flat"),
]


def _layout(plan, max_t):
    slot_cols = (max_t + 15) & ~15
    if plan[0] not in (2, 3, 4):
        return "reread"
    return "compact" if plan[2] <= COMPACT_TILES and plan[1] * slot_cols <= COMPACT_COLS else "full"


def test_both_layouts_match_the_oracle(sel):
    seen = set()
    for w, kern in CASES:
        x = inputs.make_numpy(w)
        xd = to_device(x, w)
        s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel=kern)
        plan = s.score_plan(x["text_offsets"], x["seq_offsets"])
        lay = _layout(plan, int(np.max(np.diff(x["text_offsets"]))))
        assert lay != "reread", (w.name, plan)
        seen.add(lay)
        g = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], seq_offsets_h=x["seq_offsets"],
                    text_offsets_h=x["text_offsets"])
        s.check_device()
        g = g.cpu().numpy()
        o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype)
        assert_scores_close(g, o, w.dtype)
        # repeated launches give the same bits (the ring's order of stages and
        # threads is fixed by the plan)
        for _ in range(3):
            g2 = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], seq_offsets_h=x["seq_offsets"],
                         text_offsets_h=x["text_offsets"])
            s.check_device()
            assert np.array_equal(g.view(np.uint32), g2.cpu().numpy().view(np.uint32)), (w.name, plan)
        s.close()
    assert seen == {"compact", "full"}, seen
