"""Canary guard bands around every output of the selection path.

Each output buffer (scores, kept indices, output offsets, gathered rows) is
carved out of a larger device allocation whose bytes before and after it are
filled with a canary pattern. After score, top-k, the one-call score + top-k
and the gather, the outputs must equal the oracle's and every canary byte must
still be there: no kernel writes outside its output. The cases span the
kernels and schedules the planner picks (resident with one and two TMEM
buffers, the flattened schedule, the re-read kernel, e4m3) and ragged tails."""
import math

import numpy as np
import pytest

import oracle
from gpu_util import assert_scores_close, to_device
from paper_2506_07416_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

CANARY = 0xA5
GUARD = 4096  # bytes on each side (a multiple of 256, so the outputs stay aligned)


@pytest.fixture(scope="module")
def sel():
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    from paper_2506_07416_gb300 import select
    return select


class Guarded:
    """A device tensor of `shape` / `dtype` inside a canary-filled byte buffer."""

    def __init__(self, shape, dtype):
        shape = tuple(shape)
        eb = torch.empty((), dtype=dtype).element_size()
        self.nbytes = int(np.prod(shape, dtype=np.int64)) * eb
        self.raw = torch.full((GUARD + self.nbytes + GUARD,), CANARY, dtype=torch.uint8, device="cuda")
        self.t = self.raw[GUARD:GUARD + self.nbytes].view(dtype).view(shape)

    def intact(self):
        head = self.raw[:GUARD]
        tail = self.raw[GUARD + self.nbytes:]
        return bool((head == CANARY).all()) and bool((tail == CANARY).all())


def _wl(name, n, t, hq=8, hkv=8, d=128, dtype="bf16", seed=61):
    return inputs.Workload(name, len(n), list(n), list(t), hq, hkv, d, 256, dtype, keep_ratio=0.3,
                           sigma=1.0 / math.sqrt(d), seed=seed, gather=("hidden", "k", "v"))


CASES = [
    (_wl("ragged_resident", [700, 129, 1536, 1], [64, 16, 40, 7]), "auto"),
    (_wl("two_buffers", [384, 256, 130], [32, 16, 20], hq=16, hkv=16, seed=62), "resident_2buf"),
    (_wl("flat_uniform", [3 * 128 + 5] * 12, [48] * 12, seed=63), "resident_flat"),
    (_wl("reread_long_text", [1000, 77], [128, 100], hq=28, hkv=4, seed=64), "reread"),
    (_wl("e4m3_ragged", [576, 1152, 100], [32, 128, 71], dtype="e4m3", seed=65), "auto"),
]


@pytest.mark.parametrize("w,kern", CASES, ids=lambda c: c.name if hasattr(c, "name") else c)
def test_outputs_stay_inside_their_buffers(sel, w, kern):
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    so, to = x["seq_offsets"], x["text_offsets"]
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype, score_kernel=kern)

    # scores
    sc = Guarded((w.total_vis,), torch.float32)
    s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"], out=sc.t,
            seq_offsets_h=so, text_offsets_h=to)
    s.check_device()
    assert sc.intact()
    g = sc.t.cpu().numpy()
    o = oracle.score(x["q"], x["k"], so, to, w.hq, w.hkv, w.head_dim, w.dtype, x["q_scale"], x["k_scale"])
    assert_scores_close(g, o, w.dtype)

    # top-k on the GPU scores
    okept, ooff = oracle.topk(so, g, keep_ratio=0.3)
    kept = Guarded((max(1, len(okept)),), torch.int32)
    off = Guarded((w.batch + 1,), torch.int32)
    k_out, off_d, off_h = s.topk(sc.t, xd["seq_offsets"], keep_ratio=0.3, seq_offsets_h=so, kept_idx=kept.t,
                                 out_offsets=off.t)
    s.check_device()
    assert kept.intact() and off.intact()
    np.testing.assert_array_equal(k_out.cpu().numpy(), okept)
    np.testing.assert_array_equal(off_d.cpu().numpy(), ooff)

    # one-call score + top-k into guarded buffers (same bits and indices)
    sc2 = Guarded((w.total_vis,), torch.float32)
    kept2 = Guarded((max(1, len(okept)),), torch.int32)
    off2 = Guarded((w.batch + 1,), torch.int32)
    s2, k2, o2d, _ = s.score_topk(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"],
                                  xd["k_scale"], keep_ratio=0.3, seq_offsets_h=so, text_offsets_h=to,
                                  out=sc2.t, kept_idx=kept2.t, out_offsets=off2.t)
    s.check_device()
    assert sc2.intact() and kept2.intact() and off2.intact()
    assert np.array_equal(s2.cpu().numpy().view(np.uint32), g.view(np.uint32))
    np.testing.assert_array_equal(k2.cpu().numpy(), okept)
    np.testing.assert_array_equal(o2d.cpu().numpy(), ooff)

    # gather of hidden, K and V rows into guarded buffers
    srcs = [xd["hidden"], xd["k"], xd["v"]]
    dsts = [Guarded((len(okept),) + tuple(t.shape[1:]), t.dtype) for t in srcs]
    s.compact(k_out, len(okept), srcs, [d.t for d in dsts])
    s.check_device()
    for d, name in zip(dsts, ("hidden", "k", "v")):
        assert d.intact(), name
        got = d.t.cpu()
        ref = oracle.compact(okept, x[name])
        np.testing.assert_array_equal(got.view(torch.int16).numpy().view(ref.dtype) if got.dtype == torch.bfloat16
                                      else got.numpy().view(ref.dtype), ref)
    s.close()
