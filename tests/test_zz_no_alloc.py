"""litevlm_select_score_noalloc: the score path with its scratch in the
library's static device arrays, no handle and no allocation.

The GPU test compares two consecutive calls with the handle-based
litevlm_select_score on the same inputs. Both take the same launch plan and
the kernels reduce in a fixed order, so the scores must be bit-identical; the
second call runs on scratch the first one has used (each call clears the fold
tickets it needs before its launch). One case is also compared directly with
the oracle at the bf16 tolerance. Named to be collected after the other test
files, so it also runs after them in one process (and the library's static
scratch has already been used)."""
import os

import numpy as np
import pytest

from paper_2506_07416_gb300 import inputs

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sel():
    from paper_2506_07416_gb300 import _build
    if not os.path.exists(_build.LIB):
        _build.build()
    from paper_2506_07416_gb300 import select
    return select


def _case(name, hq, hkv, d, dtype, n_vis, n_txt, seed=11):
    return inputs.Workload(name, len(n_vis), list(n_vis), list(n_txt), hq, hkv, d, 256, dtype, keep_ratio=0.3,
                           sigma=1.0 / np.sqrt(d), seed=seed)


CASES = [
    inputs.workload("single"),                                                   # 16 head groups: partials + tickets
    _case("ragged", 16, 16, 128, "bf16", [1, 700, 0, 1536, 129], [64, 5, 3, 64, 33]),
    _case("gqa", 28, 4, 128, "bf16", [1000, 2049], [128, 77]),
    _case("e4m3", 8, 8, 128, "e4m3", [576, 1152, 100], [32, 128, 50]),
    _case("d64", 4, 4, 64, "bf16", [300, 5, 64], [16, 3, 1]),
]


def test_noalloc_rejects_batches_beyond_the_static_scratch(sel):
    """Host-side check, before any CUDA call: total_visual / 128 + 2 * batch + 2 > 16384."""
    so = np.array([0, 3_000_000], np.int32)
    to = np.array([0, 16], np.int32)
    with pytest.raises(sel.LitevlmError) as ei:
        sel.score_noalloc(16, 16, 128, "bf16", 1, 0, 0, to, 0, 0, so, 1.0, 1.0, 0, 8, stream=0)
    assert ei.value.name == "WORKSPACE"
    with pytest.raises(sel.LitevlmError) as ei:
        sel.score_noalloc(6, 4, 128, "bf16", 1, 0, 0, to, 0, 0, so, 1.0, 1.0, 0, 8, stream=0)
    assert ei.value.name == "INVALID_ARG"


@pytest.mark.gpu
@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_noalloc_matches_handle_path_on_two_consecutive_calls(sel, w):
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    xd = inputs.make_torch(w, "cuda")
    so, to = w.seq_offsets(), w.text_offsets()
    s = sel.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype)
    ref = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], xd["q_scale"], xd["k_scale"],
                  seq_offsets_h=so, text_offsets_h=to)
    s.check_device()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    outs = []
    for _ in range(2):
        out = torch.full((w.total_vis,), float("nan"), dtype=torch.float32, device="cuda")
        sel.score_noalloc(w.hq, w.hkv, w.head_dim, w.dtype, w.batch, xd["q"], xd["text_offsets"], to, xd["k"],
                          xd["seq_offsets"], so, xd["q_scale"], xd["k_scale"], out, err)
        outs.append(out)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    for out in outs:
        assert torch.equal(out, ref)
    s.close()


@pytest.mark.gpu
def test_noalloc_matches_the_oracle(sel):
    import oracle
    from gpu_util import assert_scores_close, to_device
    w = CASES[1]
    x = inputs.make_numpy(w)
    xd = to_device(x, w)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = torch.full((w.total_vis,), float("nan"), dtype=torch.float32, device="cuda")
    sel.score_noalloc(w.hq, w.hkv, w.head_dim, w.dtype, w.batch, xd["q"], xd["text_offsets"], x["text_offsets"],
                      xd["k"], xd["seq_offsets"], x["seq_offsets"], 1.0, 1.0, out, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    o = oracle.score(x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype)
    assert_scores_close(out.cpu().numpy(), o, w.dtype)


@pytest.mark.gpu
def test_noalloc_rejects_head_groups_beyond_the_partial_scratch(sel):
    """Limit 2: a launch that splits the query heads over G > 1 groups needs G x
    total_visual partial scores; beyond the static 1048576 floats the call
    returns WORKSPACE, enqueues nothing and leaves the output as it was."""
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    found = None
    for n, t, hq, hkv in ((65536, 64, 32, 32), (60000, 128, 28, 4), (50000, 16, 16, 16), (65536, 128, 32, 8)):
        so = np.array([0, n], np.int32)
        to = np.array([0, t], np.int32)
        s = sel.Selector(1, n, t, hq, hkv, 128, "bf16")
        plan = s.score_plan(to, so)
        s.close()
        if plan[0] not in (4, 7) and plan[3] > 1 and plan[3] * n > (1 << 20):
            found = (n, t, hq, hkv, so, to)
            break
    assert found is not None, "no shape among the candidates splits its heads beyond the scratch"
    n, t, hq, hkv, so, to = found
    q = torch.zeros((t, hq, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((n, hkv, 128), dtype=torch.bfloat16, device="cuda")
    so_d, to_d = torch.from_numpy(so).cuda(), torch.from_numpy(to).cuda()
    out = torch.full((n,), float("nan"), dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(sel.LitevlmError) as ei:
        sel.score_noalloc(hq, hkv, 128, "bf16", 1, q, to_d, to, k, so_d, so, 1.0, 1.0, out, err)
    assert ei.value.name == "WORKSPACE"
    torch.cuda.synchronize()
    assert bool(torch.isnan(out).all()) and int(err.item()) == 0
