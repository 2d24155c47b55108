"""Parity of the layer-0 projection (litevlm_select_fold_norm / rope_table /
project) with the oracle's fp64 RoPE(W . RMSNorm(x) + b), through the C-ABI.

Bar, derived from the arithmetic: the GPU rounds W * gamma to bf16 once
(relative 2^-9 per weight, random signs: about 1.1e-3 x rms(y) per output,
under 8e-3 x rms(y) at five sigma) and the output to bf16 (2^-9 |y|); the fp32
accumulation, the fp32 RoPE angle (below 3e-4 rad for positions < 4096) and
sincosf add far less. So |gpu - oracle| <= 4e-3 |oracle| + 1e-2 rms(oracle).
A transposed weight, a wrong pairing or sign of the rotation, a dropped norm
or bias each miss it by orders of magnitude."""
import math

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
    s = select.Selector(4, 4096, 1024, 4, 4, 128, "bf16")
    yield s
    s.close()


def _bf16_dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16).copy()).view(torch.bfloat16).cuda()


def _close(g, o):
    rms = float(np.sqrt(np.mean(o * o)))
    err = np.abs(g - o)
    bad = err > 4e-3 * np.abs(o) + 1e-2 * rms
    assert not bad.any(), f"{int(bad.sum())} of {o.size} outside; max err / rms {float(err.max()) / rms:.3e}"


def _run(sel, rows, hidden, out_f, head_dim, bias, eps=1e-6, base=1e6, max_pos=4096, seed=6):
    x, g, w, b, pos = inputs.projection_numpy(rows, hidden, out_f, seed=seed, bias=bias, max_position=max_pos)
    wf = sel.fold_norm(_bf16_dev(w), torch.from_numpy(g).cuda())
    table = sel.rope_table(max_pos, head_dim, base) if head_dim else None
    y = sel.project(_bf16_dev(x), wf, None if b is None else torch.from_numpy(b).cuda(), eps, head_dim,
                    torch.from_numpy(pos).cuda() if head_dim else None, table)
    sel.check_device()
    gy = y.float().cpu().numpy()
    oy = oracle.project(x, g, eps, w, b, head_dim, pos, base)
    _close(gy, oy)
    return gy, oy


@pytest.mark.parametrize("rows,hidden,out_f,head_dim,bias", [
    (300, 2048, 2048, 128, False),   # keys of 16 heads x 128 from hidden 2048, ragged last row tile
    (77, 896, 896, 64, True),        # queries of 14 heads x 64 with bias, hidden not a multiple of 64
    (129, 136, 384, 0, False),       # no rotation, 128-column tiles
    (200, 3584, 512, 128, True),     # 4 KV heads x 128 from hidden 3584
    (1, 512, 256, 128, False),       # one row
    (4900, 128, 4096, 128, True),    # enough tiles for the 256-row variant, ragged last tile
])
def test_project_matches_oracle(sel, rows, hidden, out_f, head_dim, bias):
    _run(sel, rows, hidden, out_f, head_dim, bias)


def test_project_fold_is_w_times_gamma(sel):
    """fold_norm alone: bit-exact bf16(w * gamma) (one fp32 product, rounded once)."""
    rng = np.random.Generator(np.random.PCG64(3))
    w = inputs.f32_to_bf16_bits(rng.standard_normal((256, 200)).astype(np.float32))
    g = rng.uniform(0.5, 1.5, 200).astype(np.float32)
    got = sel.fold_norm(_bf16_dev(w), torch.from_numpy(g).cuda()).view(torch.int16).cpu().numpy().view(np.uint16)
    want = inputs.f32_to_bf16_bits(inputs.bf16_bits_to_f32(w) * g[None, :])
    np.testing.assert_array_equal(got, want)


def test_rope_table_values(sel):
    t = sel.rope_table(5000, 128, 1e6).cpu().numpy().astype(np.float64)
    p = np.arange(5000)[:, None]
    theta = np.power(1e6, -2.0 * np.arange(64) / 128.0)
    a = p * theta[None, :]
    np.testing.assert_allclose(t[..., 0], np.cos(a), atol=5e-4)  # fp32 angle: |error| < 5000 * 2^-24 * 2
    np.testing.assert_allclose(t[..., 1], np.sin(a), atol=5e-4)


def test_project_bad_positions_flagged(sel):
    from paper_2506_07416_gb300 import select
    x, g, w, b, pos = inputs.projection_numpy(10, 256, 256, seed=8)
    wf = sel.fold_norm(_bf16_dev(w), torch.from_numpy(g).cuda())
    table = sel.rope_table(64, 128, 1e4)
    pos = pos % 64
    pos[3] = 64
    sel.project(_bf16_dev(x), wf, None, 1e-6, 128, torch.from_numpy(pos).cuda(), table)
    with pytest.raises(select.LitevlmError) as e:
        sel.check_device()
    assert e.value.name == "DEVICE_BOUNDS"
    with pytest.raises(select.LitevlmError) as e:
        sel.project(_bf16_dev(x), wf, None, 1e-6, 96, torch.from_numpy(pos).cuda(), table)
    assert e.value.name == "UNSUPPORTED"


def test_projection_feeds_the_scores(sel):
    """x -> q, k on the GPU -> scores, against the oracle chain (projection in
    fp64, rounded to bf16, then the score): the two q / k differ by bf16
    roundings, so the scores agree to the e4m3 tolerance."""
    from gpu_util import assert_scores_close
    from paper_2506_07416_gb300 import select
    H, hq, d, N, T = 512, 4, 128, 700, 24
    xv, g, wk, _, _ = inputs.projection_numpy(N, H, hq * d, seed=11)
    xt, _, wq, _, _ = inputs.projection_numpy(T, H, hq * d, seed=12)
    pos_v = (16 + np.arange(N)).astype(np.int32)
    pos_t = (16 + N + np.arange(T)).astype(np.int32)
    table = sel.rope_table(2048, d, 1e6)
    gk = sel.project(_bf16_dev(xv), sel.fold_norm(_bf16_dev(wk), torch.from_numpy(g).cuda()), None, 1e-6, d,
                     torch.from_numpy(pos_v).cuda(), table)
    gq = sel.project(_bf16_dev(xt), sel.fold_norm(_bf16_dev(wq), torch.from_numpy(g).cuda()), None, 1e-6, d,
                     torch.from_numpy(pos_t).cuda(), table)
    so = np.array([0, N], np.int32)
    to = np.array([0, T], np.int32)
    s = select.Selector(1, N, T, hq, hq, d, "bf16")
    sc = s.score(gq.view(T, hq, d), torch.from_numpy(to).cuda(), gk.view(N, hq, d), torch.from_numpy(so).cuda(),
                 seq_offsets_h=so, text_offsets_h=to).cpu().numpy()
    s.check_device()
    qo = inputs.f32_to_bf16_bits(oracle.project(xt, g, 1e-6, wq, None, d, pos_t, 1e6).astype(np.float32))
    ko = inputs.f32_to_bf16_bits(oracle.project(xv, g, 1e-6, wk, None, d, pos_v, 1e6).astype(np.float32))
    o = oracle.score(qo.reshape(T, hq, d), ko.reshape(N, hq, d), so, to, hq, hq, d, "bf16")
    assert_scores_close(sc, o, "e4m3")
    s.close()


def _e4m3_decode(codes_u8, scale):
    return torch.from_numpy(codes_u8).view(torch.float8_e4m3fn).float().numpy().astype(np.float64) * scale


def test_project_e4m3_output(sel):
    """e4m3 output under a static per-tensor scale: the codes decode to the
    oracle's y within the e4m3 rounding (at most 1/16 relative for normal
    values) plus a small absolute term for the subnormal range; with a scale
    too small, values saturate at +-448 * scale instead of overflowing."""
    rows, H, O, d = 300, 1024, 512, 128
    x, g, w, b, pos = inputs.projection_numpy(rows, H, O, seed=13, bias=True, max_position=2048)
    wf = sel.fold_norm(_bf16_dev(w), torch.from_numpy(g).cuda())
    table = sel.rope_table(2048, d, 1e6)
    oy = oracle.project(x, g, 1e-6, w, b, d, pos, 1e6)
    scale = float(np.abs(oy).max()) / 448.0
    y8 = sel.project(_bf16_dev(x), wf, torch.from_numpy(b).cuda(), 1e-6, d, torch.from_numpy(pos).cuda(), table,
                     out_scale=scale)
    sel.check_device()
    assert y8.dtype == torch.uint8
    gy = _e4m3_decode(y8.cpu().numpy(), scale)
    rms = float(np.sqrt(np.mean(oy * oy)))
    bad = np.abs(gy - oy) > 0.0625 * np.abs(oy) + 0.02 * rms
    assert not bad.any(), int(bad.sum())
    small = scale / 8
    y8 = sel.project(_bf16_dev(x), wf, torch.from_numpy(b).cuda(), 1e-6, d, torch.from_numpy(pos).cuda(), table,
                     out_scale=small)
    gs = _e4m3_decode(y8.cpu().numpy(), small)
    assert np.all(np.isfinite(gs)) and np.abs(gs).max() <= 448 * small * (1 + 1e-6)
    big = np.abs(oy) > 448 * small * 1.1
    assert np.all(np.abs(gs[big]) == 448 * small)


def test_e4m3_projection_feeds_the_e4m3_scores(sel):
    """x -> e4m3 q, k (static scales) -> the e4m3 score kernel, against the
    oracle chain (fp64 projection, the same scales, torch's e4m3 rounding, the
    e4m3 score oracle); the two codes may differ by one e4m3 rounding, so the
    scores agree to the e4m3 tolerance."""
    from gpu_util import assert_scores_close
    from paper_2506_07416_gb300 import select
    H, hq, d, N, T = 512, 8, 128, 700, 40
    xv, g, wk, _, _ = inputs.projection_numpy(N, H, hq * d, seed=21)
    xt, _, wq, _, _ = inputs.projection_numpy(T, H, hq * d, seed=22)
    pos_v = (16 + np.arange(N)).astype(np.int32)
    pos_t = (16 + N + np.arange(T)).astype(np.int32)
    ko = oracle.project(xv, g, 1e-6, wk, None, d, pos_v, 1e6)
    qo = oracle.project(xt, g, 1e-6, wq, None, d, pos_t, 1e6)
    ks, qs = float(np.abs(ko).max()) / 448.0, float(np.abs(qo).max()) / 448.0
    table = sel.rope_table(2048, d, 1e6)
    gk = sel.project(_bf16_dev(xv), sel.fold_norm(_bf16_dev(wk), torch.from_numpy(g).cuda()), None, 1e-6, d,
                     torch.from_numpy(pos_v).cuda(), table, out_scale=ks)
    gq = sel.project(_bf16_dev(xt), sel.fold_norm(_bf16_dev(wq), torch.from_numpy(g).cuda()), None, 1e-6, d,
                     torch.from_numpy(pos_t).cuda(), table, out_scale=qs)
    so, to = np.array([0, N], np.int32), np.array([0, T], np.int32)
    s = select.Selector(1, N, T, hq, hq, d, "e4m3")
    sc = s.score(gq.view(T, hq, d), torch.from_numpy(to).cuda(), gk.view(N, hq, d), torch.from_numpy(so).cuda(),
                 q_scale=qs, k_scale=ks, seq_offsets_h=so, text_offsets_h=to).cpu().numpy()
    s.check_device()
    enc = lambda a, sc_: torch.from_numpy((a / sc_).astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    o = oracle.score(enc(qo, qs).reshape(T, hq, d), enc(ko, ks).reshape(N, hq, d), so, to, hq, hq, d, "e4m3", qs, ks)
    assert_scores_close(sc, o, "e4m3")
    s.close()
