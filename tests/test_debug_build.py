"""The debug variant of the library (NVTX ranges around every C-ABI call,
device / host mirror checks): it builds, loads without a GPU and exports every
declared function (host part); on a GPU, run in a child process that loads it
through LITEVLM_LIB, its results match the oracle and a device offsets array
that differs from its host mirror is refused with INVALID_ARG before any
launch."""
import ctypes
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def debug_lib():
    from paper_2506_07416_gb300 import _build
    return _build.build(debug=True)


def test_debug_variant_builds_and_exports_every_symbol(debug_lib):
    from test_abi_host import declared_functions
    lib = ctypes.CDLL(debug_lib)
    for n in declared_functions():
        assert hasattr(lib, n), n


CHILD = r'''
import json, math, sys
import numpy as np
import torch
sys.path.insert(0, sys.argv[1]); sys.path.insert(0, sys.argv[1] + "/tests")
import oracle
from gpu_util import to_device, rel_err
from paper_2506_07416_gb300 import inputs, select
out = {"lib": select.LIB_PATH}
w = inputs.Workload("dbg", 3, [300, 129, 640], [16, 40, 7], 8, 4, 128, 256, "bf16", keep_ratio=0.3,
                    sigma=1 / math.sqrt(128), seed=71)
x = inputs.make_numpy(w)
xd = to_device(x, w)
s = select.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, "bf16")
so, to = x["seq_offsets"], x["text_offsets"]
g = s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], seq_offsets_h=so, text_offsets_h=to)
kept, off_d, off_h = s.topk(g, xd["seq_offsets"], keep_ratio=0.3, seq_offsets_h=so)
s.check_device()
o = oracle.score(x["q"], x["k"], so, to, w.hq, w.hkv, w.head_dim, "bf16")
out["max_rel"] = float(rel_err(g.cpu().numpy(), o))
ok, ooff = oracle.topk(so, g.cpu().numpy(), keep_ratio=0.3)
out["topk_equal"] = bool(np.array_equal(kept.cpu().numpy(), ok)) and bool(np.array_equal(off_h, ooff))
# a host mirror that differs from the device array
bad = so.copy(); bad[1] += 1
try:
    s.score(xd["q"], xd["text_offsets"], xd["k"], xd["seq_offsets"], seq_offsets_h=bad, text_offsets_h=to)
    out["mirror"] = "accepted"
except select.LitevlmError as e:
    out["mirror"] = [e.name, str(e)]
kk = np.full(w.batch, 5, np.int32)
try:
    k_d = torch.from_numpy(kk + 1).cuda()  # differs from the host keep_k
    select.topk(s.handle, w.batch, g, xd["seq_offsets"], so, k_d, kk, 0.0,
                torch.empty(64, dtype=torch.int32, device="cuda"), torch.empty(4, dtype=torch.int32, device="cuda"),
                np.zeros(4, np.int32), None)
    out["keep_mirror"] = "accepted"
except select.LitevlmError as e:
    out["keep_mirror"] = [e.name, str(e)]
s.check_device()
print(json.dumps(out))
'''


@pytest.mark.gpu
def test_debug_variant_matches_the_oracle_and_checks_mirrors(debug_lib):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.fail("the GPU tests need a CUDA device")
    env = dict(os.environ, LITEVLM_LIB=debug_lib)
    r = subprocess.run([sys.executable, "-c", CHILD, ROOT], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-3000:]
    out = json.loads(r.stdout.strip().splitlines()[-1])
    assert out["lib"] == debug_lib
    assert out["max_rel"] < 2e-3, out
    assert out["topk_equal"], out
    assert out["mirror"][0] == "INVALID_ARG" and "differs from its host mirror" in out["mirror"][1], out
    assert out["keep_mirror"][0] == "INVALID_ARG" and "keep_k" in out["keep_mirror"][1], out
