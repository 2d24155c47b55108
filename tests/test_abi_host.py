"""The C-ABI library on the host: it loads without a GPU, exports every function
declared in include/litevlm_select.h, its config struct matches the header, and
argument errors are reported before any CUDA work. No compute calls here."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "litevlm_select.h")


@pytest.fixture(scope="module")
def sel():
    from paper_2506_07416_gb300 import _build
    if not os.path.exists(_build.LIB):
        _build.build()
    from paper_2506_07416_gb300 import select
    return select


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(litevlm_\w+)\s*\(", text)))


def test_exports_every_declared_symbol(sel):
    names = declared_functions()
    assert len(names) >= 8
    lib = ctypes.CDLL(sel.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(sel.EXPORTS) == names


def test_config_struct_layout_matches_header(tmp_path, sel):
    src = tmp_path / "layout.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "litevlm_select.h"\n'
                   "int main(void){printf(\"%zu %zu %zu %zu %zu %zu %zu %zu %zu\\n\", sizeof(litevlm_select_config_t),"
                   "offsetof(litevlm_select_config_t,max_batch),offsetof(litevlm_select_config_t,max_total_visual),"
                   "offsetof(litevlm_select_config_t,max_total_text),offsetof(litevlm_select_config_t,num_q_heads),"
                   "offsetof(litevlm_select_config_t,num_kv_heads),offsetof(litevlm_select_config_t,head_dim),"
                   "offsetof(litevlm_select_config_t,qk_dtype),offsetof(litevlm_select_config_t,flags));return 0;}\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)], check=True)
    got = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    C = sel.Config
    want = [ctypes.sizeof(C)] + [getattr(C, f).offset for f, _ in C._fields_]
    assert got == want


def test_status_strings(sel):
    for code in range(7):
        s = sel.LIB.litevlm_status_string(code)
        assert s and s != b"unknown status"
    assert sel.LIB.litevlm_status_string(99) == b"unknown status"


def _cfg(sel, **kw):
    base = dict(max_batch=4, max_total_visual=1024, max_total_text=256, num_q_heads=8, num_kv_heads=2,
                head_dim=128, qk_dtype=0, flags=0)
    base.update(kw)
    return sel.Config(**base)


@pytest.mark.parametrize("kw,status", [
    (dict(num_q_heads=6, num_kv_heads=4), 1),
    (dict(max_batch=0), 1),
    (dict(max_total_visual=-5), 1),
    (dict(flags=3), 1),
    (dict(flags=-1), 1),
    (dict(flags=2 | 128 | 512), 1),  # an unknown bit beside valid ones
    (dict(flags=256), 1),
    (dict(qk_dtype=7), 1),
    (dict(head_dim=96), 2),
    (dict(head_dim=64, qk_dtype=1), 2),
])
def test_create_rejects_bad_config_before_cuda(sel, kw, status):
    h = ctypes.c_void_p(1234)
    rc = sel.LIB.litevlm_select_create(ctypes.byref(_cfg(sel, **kw)), ctypes.byref(h))
    assert rc == status
    assert h.value is None
    assert sel.LIB.litevlm_select_last_error(None)


def test_null_arguments(sel):
    h = ctypes.c_void_p()
    assert sel.LIB.litevlm_select_create(None, ctypes.byref(h)) == 1
    assert sel.LIB.litevlm_select_create(ctypes.byref(_cfg(sel)), None) == 1
    assert sel.LIB.litevlm_select_destroy(None) == 0
    assert sel.LIB.litevlm_select_score(None, 1, None, None, None, None, None, None, 1.0, 1.0, None, None) == 1
    assert sel.LIB.litevlm_select_topk(None, 1, None, None, None, None, None, 0.5, None, None, None, None) == 1
    assert sel.LIB.litevlm_select_compact(None, 1, None, 1, 1, None, None, None, None) == 1
    assert sel.LIB.litevlm_select_check_device(None, None) == 1


def test_create_without_gpu_reports_cuda_error(sel):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    h = ctypes.c_void_p()
    rc = sel.LIB.litevlm_select_create(ctypes.byref(_cfg(sel)), ctypes.byref(h))
    assert rc == 4 and h.value is None
    assert b"create" in sel.LIB.litevlm_select_last_error(None)


def test_keep_offsets_match_the_oracle_keep_count(sel):
    # litevlm_select_keep_offsets is the library's own k_b = floor((double)r * N_b)
    # (Results, "Visual Token Compression"); it must agree with the oracle's
    # litevlm_oracle_keep_count request by request, on the bench sizes, the
    # paper's Table 1 sizes and random ones, for ratios that are not exact in fp32
    import numpy as np
    import oracle
    rng = np.random.Generator(np.random.PCG64(11))
    sizes = [0, 1, 7, 128, 576, 896, 1536, 3072, 3456, 6144, 65536] + list(rng.integers(0, 10000, size=40))
    so = np.zeros(len(sizes) + 1, np.int32)
    so[1:] = np.cumsum(sizes)
    for r in (0.0, 0.1, 0.2, 0.25, 0.3, 1.0 / 3.0, 0.5, 0.7, 0.8, 0.9, 0.999, 1.0):
        off = sel.keep_offsets(so, None, r)
        want = np.concatenate([[0], np.cumsum([oracle.keep_count(int(n), r) for n in sizes])])
        assert np.array_equal(off, want), r
    kk = np.array([min(n, 3) for n in sizes], np.int32)
    off = sel.keep_offsets(so, kk, 0.0)
    assert np.array_equal(off, np.concatenate([[0], np.cumsum(kk)]))
    assert sel.keep_offsets(np.zeros(1, np.int32), None, 0.5).tolist() == [0]


def test_keep_offsets_rejects_bad_arguments_and_leaves_the_output(sel):
    import numpy as np
    so = np.array([0, 10, 30], np.int32)
    out = np.full(3, -7, np.int32)
    L = sel.LIB
    assert L.litevlm_select_keep_offsets(2, so.ctypes.data, None, 1.5, out.ctypes.data) == 1
    assert L.litevlm_select_keep_offsets(2, so.ctypes.data, None, float("nan"), out.ctypes.data) == 1
    bad_k = np.array([3, 21], np.int32)  # 21 > N_1 = 20
    assert L.litevlm_select_keep_offsets(2, so.ctypes.data, bad_k.ctypes.data, 0.0, out.ctypes.data) == 1
    assert b"keep_k[1]" in L.litevlm_select_last_error(None)
    neg = np.array([0, 10, 5], np.int32)
    assert L.litevlm_select_keep_offsets(2, neg.ctypes.data, None, 0.5, out.ctypes.data) == 1
    assert L.litevlm_select_keep_offsets(2, so.ctypes.data, None, 0.5, None) == 1
    assert L.litevlm_select_keep_offsets(-1, so.ctypes.data, None, 0.5, out.ctypes.data) == 1
    assert out.tolist() == [-7, -7, -7]


def test_wait_budget_setter_needs_a_handle(sel):
    assert sel.LIB.litevlm_select_set_wait_budget(None, 100) == 1


def test_debug_flags_setter_needs_a_handle(sel):
    assert sel.LIB.litevlm_select_set_debug_flags(None, 0) == 1
