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
