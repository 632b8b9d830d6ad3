"""CPU-only checks of the C ABI library: it builds for sm_103a, loads without a GPU, exports every
function declared in include/stepkv.h, and rejects bad arguments on the host before touching CUDA."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "stepkv.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_22158_gb300 import binding, build
    build.build_library()
    return binding.load_library()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"\b(stepkv_[a-z_]+)\s*\(", src)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("stepkv_score", "stepkv_select", "stepkv_compact", "stepkv_compress"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2609_22158_gb300 import binding
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in binding.SIGNATURES, f"binding lacks a signature for {name}"


def test_default_params_are_table_h(lib):
    from paper_2609_22158_gb300 import binding
    p = binding.default_params()
    assert abs(p.lam - 0.3) < 1e-7 and abs(p.w_r - 0.85) < 1e-7 and abs(p.w_c - 0.15) < 1e-7
    assert p.r_min == -1.0 and p.r_max == 2.0 and p.s_max == 8.0
    assert p.eta == 1.5 and abs(p.alpha - 0.2) < 1e-7 and abs(p.beta - 0.8) < 1e-7 and p.sal_norm == 0
    assert p.sal_pool == 1 and p.sal_pool_mode == binding.POOL_MAX  # no pooling by default


def test_status_strings(lib):
    for code in range(7):
        assert lib.stepkv_status_string(code)
    assert lib.stepkv_status_string(99) == b"unknown status"
    assert lib.stepkv_version() >= 1000


def test_workspace_sizes(lib):
    assert lib.stepkv_score_workspace_size(3, 8, 32, 32768, 64) > 0
    assert lib.stepkv_score_workspace_size(0, 8, 32, 32768, 64) == 0
    assert lib.stepkv_select_workspace_size(24, 32768, 40) > 0
    assert lib.stepkv_select_workspace_size(24, 32768, 0) == 0


def test_score_rejects_bad_arguments_on_host(lib):
    from paper_2609_22158_gb300.binding import STEPKV_EINVAL, STEPKV_EUNSUPPORTED
    arr = (ctypes.c_void_p * 1)(256)
    p = ctypes.cast(arr, ctypes.c_void_p)
    ws = ctypes.c_void_p(1 << 20)
    # d not supported
    assert lib.stepkv_score(1, p, 96 * 100, p, 96 * 10, 2, 8, 96, 100, 10, 4096, ws, 1 << 30, None, None) == STEPKV_EUNSUPPORTED
    # Hq not a multiple of Hkv
    assert lib.stepkv_score(1, p, 128 * 100, p, 128 * 10, 3, 8, 128, 100, 10, 4096, ws, 1 << 30, None, None) == STEPKV_EINVAL
    # W > T
    assert lib.stepkv_score(1, p, 128 * 100, p, 128 * 200, 2, 8, 128, 100, 200, 4096, ws, 1 << 30, None, None) == STEPKV_EINVAL
    # too many layers for one call
    assert lib.stepkv_score(9, p, 128 * 100, p, 128 * 10, 2, 8, 128, 100, 10, 4096, ws, 1 << 30, None, None) == STEPKV_EUNSUPPORTED
    # head stride smaller than T*d
    assert lib.stepkv_score(1, p, 128 * 99, p, 128 * 10, 2, 8, 128, 100, 10, 4096, ws, 1 << 30, None, None) == STEPKV_EINVAL


def test_score_lse_rejects_bad_statistics_on_host(lib):
    """stepkv_score_lse checks the per-layer row log-sum-exp pointers (present, 4-byte aligned) on the host,
    after the arguments it shares with stepkv_score, before anything is enqueued."""
    from paper_2609_22158_gb300.binding import STEPKV_EINVAL, STEPKV_EUNSUPPORTED
    kq = (ctypes.c_void_p * 2)(256, 512)
    p = ctypes.cast(kq, ctypes.c_void_p)
    ws = ctypes.c_void_p(1 << 20)
    sal = ctypes.c_void_p(4096)
    call = lambda lse, n_layers=2, sal_=sal: lib.stepkv_score_lse(n_layers, p, 128 * 100, p, 128 * 10, lse, 2, 8, 128,
                                                                   100, 10, sal_, ws, 1 << 30, None, None)
    assert call(None) == STEPKV_EINVAL                                               # no statistics at all
    assert call(ctypes.cast((ctypes.c_void_p * 2)(1024, None), ctypes.c_void_p)) == STEPKV_EINVAL   # layer 1 missing
    assert call(ctypes.cast((ctypes.c_void_p * 2)(1024, 1026), ctypes.c_void_p)) == STEPKV_EINVAL   # misaligned
    good = ctypes.cast((ctypes.c_void_p * 2)(1024, 2048), ctypes.c_void_p)
    assert call(good, sal_=None) == STEPKV_EINVAL                                    # no output
    assert call(good, n_layers=9) == STEPKV_EUNSUPPORTED                             # the shared checks come first


def test_select_rejects_bad_arguments_on_host(lib):
    from paper_2609_22158_gb300 import binding as B
    steps = B.CSteps(0, 256, 256, 256, None, 256, None)
    params = B.Params().c()
    bud = B.budget_ratio(1, 10)
    out = B.CSelOut(256, 10, 256, None, None, None, None, None, None, None, None)
    args = lambda s, pr, b, o: lib.stepkv_select(256, 1, 100, 256, 256, ctypes.byref(s), ctypes.byref(pr),
                                                 ctypes.byref(b), ctypes.byref(o), 256, 1 << 20, None, None)
    assert args(steps, params, bud, out) == B.STEPKV_EINVAL          # n_steps = 0
    steps.n_steps = 4
    bad = B.budget_ratio(1, 0)
    assert args(steps, params, bad, out) == B.STEPKV_EINVAL          # zero denominator
    bad_norm = B.Params(sal_norm=7).c()
    assert args(steps, bad_norm, bud, out) == B.STEPKV_EINVAL
    for pool, mode in ((0, B.POOL_MAX), (4, B.POOL_MAX), (65, B.POOL_MAX), (3, 2)):  # even, too wide, bad mode
        assert args(steps, B.Params(sal_pool=pool, sal_pool_mode=mode).c(), bud, out) == B.STEPKV_EINVAL
    out.kept_idx = None
    assert args(steps, params, bud, out) == B.STEPKV_EINVAL


def test_compact_rejects_bad_arguments_on_host(lib):
    from paper_2609_22158_gb300 import binding as B
    a = (ctypes.c_void_p * 1)(256)
    same = ctypes.cast(a, ctypes.c_void_p)
    other = ctypes.cast((ctypes.c_void_p * 1)(512), ctypes.c_void_p)
    # in-place compaction is refused
    assert lib.stepkv_compact(1, same, None, 128 * 100, 2, 128, 100, 256, 256, 50, same, None, 128 * 50,
                              None, None, None, None, None, None) == B.STEPKV_EUNSUPPORTED
    # misaligned row size (d*2 not a multiple of 16)
    assert lib.stepkv_compact(1, same, None, 100 * 4, 2, 4, 100, 256, 256, 50, other, None, 4 * 50,
                              None, None, None, None, None, None) == B.STEPKV_EINVAL
    # output head stride too small for kept_cap
    assert lib.stepkv_compact(1, same, None, 128 * 100, 2, 128, 100, 256, 256, 50, other, None, 128 * 49,
                              None, None, None, None, None, None) == B.STEPKV_EINVAL


def test_decode_rejects_bad_arguments_on_host(lib):
    from paper_2609_22158_gb300 import binding as B
    p = ctypes.cast((ctypes.c_void_p * 1)(256), ctypes.c_void_p)
    ws = ctypes.c_void_p(1 << 20)
    call = lambda Hkv, Hq, d, stride, n, cap, w=ws: lib.stepkv_decode(1, p, p, p, stride, Hkv, Hq, d, None, n, cap,
                                                                       p, w, 1 << 30, None, None)
    assert call(2, 8, 96, 96 * 100, 50, 100) == B.STEPKV_EUNSUPPORTED    # d
    assert call(2, 6, 128, 128 * 100, 50, 100) == B.STEPKV_EUNSUPPORTED   # G = 3
    assert call(3, 8, 128, 128 * 100, 50, 100) == B.STEPKV_EINVAL         # Hq % Hkv
    assert call(2, 8, 128, 128 * 99, 50, 100) == B.STEPKV_EINVAL          # head stride below capacity
    assert call(2, 8, 128, 128 * 100, 101, 100) == B.STEPKV_EINVAL        # host n above capacity
    assert call(2, 8, 128, 128 * 100, 0, 100) == B.STEPKV_EINVAL          # no keys
    assert call(2, 8, 128, 128 * 100, 50, 100, ctypes.c_void_p(1 << 20 | 8)) == B.STEPKV_EINVAL  # ws alignment
    assert lib.stepkv_decode_workspace_size(32, 8, 32, 128, 8272) > 0
    assert lib.stepkv_decode_workspace_size(32, 8, 32, 96, 8272) == 0


def test_binding_fails_loudly_without_library(tmp_path):
    from paper_2609_22158_gb300 import binding
    with pytest.raises(binding.StepKVError):
        binding.load_library(str(tmp_path / "missing.so"))


def test_ctypes_structs_mirror_the_header(tmp_path):
    """The binding's ctypes structs have the size and field offsets of the C structs in include/stepkv.h
    (compiled here with the system C compiler), so a struct passed through the ABI is read as written."""
    import shutil
    import subprocess
    from paper_2609_22158_gb300 import binding as B
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    mirrors = {"stepkv_params_t": B.CParams, "stepkv_budget_t": B.CBudget, "stepkv_steps_t": B.CSteps,
               "stepkv_select_out_t": B.CSelOut, "stepkv_problem_t": B.CProblem}
    c_names = {"lambda_": "lambda"}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "stepkv.h"', 'int main(void) {']
    for cname, py in mirrors.items():
        lines.append(f'  printf("{cname} size %zu\\n", sizeof({cname}));')
        for f, _ in py._fields_:
            lines.append(f'  printf("{cname} {f} %zu\\n", offsetof({cname}, {c_names.get(f, f)}));')
    lines += ['  return 0;', '}']
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run([cc, "-std=c99", "-I", inc, str(src), "-o", str(exe)], check=True)
    got = {}
    for ln in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines():
        name, field, val = ln.split()
        got[(name, field)] = int(val)
    for cname, py in mirrors.items():
        assert got[(cname, "size")] == ctypes.sizeof(py), cname
        for f, _ in py._fields_:
            assert got[(cname, f)] == getattr(py, f).offset, (cname, f)


def _build_c_program(tmp_path):
    """tests/c/compress_from_c.c compiled with the system C compiler against include/stepkv.h and the
    in-tree library (plain C: no Python, no PyTorch on the path)."""
    import shutil
    import subprocess
    from paper_2609_22158_gb300 import build
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lib_path = build.build_library()
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    exe = tmp_path / "compress_from_c"
    cmd = [cc, "-std=c99", "-O1", "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"),
           os.path.join(ROOT, "tests", "c", "compress_from_c.c"), "-o", str(exe), lib_path,
           "-Wl,-rpath," + os.path.dirname(lib_path), "-L" + os.path.join(cuda, "lib64"), "-lcudart",
           "-Wl,-rpath," + os.path.join(cuda, "lib64")]
    subprocess.run(cmd, check=True)
    return exe


def test_c_program_uses_the_abi(tmp_path):
    import subprocess
    exe = _build_c_program(tmp_path)
    out = subprocess.run([str(exe), "host"], check=True, capture_output=True, text=True).stdout.split("\n")
    fields = dict((ln.split(" ", 1)[0], ln.split(" ", 1)[1]) for ln in out if ln)
    assert [float(x) for x in fields["params"].split()] == pytest.approx(
        [0.3, 0.85, 0.15, -1.0, 2.0, 8.0, 1.5, 0.2, 0.8, 0.0], abs=1e-6)
    from paper_2609_22158_gb300 import binding
    assert fields["status"] == binding.load_library().stepkv_status_string(1).decode()
    assert int(fields["compress_null"]) == 1  # STEPKV_EINVAL before anything is enqueued
    assert int(fields["workspace_empty"]) == 0
