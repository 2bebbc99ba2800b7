"""C-ABI checks that need no GPU: the library builds, loads, exports every
entry point declared in include/zo.h, and rejects bad arguments on the host
before touching CUDA."""
import ctypes
import os
import re

import pytest

from paper_2609_38095_gb300 import build as zo_build
from paper_2609_38095_gb300 import zo

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    zo_build.build()
    return zo._lib()


def header_functions():
    src = open(os.path.join(ROOT, "include", "zo.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(zo_[a-z0-9_]+)\s*\(", src)))


def test_exports_every_declared_symbol(L):
    names = header_functions()
    assert len(names) >= 12
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(zo.EXPORTS)


def test_version_and_strings(L):
    assert zo.version() == 10400
    for s in (0, -1, -2, -3, -4, -5, -6, -7):
        assert zo.status_string(s).startswith("ZO_")
    assert "unknown" in zo.status_string(99)
    assert L.zo_last_cuda_error() == b""


def tensors(*specs, packing=0):
    arr = (zo.zo_tensor * len(specs))()
    for i, (ptr, numel, dtype) in enumerate(specs):
        arr[i].ptr, arr[i].numel, arr[i].dtype, arr[i].packing = ptr, numel, dtype, packing
    return arr


FAKE = 0x7F0000000000  # never dereferenced: validation rejects first


def test_perturb_validation(L):
    ok = tensors((FAKE, 16, 1))
    assert L.zo_perturb(ok, -1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_perturb(None, 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_perturb(tensors((FAKE, 16, 3)), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_DTYPE
    assert L.zo_perturb(tensors((FAKE + 1, 16, 1)), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ALIGN
    assert L.zo_perturb(tensors((FAKE + 2, 16, 0)), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ALIGN
    assert L.zo_perturb(tensors((0, 16, 1)), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_perturb(tensors((FAKE, -1, 1)), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_perturb(ok, 1, 1, 0, float("nan"), None) == zo.ZO_ERR_ARG
    assert L.zo_perturb(ok, 1, 1, 0, float("inf"), None) == zo.ZO_ERR_ARG
    for bad in (2, 3, -1, 16):
        assert L.zo_perturb(tensors((FAKE, 16, 1), packing=bad), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    mixed = tensors((FAKE, 16, 1), (FAKE + 64, 16, 1), packing=8)
    mixed[1].packing = 1                     # every tensor of a list names the same packing
    assert L.zo_perturb(mixed, 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    mixed[1].packing = 0
    assert L.zo_perturb(mixed, 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_perturb(None, 0, 1, 0, 1e-3, None) == zo.ZO_OK  # empty list: nothing to do


def test_perturb_pair_validation(L):
    th = tensors((FAKE, 16, 1), (FAKE + 64, 40, 2))
    pl = tensors((FAKE + 4096, 16, 1), (FAKE + 8192, 40, 2))
    mi = tensors((FAKE + 16384, 16, 1), (FAKE + 32768, 40, 2))
    f = L.zo_perturb_pair
    assert f(th, pl, mi, -1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert f(th, None, mi, 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert f(th, pl, mi, 2, 1, 0, float("nan"), None) == zo.ZO_ERR_ARG
    assert f(th, tensors((FAKE + 4096, 16, 1), (FAKE + 8192, 41, 2)), mi, 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert f(th, pl, tensors((FAKE + 16384, 16, 1), (FAKE + 32768, 40, 1)), 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert f(th, pl, tensors((FAKE + 4096, 16, 1), (FAKE + 32768, 40, 2)), 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert f(th, pl, tensors((FAKE + 16385, 16, 1), (FAKE + 32768, 40, 2)), 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ALIGN
    assert f(th, pl, tensors((FAKE + 16384, 16, 3), (FAKE + 32768, 40, 2)), 2, 1, 0, 1e-3, None) == zo.ZO_ERR_DTYPE
    assert f(None, None, None, 0, 1, 0, 1e-3, None) == zo.ZO_OK
    # plus / minus follow theta's probes: no packing of their own, or theta's
    th8 = tensors((FAKE, 16, 1), (FAKE + 64, 40, 2), packing=8)
    pl1 = tensors((FAKE + 4096, 16, 1), (FAKE + 8192, 40, 2), packing=1)
    assert f(th8, pl1, mi, 2, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert f(th, tensors((FAKE + 4096, 16, 1), (FAKE + 8192, 40, 2), packing=8), mi, 2, 1, 0, 1e-3,
             None) == zo.ZO_ERR_ARG     # theta follows the default (1)


def test_param_list_packing_argument():
    with pytest.raises(ValueError):
        zo.ParamList([], packing=4)


def test_update_validation(L):
    ok = tensors((FAKE, 16, 1))
    c = ctypes.c_void_p(FAKE)
    for fn in (L.zo_update, L.zo_update_sequential):
        assert fn(ok, 1, 1, c, 0, 1e-3, None, None) == zo.ZO_ERR_ARG
        assert fn(ok, 1, 1, c, zo.ZO_MAX_PROBES + 1, 1e-3, None, None) == zo.ZO_ERR_TOO_MANY_PROBES
        assert fn(ok, 1, 1, None, 4, 1e-3, None, None) == zo.ZO_ERR_ARG
        assert fn(ok, 1, 1, c, 4, float("nan"), None, None) == zo.ZO_ERR_ARG
        assert fn(tensors((FAKE, 16, 9)), 1, 1, c, 4, 1e-3, None, None) == zo.ZO_ERR_DTYPE
        assert fn(None, 0, 1, c, 4, 1e-3, None, None) == zo.ZO_OK


def test_precondition_validation(L):
    p = ctypes.c_void_p(FAKE)
    f = L.zo_precondition_ex
    assert f(p, 0, 1e-3, 0.1, 1.0, 0, p, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(p, zo.ZO_MAX_PROBES + 1, 1e-3, 0.1, 1.0, 0, p, None, None, p, None) == zo.ZO_ERR_TOO_MANY_PROBES
    assert f(p, 4, 0.0, 0.1, 1.0, 0, p, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(p, 4, float("inf"), 0.1, 1.0, 0, p, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(p, 4, 1e-3, -0.1, 1.0, 0, p, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(p, 4, 1e-3, 1.5, 1.0, 0, p, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(p, 4, 1e-3, 0.1, 0.0, 0, p, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(None, 4, 1e-3, 0.1, 1.0, 0, p, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(p, 4, 1e-3, 0.1, 1.0, 0, None, None, None, p, None) == zo.ZO_ERR_ARG
    assert f(p, 4, 1e-3, 0.1, 1.0, 0, p, None, None, None, None) == zo.ZO_ERR_ARG
    assert L.zo_precondition(p, 0, 1e-3, p, p, None) == zo.ZO_ERR_ARG
    for bad_flags in (4, 8, -1, 1 << 30):
        assert f(p, 4, 1e-3, 0.1, 1.0, bad_flags, p, None, None, p, None) == zo.ZO_ERR_ARG


def test_probe_view_and_loss_validation(L):
    p = ctypes.c_void_p(FAKE)
    assert L.zo_probe_bytes(1, 0, -1, 4, p, None) == zo.ZO_ERR_ARG
    assert L.zo_probe_bytes(1, 0, 0, -4, p, None) == zo.ZO_ERR_ARG
    assert L.zo_probe_bytes(1, 0, 0, 4, None, None) == zo.ZO_ERR_ARG
    assert L.zo_probe_bytes(1, 0, 0, 0, None, None) == zo.ZO_OK
    assert L.zo_probe_signs(1, 0, 0, -1, p, None) == zo.ZO_ERR_ARG
    assert L.zo_probe_signs(1, 0, 0, 0, None, None) == zo.ZO_OK
    ws = L.zo_quadratic_loss_workspace_size(1 << 20)
    assert ws > 0
    assert L.zo_quadratic_loss(p, p, -1, p, p, ws, None) == zo.ZO_ERR_ARG
    assert L.zo_quadratic_loss(p, p, 16, None, p, ws, None) == zo.ZO_ERR_ARG
    assert L.zo_quadratic_loss(p, p, 16, p, None, ws, None) == zo.ZO_ERR_WORKSPACE
    assert L.zo_quadratic_loss(p, p, 16, p, p, ws - 8, None) == zo.ZO_ERR_WORKSPACE


def test_binding_rejects_cpu_tensors():
    import torch
    with pytest.raises(TypeError):
        zo.ParamList([torch.zeros(4)])


def test_static_loss_validation(L):
    p = ctypes.c_void_p(FAKE)
    f = L.zo_quadratic_loss_static
    assert f(p, p, -1, p, None) == zo.ZO_ERR_ARG
    assert f(p, p, 16, None, None) == zo.ZO_ERR_ARG
    assert f(None, p, 16, p, None) == zo.ZO_ERR_ARG
    assert f(p, p, zo.ZO_QUADRATIC_LOSS_STATIC_MAX_N + 1, p, None) == zo.ZO_ERR_WORKSPACE


def test_perturb_quadratic_loss_validation(L):
    """zo_perturb_quadratic_loss rejects bad arguments on the host, before
    any CUDA call (the pointers here are never dereferenced)."""
    p = ctypes.c_void_p(FAKE)
    f = L.zo_perturb_quadratic_loss
    ws = L.zo_perturb_quadratic_loss_workspace_size(1 << 20)
    assert ws >= 8 and ws % 8 == 0

    def call(n=16, packing=0, nops=1, sa=1e-3, sb=1e-3, out=p, copies=1, stride=1, theta=p, a=p, w=p, wb=ws):
        return f(theta, a, n, 1, packing, nops, 0, sa, 1, sb, out, copies, stride, w, wb, None)

    assert call(n=-1) == zo.ZO_ERR_ARG
    assert call(nops=3) == zo.ZO_ERR_ARG and call(nops=-1) == zo.ZO_ERR_ARG
    assert call(sa=float("nan")) == zo.ZO_ERR_ARG
    assert call(nops=2, sb=float("inf")) == zo.ZO_ERR_ARG
    assert call(copies=0) == zo.ZO_ERR_ARG and call(stride=0) == zo.ZO_ERR_ARG
    assert call(out=None) == zo.ZO_ERR_ARG and call(theta=None) == zo.ZO_ERR_ARG
    assert call(packing=2) == zo.ZO_ERR_ARG
    assert call(theta=ctypes.c_void_p(FAKE + 2)) == zo.ZO_ERR_ALIGN
    assert call(a=ctypes.c_void_p(FAKE + 1)) == zo.ZO_ERR_ALIGN
    assert call(w=None) == zo.ZO_ERR_WORKSPACE and call(wb=ws - 8) == zo.ZO_ERR_WORKSPACE
    assert call(w=ctypes.c_void_p(FAKE + 4)) == zo.ZO_ERR_ALIGN


def test_packing_switch(L):
    assert zo.get_packing() == 1
    assert L.zo_set_packing(3) == zo.ZO_ERR_ARG
    assert L.zo_set_packing(0) == zo.ZO_ERR_ARG
    assert zo.get_packing() == 1
    with zo.packing(8):
        assert zo.get_packing() == 8
    assert zo.get_packing() == 1


def test_perturb2_and_update_ex_validation(L):
    ok = tensors((FAKE, 16, 1))
    c = ctypes.c_void_p(FAKE)
    assert L.zo_perturb2(ok, 1, 1, 0, 1e-3, 1, float("nan"), None) == zo.ZO_ERR_ARG
    assert L.zo_perturb2(ok, 1, 1, 0, float("inf"), 1, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_perturb2(tensors((FAKE + 1, 16, 1)), 1, 1, 0, 1e-3, 1, 1e-3, None) == zo.ZO_ERR_ALIGN
    assert L.zo_perturb2(None, 0, 1, 0, 1e-3, 1, 1e-3, None) == zo.ZO_OK
    assert L.zo_update_ex(ok, 1, 1, c, 4, 1e-3, None, 1, 3, float("nan"), None) == zo.ZO_ERR_ARG
    assert L.zo_update_ex(ok, 1, 1, c, 0, 1e-3, None, 1, 3, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_update_ex(None, 0, 1, c, 4, 1e-3, None, 1, 3, 1e-3, None) == zo.ZO_OK


def test_tensor_block_limit(L):
    """One tensor may span fewer than 2^31 16-element blocks (a launch's
    32-bit block offsets); larger tensors are rejected on the host."""
    big = (1 << 31) * 16
    assert L.zo_perturb(tensors((FAKE, big, 1)), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG
    assert L.zo_perturb(tensors((FAKE, big - 16 + 1, 1)), 1, 1, 0, 1e-3, None) == zo.ZO_ERR_ARG


def test_header_is_plain_c_and_links_from_c(tmp_path, L):
    """include/zo.h compiles as C99 with warnings as errors, and a C program
    links against libzo.so and calls it (host-only entry points: no GPU)."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    src = tmp_path / "use_zo.c"
    src.write_text(
        "#include <stdio.h>\n#include <string.h>\n#include \"zo.h\"\n"
        "int main(void) {\n"
        "  zo_tensor t = {0, 0, ZO_BF16, 0};\n"
        "  if (zo_version() != 10400) return 1;\n"
        "  if (strncmp(zo_status_string(ZO_ERR_ARG), \"ZO_ERR_ARG\", 10) != 0) return 2;\n"
        "  if (zo_perturb(&t, -1, 1, 0, 1e-3f, NULL) != ZO_ERR_ARG) return 3;\n"
        "  if (zo_set_packing(3) != ZO_ERR_ARG) return 4;\n"
        "  if (zo_quadratic_loss_workspace_size(1 << 20) <= 0) return 5;\n"
        "  puts(\"ok\");\n  return 0;\n}\n")
    lib = zo.LIB_PATH
    exe = tmp_path / "use_zo"
    inc = os.path.join(ROOT, "include")
    cmd = [gcc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-I", inc, str(src), "-o", str(exe),
           "-L", os.path.dirname(lib), "-l:" + os.path.basename(lib), "-Wl,-rpath," + os.path.dirname(lib)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", (r.returncode, r.stdout, r.stderr)

