"""C-ABI library checks that need no GPU: it builds for sm_103a, loads, exports every
function include/dptq.h declares, and rejects bad arguments before touching CUDA."""
import ctypes
import os
import re
import subprocess
import sys
import textwrap

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_12487_gb300 import dptq
    return dptq.load()


def declared_functions():
    names = []
    for fname in os.listdir(os.path.join(ROOT, "include")):
        if not fname.endswith(".h"):
            continue
        src = open(os.path.join(ROOT, "include", fname)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*(dptq_[a-z0-9_]+)\s*\(", src, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("dptq_pack_weights", "dptq_rotate_quant_act", "dptq_qlinear"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2606_12487_gb300 import dptq
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in dptq.EXPORTS, f"binding lacks {name}"


def test_library_is_built_for_sm103a():
    from paper_2606_12487_gb300 import build
    assert "arch=compute_103a,code=sm_103a" in build.ARCH
    assert os.path.exists(build.LIB)


def test_status_strings(lib):
    assert lib.dptq_status_str(0) == b"ok"
    assert lib.dptq_status_str(5) == b"device wait timed out"


def test_argument_checks_need_no_gpu(lib):
    P = ctypes.c_void_p
    dummy = P(16)
    h = P()
    # bits outside {4, 8}
    assert lib.dptq_rotate_quant_act(dummy, 4, 256, 256, 5, dummy, dummy, None) == 1
    assert b"bits" in lib.dptq_last_error_message()
    # K not a multiple of 32 / bad Hadamard layout / null pointers / sizes
    assert lib.dptq_rotate_quant_act(dummy, 4, 100, 64, 4, dummy, dummy, None) == 2
    # a tail of 96 = 12 x 8 has a Paley factor (11 is prime): the shape checks pass
    assert lib.dptq_rotate_quant_act(dummy, 4, 1536 + 96, 512, 4, dummy, dummy, None) != 2
    # a tail of 736 = 23 x 32 has none of order at most 256 (91, 183 composite; 368 too large)
    assert lib.dptq_rotate_quant_act(dummy, 4, 1024 + 736, 1024, 4, dummy, dummy, None) == 2
    assert b"Paley" in lib.dptq_last_error_message()
    assert lib.dptq_rotate_quant_act(None, 4, 256, 256, 4, dummy, dummy, None) == 1
    assert lib.dptq_rotate_quant_act(dummy, -1, 256, 256, 4, dummy, dummy, None) == 1
    assert lib.dptq_rotate_quant_act(dummy, 0, 256, 256, 4, dummy, dummy, None) == 0   # M == 0: no-op
    assert lib.dptq_pack_weights(None, 16, 256, 256, 1, ctypes.byref(h)) == 1
    assert lib.dptq_pack_weights(dummy, 0, 256, 256, 1, ctypes.byref(h)) == 1
    assert lib.dptq_pack_weights(dummy, 24, 256, 256, 1, ctypes.byref(h)) == 2          # N % 16
    assert lib.dptq_qlinear(None, dummy, 4, 4, dummy, None) == 1
    assert lib.dptq_qlinear(None, dummy, 4, 3, dummy, None) == 1
    assert lib.dptq_get_shape(None, None, None, None) == 1
    lib.dptq_destroy(None)


def test_binding_has_no_cpu_fallback():
    # The binding forwards to the library only; it contains no compute path of its own.
    src = open(os.path.join(ROOT, "paper_2606_12487_gb300", "dptq.py")).read()
    assert "import oracle" not in src and "from oracle" not in src
    for banned in ("numpy.matmul", "torch.matmul", "@ ", "hadamard"):
        assert banned not in src


def test_next_entry_points_check_arguments_without_gpu(lib):
    P = ctypes.c_void_p
    dummy = P(16)
    h = P()
    # randomized Hadamard packing: null signs
    assert lib.dptq_pack_weights_rh(dummy, 16, 256, 256, None, 1, ctypes.byref(h)) == 1
    # misaligned device signs
    assert lib.dptq_rotate_quant_act_rh(dummy, 4, 256, 256, 4, P(17), dummy, dummy, None) == 1
    assert lib.dptq_rotate_act_rh(dummy, 4, 256, 256, P(18), dummy, None) == 1
    # KV4: null pointers, group not a multiple of 128 / not dividing cols, rows == 0
    assert lib.dptq_kv4_quantize(None, 4, 256, 128, dummy, dummy, None) == 1
    assert lib.dptq_kv4_quantize(dummy, 4, 256, 100, dummy, dummy, None) == 2
    assert lib.dptq_kv4_quantize(dummy, 4, 384, 256, dummy, dummy, None) == 2
    assert lib.dptq_kv4_quantize(dummy, 0, 256, 128, dummy, dummy, None) == 0
    # policy: bits, eps, sizes, null pointers, L == 0
    D = ctypes.c_double
    assert lib.dptq_sensitivity_policy(dummy, dummy, 2, 8, 64, 5, D(1e-6), D(0.1), D(20.0), dummy, dummy, dummy, None) == 1
    assert lib.dptq_sensitivity_policy(dummy, dummy, 2, 8, 64, 4, D(-1.0), D(0.1), D(20.0), dummy, dummy, dummy, None) == 1
    assert lib.dptq_sensitivity_policy(dummy, dummy, 2, 8, 63, 4, D(1e-6), D(0.1), D(20.0), dummy, dummy, dummy, None) == 1
    assert lib.dptq_sensitivity_policy(None, dummy, 2, 8, 64, 4, D(1e-6), D(0.1), D(20.0), dummy, dummy, dummy, None) == 1
    assert lib.dptq_sensitivity_policy(dummy, dummy, 0, 8, 64, 4, D(1e-6), D(0.1), D(20.0), dummy, dummy, dummy, None) == 0


def test_nvtx_ranges_need_no_tool():
    """With DPTQ_NVTX=1 every entry point opens and closes an NVTX range named after it;
    with no profiler attached the calls behave as without (argument errors included)."""
    code = textwrap.dedent("""
        import ctypes
        from paper_2606_12487_gb300 import dptq
        lib = dptq.load()
        d = ctypes.c_void_p(16)
        print(lib.dptq_rotate_quant_act(d, 4, 256, 256, 5, d, d, None),
              lib.dptq_rotate_quant_act(d, 4, 100, 64, 4, d, d, None),
              lib.dptq_qlinear(None, d, 4, 4, d, None))
    """)
    env = dict(os.environ, DPTQ_NVTX="1")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.split() == ["1", "2", "1"]
