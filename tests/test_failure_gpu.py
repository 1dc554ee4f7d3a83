"""Failure handling of the library on the GPU, without faulting it: allocation failures
injected on the host (DPTQ_FAULT_ALLOC), scratch growth that must not free memory that
earlier work still uses, and bounded in-kernel waits that run out."""
import os
import subprocess
import sys
import textwrap

import pytest

from paper_2606_12487_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def dp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12487_gb300 import dptq
    dptq.load()
    return dptq


def test_scratch_growth_keeps_buffers_of_captured_graphs(dp):
    """A graph captured with the scratch at one size keeps its buffer addresses; a later
    call that needs more scratch must allocate new buffers and leave the old ones
    allocated (the host-side query checks that), so replaying the graph stays valid."""
    wl = inputs.llama2_7b_decode()
    K, N, B = 2048, 256, 2048
    layer = dp.dptq_pack_weights(torch.from_numpy(inputs.weights(N, K, layer=2)).cuda(), B)
    small = torch.from_numpy(inputs.activations(wl, 8, K)).cuda()
    out_s = torch.empty((8, N), dtype=torch.float16, device="cuda")
    dp.dptq_qlinear(layer, small, 4, out_s)            # sizes the scratch for this call
    torch.cuda.synchronize()
    ref = out_s.clone()
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        dp.dptq_qlinear(layer, small, 4, out_s)
    before = {p for p, _, alive in dp.dptq_scratch_buffers() if alive}
    assert before, "no scratch buffers reported"
    # More tokens than the device's scratch holds (earlier tests in the same process may
    # have grown it): the scratch must grow.
    act_bytes = dp.dptq_scratch_buffers()[0][1]
    M_big = max(40000, act_bytes // (2 * K) + 512)
    big = torch.from_numpy(inputs.activations(wl, M_big, K)).cuda()
    out_b = torch.empty((M_big, N), dtype=torch.float16, device="cuda")
    dp.dptq_qlinear(layer, big, 8, out_b)
    torch.cuda.synchronize()
    after = dp.dptq_scratch_buffers()
    live = {p for p, _, alive in after if alive}
    assert before <= live, "a buffer captured by the graph was freed by scratch growth"
    assert len(after) > len(before), "the large call did not grow the scratch"
    out_s.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(out_s.view(torch.int16), ref.view(torch.int16))
    dp.dptq_last_device_error()
    layer.close()


def _child(code, fail_at):
    env = dict(os.environ, DPTQ_FAULT_ALLOC=str(fail_at))
    r = subprocess.run([sys.executable, "-c", textwrap.dedent(code)], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    return r.stdout


CHILD = """
import torch
from paper_2606_12487_gb300 import dptq, inputs
dptq.load()
W = torch.from_numpy(inputs.weights(256, 1024)).cuda()
x = torch.from_numpy(inputs.activations(inputs.llama2_7b_decode(), 4, 1024)).cuda()
out = torch.empty((4, 256), dtype=torch.float16, device="cuda")
def attempt(fn):
    try:
        fn()
        return "ok"
    except dptq.DptqError as e:
        return "oom" if e.status == 4 else f"status{e.status}"
res = []
layer = None
def pack():
    global layer
    layer = dptq.dptq_pack_weights(W, 1024)
res.append(attempt(pack))
if layer is None:
    res.append(attempt(pack))
res.append(attempt(lambda: dptq.dptq_qlinear(layer, x, 4, out)))
if res[-1] != "ok":
    res.append(attempt(lambda: dptq.dptq_qlinear(layer, x, 4, out)))
torch.cuda.synchronize()
ref = out.clone()
dptq.dptq_qlinear(layer, x, 4, out)
torch.cuda.synchronize()
print(" ".join(res), "same" if torch.equal(out, ref) else "differs")
"""


@pytest.mark.parametrize("fail_at,expect", [(1, "oom ok ok same"), (3, "ok oom ok same"), (5, "ok oom ok same"),
                                            (6, "ok oom ok same")])
def test_injected_allocation_failure_reports_oom(fail_at, expect):
    """The n-th device allocation fails (host-side injection, no real exhaustion): the
    failing call returns DPTQ_ERR_OOM and leaves nothing half-built, and the same call
    made again succeeds.  Allocations: 1-2 the handle's packed weights and scales, 3-5
    the per-device split-tile sums, counters and error word, 6-7 the activation planes
    and token scales."""
    out = _child(CHILD, fail_at).strip().splitlines()[-1]
    assert out == expect, out


TIMEOUT_CHILD = """
import torch
from paper_2606_12487_gb300 import dptq, inputs
lib = dptq.load()
M, K, N = 32, 4096, 4096
W = torch.from_numpy(inputs.weights(N, K, layer=1)).cuda()
x = torch.from_numpy(inputs.activations(inputs.llama2_7b_decode(), M, K)).cuda()
layer = dptq.dptq_pack_weights(W, 4096)
ref = torch.empty((M, N), dtype=torch.float16, device="cuda")
dptq.dptq_qlinear_quantize(layer, x, 4)
dptq.dptq_qlinear_gemm(layer, M, 4, ref)     # two launches: untouched by the hook
torch.cuda.synchronize()
assert lib.dptq_last_device_error(None) == 0
out = torch.zeros_like(ref)
dptq.dptq_qlinear(layer, x, 4, out)          # first fused launch: waits for a row that never comes
torch.cuda.synchronize()
st1 = lib.dptq_last_device_error(None)
msg = lib.dptq_last_error_message().decode()
dptq.dptq_qlinear(layer, x, 4, out)          # the next launch runs normally
torch.cuda.synchronize()
st2 = lib.dptq_last_device_error(None)
same = torch.equal(out.view(torch.int16), ref.view(torch.int16))
print(st1, st2, "same" if same else "differs", "|", msg)
"""


def test_bounded_wait_times_out_and_recovers():
    """A fused launch is made to wait for one more published token row than its CTAs
    publish (host-side test hook), with the wait bound shortened to 200k cycles (~0.1 ms).
    Every CTA's bounded wait runs out: the kernel records the time-out, drains its own
    copies, frees its tensor memory and returns, and dptq_last_device_error reports
    DPTQ_ERR_TIMEOUT and clears the scratch.  The next launch is then bit-identical to
    the two-launch path.  No GPU fault is involved: the wait ends by its bound."""
    env = dict(os.environ, DPTQ_WAIT_CYCLES="200000", DPTQ_TEST_ROWS_SHORTFALL="1")
    r = subprocess.run([sys.executable, "-c", textwrap.dedent(TIMEOUT_CHILD)], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    line = r.stdout.strip().splitlines()[-1]
    assert line.startswith("5 0 same"), line
    assert "timed out" in line


DEBUG_CHILD = """
import hashlib
import torch
from paper_2606_12487_gb300 import dptq, inputs
lib = dptq.load()
dptq.dptq_reserve(192, 11008, 0)
wl = inputs.llama2_7b_decode()
h = hashlib.sha256()
# fused: slices of 1024 (four parts), slices of 2048 (two parts), whole blocks; the two
# launches at M = 5 and N = 384; a 192-token prefill tile at A4 and A8
for M, N, K, B in [(32, 22016, 4096, 4096), (64, 4096, 4096, 4096), (32, 4096, 11008, 256), (5, 384, 11008, 256),
                   (192, 1024, 4096, 2048)]:
    W = torch.from_numpy(inputs.weights(N, K, layer=3, proj=1)).cuda()
    layer = dptq.dptq_pack_weights(W, B)
    x = torch.from_numpy(inputs.activations(wl, M, K)).cuda()
    for bits in (4, 8):
        out = torch.empty((M, N), dtype=torch.float16, device="cuda")
        dptq.dptq_qlinear(layer, x, bits, out)
        torch.cuda.synchronize()
        h.update(out.cpu().numpy().tobytes())
    layer.close()
print(dptq.lib_path().split("/")[-2], lib.dptq_last_device_error(None), h.hexdigest())
"""


def test_debug_build_checks_pass_and_match_release():
    """The DPTQ_DEBUG library checks the index arithmetic of the kernels' global accesses
    (producers' tile copies, split-tile slots, the fused row parts' loads, stores and
    maximum slots) and records the first failing check in the error word instead of
    making the access.  On the fused, split and prefill paths no check fails, and the
    outputs are the bits of the release library's."""
    res = {}
    for flag in ("0", "1"):
        env = dict(os.environ, DPTQ_DEBUG=flag)
        r = subprocess.run([sys.executable, "-c", textwrap.dedent(DEBUG_CHILD)], cwd=ROOT, env=env,
                           capture_output=True, text=True, timeout=900)
        assert r.returncode == 0, r.stdout + r.stderr
        res[flag] = r.stdout.strip().splitlines()[-1].split()
    assert res["1"][0] == "_build_debug" and res["0"][0] == "_build"
    assert res["1"][1] == "0" and res["0"][1] == "0"
    assert res["1"][2] == res["0"][2]
