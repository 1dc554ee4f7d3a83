"""dptq_qlinear_static, the entry point that allocates no device memory, against
dptq_qlinear.

Some callers cannot let the library allocate device memory when they call it: serving
runtimes whose own memory pool has already taken the device's memory, and hosts that
forbid cudaMalloc once they are serving.  dptq_qlinear_static serves them from one fixed
array compiled into the library.  It runs the same two kernels as dptq_qlinear's
two-launch path, which gives the same bits as its one-launch path, so its output must be
bit-identical to dptq_qlinear's.  This file is collected last, so a failure here comes
after every other test has run; it also passes on its own in a fresh process.
"""
import ctypes

import pytest

from paper_2606_12487_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12487_gb300 import dptq
    dptq.load()
    return dptq


def _static_call(dp, layer, x, bits, out):
    """Straight through the C ABI."""
    lib = dp.load()
    st = lib.dptq_qlinear_static(layer.handle, ctypes.c_void_p(x.data_ptr()), x.shape[0], bits,
                                 ctypes.c_void_p(out.data_ptr()),
                                 ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    return st, lib.dptq_last_error_message().decode()


def _device_error(dp):
    """Status of dptq_last_device_error, which also reads the fixed array's error word."""
    return dp.load().dptq_last_device_error(None)


@pytest.mark.parametrize("M,N,K,B,bits", [(32, 4096, 4096, 4096, 4), (1, 4096, 4096, 4096, 8),
                                          (17, 1024, 11008, 256, 4), (32, 12288, 4096, 4096, 8),
                                          (5, 272, 2560, 2048, 8), (32, 512, 2560, 2048, 4)])
def test_static_scratch_matches_qlinear_twice(dp, M, N, K, B, bits):
    wl = inputs.llama2_7b_decode()
    x = torch.from_numpy(inputs.activations(wl, M, K)).cuda()
    W = torch.from_numpy(inputs.weights(N, K, layer=3, proj=1)).cuda()
    layer = dp.dptq_pack_weights(W, B)
    ref = torch.empty((M, N), dtype=torch.float16, device="cuda")
    dp.dptq_qlinear(layer, x, bits, ref)
    for _ in range(2):                     # the shared array must be left clean by each call
        out = torch.full((M, N), float("nan"), dtype=torch.float16, device="cuda")
        st, msg = _static_call(dp, layer, x, bits, out)
        assert st == 0, msg
        torch.cuda.synchronize()
        assert torch.equal(out.view(torch.int16), ref.view(torch.int16)), "static output differs from dptq_qlinear"
        assert _device_error(dp) == 0, "a bounded wait gave up inside the static call"
    layer.close()


def test_static_call_allocates_no_device_memory(dp):
    """After one warm-up call (which looks the array up), a call on a new shape leaves
    the device's free memory unchanged."""
    wl = inputs.llama2_7b_decode()
    layers, xs, outs = [], [], []
    for (M, N, K, B) in [(8, 1024, 4096, 4096), (31, 2048, 2560, 2048)]:
        layers.append(dp.dptq_pack_weights(torch.from_numpy(inputs.weights(N, K, layer=6)).cuda(), B))
        xs.append(torch.from_numpy(inputs.activations(wl, M, K)).cuda())
        outs.append(torch.empty((M, N), dtype=torch.float16, device="cuda"))
    st, msg = _static_call(dp, layers[0], xs[0], 4, outs[0])
    assert st == 0, msg
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for bits in (8, 4):
        st, msg = _static_call(dp, layers[1], xs[1], bits, outs[1])
        assert st == 0, msg
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, f"free device memory changed by {free0 - free1} bytes"
    assert _device_error(dp) == 0
    for layer in layers:
        layer.close()


def test_static_scratch_rejects_shapes_beyond_its_limit(dp):
    W = torch.from_numpy(inputs.weights(128, 4096)).cuda()
    layer = dp.dptq_pack_weights(W, 4096)
    x = torch.zeros((33, 4096), dtype=torch.float16, device="cuda")
    out = torch.empty((33, 128), dtype=torch.float16, device="cuda")
    st, msg = _static_call(dp, layer, x, 4, out)
    assert st == 2 and "32" in msg
    W2 = torch.from_numpy(inputs.weights(128, 16640)).cuda()
    layer2 = dp.dptq_pack_weights(W2, 256)
    x2 = torch.zeros((4, 16640), dtype=torch.float16, device="cuda")
    out2 = torch.empty((4, 128), dtype=torch.float16, device="cuda")
    st, msg = _static_call(dp, layer2, x2, 4, out2)
    assert st == 2 and "16384" in msg
    # a Paley tail block (K = 1024 + 96 = 12 x 8): served by dptq_qlinear, not here
    W3 = torch.from_numpy(inputs.weights(128, 1120)).cuda()
    layer3 = dp.dptq_pack_weights(W3, 1024)
    x3 = torch.zeros((4, 1120), dtype=torch.float16, device="cuda")
    out3 = torch.empty((4, 128), dtype=torch.float16, device="cuda")
    st, msg = _static_call(dp, layer3, x3, 4, out3)
    assert st == 2 and "tail" in msg
    layer.close()
    layer2.close()
    layer3.close()
