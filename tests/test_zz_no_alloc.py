"""unisvq_linear_noalloc: unisvq_linear's kernel choice with the tcgen05
decode pair's fold workspace in the library's static device array, against
unisvq_linear and the fp64 oracle.

Collected last on purpose (file name), and self-contained, so it passes both
after the other GPU tests and alone in a fresh process.
"""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2606_10520_gb300 import binding  # noqa: E402


def to_dev(xbits: np.ndarray):
    return torch.from_numpy(np.ascontiguousarray(xbits).view(np.int16)).view(torch.bfloat16).cuda()


def host(y):
    return y.float().cpu().numpy().astype(np.float64)


def nan_like(M, N):
    return torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")


# (N, K, d): small layers (the GEMV), and layers large enough for the tcgen05
# decode pair at 32 tokens per launch (4096^2, 8192 x 4096 with d = 8) and at
# 16 (Kp = 28672 does not fit 32 tokens' folded activations in the array)
@pytest.mark.parametrize("N,K,d", [(520, 1000, 2), (256, 512, 4), (4096, 4096, 2), (130, 4096, 1),
                                   (8192, 4096, 8), (2304, 28672, 2)])
def test_noalloc_matches_linear_on_two_calls(N, K, d):
    codes, A, B = synth.layer_inputs(9, 90, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    stream = torch.cuda.current_stream().cuda_stream
    for M in (1, 7, 16, 17, 33):
        xb = synth.activations(9, 90, 100 * N + M, M, K)
        x = to_dev(xb)
        y_api = layer.forward(x)
        y1, y2 = nan_like(M, N), nan_like(M, N)
        # two calls in a row on one stream, no synchronisation between them
        assert layer.forward_noalloc_ptr(x.data_ptr(), y1.data_ptr(), M, stream) == binding.OK
        assert layer.forward_noalloc_ptr(x.data_ptr(), y2.data_ptr(), M, stream) == binding.OK
        st = binding.sync_status()
        assert st == binding.OK, binding.status_string(st)
        yr, S = oracle.linear(xb, codes, A, B)
        ya, a1, a2 = host(y_api), host(y1), host(y2)
        tol = 2.0 ** -7 * S + 1e-6
        for yg in (a1, a2):
            assert np.all(np.abs(yg - ya) <= tol), np.abs(yg - ya).max()
            res = oracle.compare(yg, yr, S)
            assert res["ok"], res
        assert np.array_equal(a1, a2)
    layer.close()


def test_noalloc_two_layers_back_to_back_share_the_array():
    """Layer A then layer B (different K and d) on one stream with no
    synchronisation between them: the second call rewrites the array the
    first one used, in stream order, and both outputs are right."""
    la = (8192, 4096, 2)   # both large enough for the tcgen05 decode pair
    lb = (8192, 8192, 4)
    mats = [synth.layer_inputs(9, 95, i, 0, N, K, d) for i, (N, K, d) in enumerate((la, lb))]
    layers = [binding.UniSVQLinear(*m) for m in mats]
    assert all(l.query(8)["kernel"] == binding.KERNEL_SKINNY for l in layers)
    stream = torch.cuda.current_stream().cuda_stream
    M = 8
    xs = [synth.activations(9, 95, i, M, K) for i, (_, K, _) in enumerate((la, lb))]
    xd = [to_dev(x) for x in xs]
    ys = [nan_like(M, N) for N, _, _ in (la, lb)]
    for rep in range(2):
        for l, x, y in zip(layers, xd, ys):
            assert l.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), M, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    for (codes, A, B), xb, y in zip(mats, xs, ys):
        yr, S = oracle.linear(xb, codes, A, B)
        res = oracle.compare(host(y), yr, S)
        assert res["ok"], res
    for l in layers:
        l.close()


def test_noalloc_leaves_free_device_memory_unchanged():
    """After a first call (which looks up the array and loads the module),
    further calls take no device memory: cudaMemGetInfo's free bytes stay put."""
    N, K, d = 8192, 4096, 2
    codes, A, B = synth.layer_inputs(9, 96, 0, 0, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    assert layer.query(16)["kernel"] == binding.KERNEL_SKINNY
    stream = torch.cuda.current_stream().cuda_stream
    x = to_dev(synth.activations(9, 96, 0, 16, K))
    y = torch.empty((16, N), dtype=torch.bfloat16, device="cuda")
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), 16, stream) == binding.OK
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(8):
        assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), 16, stream) == binding.OK
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert binding.sync_status() == binding.OK
    layer.close()


def test_noalloc_bad_arguments():
    N, K = 128, 512
    codes = np.zeros((N, K), dtype=np.uint8)
    layer = binding.UniSVQLinear(codes, np.eye(2, dtype=np.float16), np.zeros(2, dtype=np.float16))
    x = torch.zeros((1, K), dtype=torch.bfloat16, device="cuda")
    y = torch.zeros((1, N), dtype=torch.bfloat16, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    assert layer.forward_noalloc_ptr(x.data_ptr() + 2, y.data_ptr(), 1, stream) == binding.ERR_INVALID_ARG
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), -1, stream) == binding.ERR_INVALID_ARG
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), 0, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    layer.close()
