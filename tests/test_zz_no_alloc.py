"""unisvq_linear_noalloc: the tcgen05 decode path with its fold workspace in the
library's static device array, against unisvq_linear and the fp64 oracle.

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


@pytest.mark.parametrize("N,K,d", [(520, 1000, 2), (256, 512, 4), (4096, 4096, 2), (130, 4096, 1)])
def test_noalloc_matches_linear_on_two_calls(N, K, d):
    codes, A, B = synth.layer_inputs(9, 90, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    stream = torch.cuda.current_stream().cuda_stream
    for M in (1, 7, 16, 17):
        xb = synth.activations(9, 90, 100 * N + M, M, K)
        x = to_dev(xb)
        y_api = layer.forward(x)
        y1 = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
        y2 = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
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


def test_noalloc_rejects_what_does_not_fit_and_bad_arguments():
    N, K = 128, 43776   # Kp = 43776 > 43648: the fold needs more than the static array
    codes = np.zeros((N, K), dtype=np.uint8)
    A = np.eye(2, dtype=np.float16)
    B = np.zeros(2, dtype=np.float16)
    layer = binding.UniSVQLinear(codes, A, B)
    x = torch.zeros((1, K), dtype=torch.bfloat16, device="cuda")
    y = torch.zeros((1, N), dtype=torch.bfloat16, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), 1, stream) == binding.ERR_UNSUPPORTED
    assert layer.forward_noalloc_ptr(x.data_ptr() + 2, y.data_ptr(), 1, stream) == binding.ERR_INVALID_ARG
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), -1, stream) == binding.ERR_INVALID_ARG
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), 0, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    layer.close()
