"""GPU parity of the streaming decode GEMV (UNISVQ_KERNEL_STREAM) against the
fp64 CPU oracle: single layers over d in {1, 2, 4}, ragged shapes, token
counts around the launch size (8), layers whose codes do not fit the shared
ring (refilled stages, several warps per k-group), grouped calls and an
integer-valued case that must be bit-exact.
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

binding.load()
STREAM = binding.KERNEL_STREAM


def to_dev(xbits: np.ndarray):
    return torch.from_numpy(np.ascontiguousarray(xbits).view(np.int16)).view(torch.bfloat16).cuda()


def run(layer, xbits, kernel=STREAM):
    y = layer.forward(to_dev(xbits), kernel=kernel)
    st = binding.sync_status()
    assert st == binding.OK, binding.status_string(st)
    return y.float().cpu().numpy().astype(np.float64)


def check(yg, xbits, codes, A, B):
    yr, S = oracle.linear(xbits, codes, A, B)
    res = oracle.compare(yg, yr, S)
    assert res["ok"], res
    return res


@pytest.mark.parametrize("d", [1, 2, 4])
@pytest.mark.parametrize("N,K", [(256, 1024), (520, 1000), (130, 4096), (1024, 8192), (200, 1002), (48, 132)])
def test_stream_parity(d, N, K):
    if K % d:
        pytest.skip("K % d")
    codes, A, B = synth.layer_inputs(7, 70, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (1, 2, 3, 4, 5, 7, 8, 9, 16, 17):
        xb = synth.activations(7, 70, 1000 * N + M, M, K)
        check(run(layer, xb), xb, codes, A, B)
    layer.close()


@pytest.mark.parametrize("N,K", [(11008, 4096), (4096, 11008), (28672, 1024)])
def test_stream_ring_refill(N, K):
    """Codes that do not fit the shared-memory ring: stages are released and
    refilled, and for 11008 x 4096 (ten units per CTA) two warps share each
    k-group's stages."""
    d = 2
    codes, A, B = synth.layer_inputs(8, 80, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (1, 4, 8):
        xb = synth.activations(8, 80, M, M, K)
        check(run(layer, xb), xb, codes, A, B)
    layer.close()


def test_stream_group_call():
    """q, k, v of different heights in one streaming launch; every output
    meets the bar on its own."""
    K, d = 4096, 2
    shapes = [(4096, K), (1024, K), (1024, K)]
    layers, ins = [], []
    for pi, (N, _) in enumerate(shapes):
        codes, A, B = synth.layer_inputs(9, 90, 0, pi, N, K, d)
        layers.append(binding.UniSVQLinear(codes, A, B))
        ins.append((codes, A, B))
    for M in (1, 3, 8, 11):
        xb = synth.activations(9, 90, M, M, K)
        outs = binding.linear_group(layers, to_dev(xb), kernel=STREAM)
        assert binding.sync_status() == binding.OK
        for (codes, A, B), y in zip(ins, outs):
            check(y.float().cpu().numpy().astype(np.float64), xb, codes, A, B)
    for layer in layers:
        layer.close()


def test_stream_integer_case_bit_exact():
    """Integer A (the printed D4 generator), integer B and small integer x:
    every intermediate is exact, so the output must equal the oracle's."""
    d = 4
    A = np.array([[1, -1, 0, 0], [0, 1, -1, 0], [0, 0, 1, -1], [0, 0, 1, 1]], dtype=np.float16)
    B = np.array([1, -2, 0, 1], dtype=np.float16)
    N, K = 256, 512
    g = np.random.default_rng(12)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (1, 5, 8, 12):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.05)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear(xb, codes, A, B)
        assert np.abs(yr).max() <= 256
        yg = run(layer, xb)
        assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


def test_stream_unsupported_layers():
    """d = 8 and 3-bit layers are not streamed: the forced kernel says so."""
    codes, A, B = synth.layer_inputs(10, 100, 0, 0, 256, 512, 8)
    layer = binding.UniSVQLinear(codes, A, B)
    x = to_dev(synth.activations(10, 100, 0, 1, 512))
    y = torch.empty((1, 256), dtype=torch.bfloat16, device="cuda")
    st = layer.forward_ptr(x.data_ptr(), y.data_ptr(), 1, torch.cuda.current_stream().cuda_stream, STREAM)
    assert st == binding.ERR_UNSUPPORTED
    layer.close()
