"""3-bit codes (z in {0..7}, Sec. 5.2) against the fp64 oracle: dequantised
weights bit-exact, layer outputs within the tolerance, integer cases bit-exact,
d in {1, 2, 4}, ragged shapes, token chunking, grouped calls and dispatch, on
the GEMV, the tcgen05 decode path (codes z as e4m3 bytes with the high bit
from the bit plane) and the prefill GEMM."""
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


def run(layer, xbits, kernel=binding.KERNEL_AUTO):
    y = layer.forward(to_dev(xbits), kernel=kernel)
    st = binding.sync_status()
    assert st == binding.OK, binding.status_string(st)
    return y.float().cpu().numpy().astype(np.float64)


def make(N, K, d, seed):
    codes, A, B = synth.layer_inputs_bits(seed, 60, N, K, N, K, d, 3)
    return codes, A, B, binding.UniSVQLinear(codes, A, B, bits=3)


@pytest.mark.parametrize("d", [1, 2, 4])
@pytest.mark.parametrize("N,K", [(200, 520), (128, 128), (300, 1024)])
def test_3bit_dequant_bit_exact(d, N, K):
    codes, A, B, layer = make(N, K, d, 1)
    W = layer.dequant_debug()
    assert binding.sync_status() == binding.OK
    assert np.array_equal(W.cpu().numpy(), oracle.dequant_f32(codes, A, B))
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4])
@pytest.mark.parametrize("N,K", [(256, 1024), (520, 1000), (130, 4096), (1024, 8192)])
def test_3bit_parity(d, N, K):
    if K % d:
        pytest.skip("K must be a multiple of d")
    codes, A, B, layer = make(N, K, d, 2)
    Ms = (1, 3, 8, 16, 17, 40)
    xall = synth.activations(2, 60, 100 * d, sum(Ms), K)
    yr, S = oracle.linear(xall, codes, A, B)
    o = 0
    for M in Ms:
        res = oracle.compare(run(layer, xall[o:o + M]), yr[o:o + M], S[o:o + M])
        assert res["ok"], (M, res)
        o += M
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4])
def test_3bit_integer_case_bit_exact(d):
    g = np.random.default_rng(40 + d)
    N, K = 256, 512
    codes = g.integers(0, 8, size=(N, K), dtype=np.uint8)
    A = (np.eye(d) - np.eye(d, k=1)).astype(np.float16)
    B = g.integers(-3, 4, size=d).astype(np.float16)
    layer = binding.UniSVQLinear(codes, A, B, bits=3)
    for M in (1, 7, 33):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.03)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear(xb, codes, A, B)
        assert np.abs(yr).max() <= 256
        yg = run(layer, xb)
        assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


def test_3bit_dispatch_groups_and_entry_points():
    N, K, d = 512, 1024, 2
    codes, A, B, layer = make(N, K, d, 3)
    for M in (1, 16, 64):
        assert layer.query(M)["kernel"] == binding.KERNEL_GEMV
    assert layer.query(65)["kernel"] == binding.KERNEL_PREFILL
    assert layer.query(1)["algo_bytes"] == N * K * 3 // 8 + (d * d + d) * 2 + 2 * K + 2 * N
    xb = synth.activations(3, 60, 0, 5, K)
    x = to_dev(xb)
    stream = torch.cuda.current_stream().cuda_stream
    y = torch.zeros((5, N), dtype=torch.bfloat16, device="cuda")
    for kern in (binding.KERNEL_GEMV_ROWS, binding.KERNEL_GROUPED):
        assert layer.forward_ptr(x.data_ptr(), y.data_ptr(), 5, stream, kern) == binding.ERR_UNSUPPORTED
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), 5, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    yr, S = oracle.linear(xb, codes, A, B)
    assert oracle.compare(y.float().cpu().numpy().astype(np.float64), yr, S)["ok"]
    # a group of 3-bit layers (one launch) and a mixed 2-bit/3-bit group (layer by layer)
    c2, A2, B2, l2 = make(256, K, d, 4)
    pc, pA, pB = synth.layer_inputs(3, 60, 0, 0, 384, K, d)
    plain = binding.UniSVQLinear(pc, pA, pB)
    for group, refs in (([layer, l2], [(codes, A, B), (c2, A2, B2)]), ([layer, plain], [(codes, A, B), (pc, pA, pB)])):
        ys = binding.linear_group(group, x)
        assert binding.sync_status() == binding.OK
        for (c, a, b), yy in zip(refs, ys):
            r, S2 = oracle.linear(xb, c, a, b)
            assert oracle.compare(yy.float().cpu().numpy().astype(np.float64), r, S2)["ok"]
    cl = layer.clone()
    assert np.array_equal(run(cl, xb), run(layer, xb))
    for h in (layer, l2, plain, cl):
        h.close()


@pytest.mark.parametrize("N,K", [(4096, 11008), (11008, 4096)])
def test_3bit_full_size_all_rows(N, K):
    codes, A, B, layer = make(N, K, 2, 5)
    for M in (1, 16):
        xb = synth.activations(5, 60, M, M, K)
        y = run(layer, xb)
        yr, S = oracle.linear(xb, codes, A, B)
        assert oracle.compare(y, yr, S)["ok"]
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4])
@pytest.mark.parametrize("N,K", [(256, 1024), (520, 1000), (384, 4096)])
def test_3bit_prefill_parity(d, N, K):
    """3-bit layers run the tcgen05 prefill GEMM above 64 tokens (64-pair
    codeword table for d <= 2, two 64-row pair tables for d = 4, high bits
    from the bit plane)."""
    codes, A, B, layer = make(N, K, d, 6)
    Ms = (65, 300)
    xall = synth.activations(6, 60, N + d, sum(Ms), K)
    yr, S = oracle.linear(xall, codes, A, B)
    o = 0
    for M in Ms:
        assert layer.query(M)["kernel"] == binding.KERNEL_PREFILL
        res = oracle.compare(run(layer, xall[o:o + M]), yr[o:o + M], S[o:o + M])
        assert res["ok"], (M, res)
        o += M
    res = oracle.compare(run(layer, xall[:7], binding.KERNEL_PREFILL), yr[:7], S[:7])
    assert res["ok"], res
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4])
def test_3bit_prefill_integer_case_bit_exact(d):
    g = np.random.default_rng(50 + d)
    N, K = 256, 512
    codes = g.integers(0, 8, size=(N, K), dtype=np.uint8)
    A = (np.eye(d) - np.eye(d, k=1)).astype(np.float16)
    B = g.integers(-3, 4, size=d).astype(np.float16)
    layer = binding.UniSVQLinear(codes, A, B, bits=3)
    x = g.integers(-1, 2, size=(130, K)).astype(np.float32) * (g.random((130, K)) < 0.03)
    xb = synth.f32_to_bf16_bits(x)
    yr, _ = oracle.linear(xb, codes, A, B)
    assert np.abs(yr).max() <= 256
    assert np.array_equal(run(layer, xb), yr)
    layer.close()


def test_3bit_d4_dispatch():
    """d = 4: the GEMV up to 64 tokens, the prefill GEMM above (pair tables)."""
    codes, A, B, layer = make(256, 512, 4, 7)
    assert layer.query(64)["kernel"] == binding.KERNEL_GEMV
    assert layer.query(200)["kernel"] == binding.KERNEL_PREFILL
    xb = synth.activations(7, 60, 4, 100, 512)
    yr, S = oracle.linear(xb, codes, A, B)
    assert oracle.compare(run(layer, xb), yr, S)["ok"]
    assert oracle.compare(run(layer, xb, binding.KERNEL_GEMV), yr, S)["ok"]
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4])
@pytest.mark.parametrize("N,K", [(256, 1024), (520, 1000), (130, 4096), (1024, 8192)])
def test_3bit_tcgen05_decode_parity(d, N, K):
    """The tcgen05 decode path on 3-bit codes: each byte of the tensor-memory
    A operand is the whole code z (z_lo from the code words, z_hi from the
    bit plane), forced at every token count of one and two launch pairs."""
    if K % d:
        pytest.skip("K must be a multiple of d")
    codes, A, B, layer = make(N, K, d, 8)
    Ms = (1, 3, 8, 16, 17, 33, 40)
    xall = synth.activations(8, 60, 100 * d + N, sum(Ms), K)
    yr, S = oracle.linear(xall, codes, A, B)
    o = 0
    for M in Ms:
        res = oracle.compare(run(layer, xall[o:o + M], binding.KERNEL_SKINNY), yr[o:o + M], S[o:o + M])
        assert res["ok"], (M, res)
        o += M
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4])
def test_3bit_tcgen05_decode_integer_case_bit_exact(d):
    g = np.random.default_rng(60 + d)
    N, K = 384, 1024
    codes = g.integers(0, 8, size=(N, K), dtype=np.uint8)
    A = (np.eye(d) - np.eye(d, k=1)).astype(np.float16)
    B = g.integers(-3, 4, size=d).astype(np.float16)
    layer = binding.UniSVQLinear(codes, A, B, bits=3)
    for M in (1, 7, 33):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.03)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear(xb, codes, A, B)
        assert np.abs(yr).max() <= 256
        assert np.array_equal(run(layer, xb, binding.KERNEL_SKINNY), yr)
    layer.close()


def test_3bit_large_layers_dispatch_to_tcgen05_decode():
    """Large 3-bit layers and groups take the tcgen05 decode path up to 64
    tokens, as 2-bit ones do; a group of them runs one launch pair."""
    K = 4096
    made = [synth.layer_inputs_bits(9, 61, i, 0, 4096, K, 2, 3) for i in range(3)]
    layers = [binding.UniSVQLinear(c, A, B, bits=3) for c, A, B in made]
    assert layers[0].query(4)["kernel"] == binding.KERNEL_GEMV          # 2^24 weights
    q = binding.query_group(layers, 4)
    assert q["kernel"] == binding.KERNEL_SKINNY and q["launches"] == 2
    xb = synth.activations(9, 61, 0, 12, K)
    ys = binding.linear_group(layers, to_dev(xb))
    assert binding.sync_status() == binding.OK
    for (c, A, B), y in zip(made, ys):
        yr, S = oracle.linear(xb, c, A, B)
        assert oracle.compare(y.float().cpu().numpy().astype(np.float64), yr, S)["ok"]
    for l in layers:
        l.close()
