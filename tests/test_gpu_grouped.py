"""Per-(row, 128-column group) affine layers (unisvq_pack_grouped) against the
fp64 oracle: dequantised weights bit-exact, layer outputs within the
tolerance, integer cases bit-exact, every vector length, ragged shapes,
token chunking, grouped calls and the entry points that accept the handle."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2606_10520_gb300 import binding  # noqa: E402

GC = 128


def to_dev(xbits: np.ndarray):
    return torch.from_numpy(np.ascontiguousarray(xbits).view(np.int16)).view(torch.bfloat16).cuda()


def dequant(layer):
    W = layer.dequant_debug()
    st = binding.sync_status()
    assert st == binding.OK, binding.status_string(st)
    return W.cpu().numpy()


def run(layer, xbits, kernel=binding.KERNEL_AUTO):
    y = layer.forward(to_dev(xbits), kernel=kernel)
    st = binding.sync_status()
    assert st == binding.OK, binding.status_string(st)
    return y.float().cpu().numpy().astype(np.float64)


def make(N, K, d, seed=0):
    codes, A, B = synth.layer_inputs_grouped(seed, 40, N, K, N, K, d)
    return codes, A, B, binding.UniSVQLinear(codes, A, B, group_cols=GC)


def check(yg, xbits, codes, A, B, rows=None):
    if rows is not None:
        yr, S = oracle.linear_grouped(xbits, codes[rows], A[rows], B[rows], GC)
        yg = yg[:, rows]
    else:
        yr, S = oracle.linear_grouped(xbits, codes, A, B, GC)
    res = oracle.compare(yg, yr, S)
    assert res["ok"], res
    return res


@pytest.mark.parametrize("d", [1, 2, 4, 8])
@pytest.mark.parametrize("N,K", [(200, 520), (128, 128), (300, 1024)])
def test_grouped_dequant_bit_exact(d, N, K):
    codes, A, B, layer = make(N, K, d, seed=1)
    W = dequant(layer)
    ref = oracle.dequant_grouped(codes, A, B, GC).astype(np.float32)
    assert np.array_equal(W, ref)
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4, 8])
@pytest.mark.parametrize("N,K", [(256, 1024), (520, 1000), (130, 4096), (1024, 8192)])
def test_grouped_parity(d, N, K):
    if K % d:
        pytest.skip("K must be a multiple of d")
    codes, A, B, layer = make(N, K, d, seed=2)
    Ms = (1, 3, 8, 16, 17, 40)
    xall = synth.activations(2, 40, 1000 * d, sum(Ms), K)
    yr, S = oracle.linear_grouped(xall, codes, A, B, GC)   # one oracle pass, sliced per call
    o = 0
    for M in Ms:
        res = oracle.compare(run(layer, xall[o:o + M]), yr[o:o + M], S[o:o + M])
        assert res["ok"], (M, res)
        o += M
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_grouped_integer_case_bit_exact(d):
    """Small integer A and B per (row, group), sparse integer x: every step is
    exact, so the output must equal the oracle bit for bit."""
    g = np.random.default_rng(30 + d)
    N, K = 256, 640
    G = K // GC
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    A = g.integers(-2, 3, size=(N, G, d, d)).astype(np.float16)
    B = g.integers(-2, 3, size=(N, G, d)).astype(np.float16)
    layer = binding.UniSVQLinear(codes, A, B, group_cols=GC)
    for M in (1, 5, 32 // d, 33):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.03)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear_grouped(xb, codes, A, B, GC)
        assert np.abs(yr).max() <= 256
        yg = run(layer, xb)
        assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


def test_grouped_maps_really_differ_per_row_and_group():
    """Scale one row's map in one group only: exactly that (row, group) moves."""
    N, K, d = 128, 512, 2
    codes, A, B, layer = make(N, K, d, seed=3)
    A2 = A.copy()
    A2[7, 2] *= 2
    layer2 = binding.UniSVQLinear(codes, A2, B, group_cols=GC)
    W1, W2 = dequant(layer), dequant(layer2)
    diff = np.argwhere(W1 != W2)
    assert diff.size and np.all(diff[:, 0] == 7) and np.all(diff[:, 1] // GC == 2)
    xb = synth.activations(3, 40, 5, 4, K)
    check(run(layer2, xb), xb, codes, A2, B)
    layer.close()
    layer2.close()


@pytest.mark.parametrize("M", [1, 8, 16])
def test_grouped_group_call_matches_oracle(M):
    K, d = 4096, 2
    shapes = [(1024, K), (520, K), (256, K)]
    made = [synth.layer_inputs_grouped(4, 41, i, 0, N, K_, d) for i, (N, K_) in enumerate(shapes)]
    layers = [binding.UniSVQLinear(c, A, B, group_cols=GC) for c, A, B in made]
    xb = synth.activations(4, 41, M, M, K)
    ys = binding.linear_group(layers, to_dev(xb))
    assert binding.sync_status() == binding.OK
    for (c, A, B), y in zip(made, ys):
        check(y.float().cpu().numpy().astype(np.float64), xb, c, A, B)
    info = binding.query_group(layers, M)
    assert info["kernel"] == binding.KERNEL_GROUPED
    for layer in layers:
        layer.close()


@pytest.mark.parametrize("N,K", [(4096, 4096), (11008, 4096), (4096, 11008)])
def test_grouped_full_size_all_rows(N, K):
    codes, A, B, layer = make(N, K, 2, seed=5)
    for M in (1, 16):
        xb = synth.activations(5, 40, M, M, K)
        check(run(layer, xb), xb, codes, A, B)
    layer.close()


def test_grouped_entry_points():
    N, K, d = 300, 1000, 2
    codes, A, B, layer = make(N, K, d, seed=6)
    info = layer.query(4)
    G = -(-K // GC)
    assert info["kernel"] == binding.KERNEL_GROUPED
    assert info["meta_bytes"] == N * G * (d * d + d) * 2
    assert info["algo_bytes"] == N * K // 4 + info["meta_bytes"] + 2 * 4 * K + 2 * 4 * N
    xb = synth.activations(6, 40, 1, 5, K)
    x = to_dev(xb)
    stream = torch.cuda.current_stream().cuda_stream
    y = torch.zeros((5, N), dtype=torch.bfloat16, device="cuda")
    for kern in (binding.KERNEL_GEMV, binding.KERNEL_SKINNY, binding.KERNEL_GEMV_ROWS):
        assert layer.forward_ptr(x.data_ptr(), y.data_ptr(), 5, stream, kern) == binding.ERR_UNSUPPORTED
    for kern in (binding.KERNEL_AUTO, binding.KERNEL_DECODE, binding.KERNEL_GROUPED, binding.KERNEL_PREFILL):
        assert layer.forward_ptr(x.data_ptr(), y.data_ptr(), 5, stream, kern) == binding.OK
    y.fill_(float("nan"))   # the results of the calls above must not survive
    assert layer.forward_noalloc_ptr(x.data_ptr(), y.data_ptr(), 5, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    check(y.float().cpu().numpy().astype(np.float64), xb, codes, A, B)
    c2 = layer.clone()
    check(run(c2, xb), xb, codes, A, B)
    # a per-matrix layer refuses the per-group kernel, and a mixed group is refused
    pc, pA, pB = synth.layer_inputs(6, 40, 0, 0, N, K, d)
    plain = binding.UniSVQLinear(pc, pA, pB)
    assert plain.forward_ptr(x.data_ptr(), y.data_ptr(), 5, stream, binding.KERNEL_GROUPED) == binding.ERR_UNSUPPORTED
    y2 = torch.zeros((5, N), dtype=torch.bfloat16, device="cuda")
    st = binding.linear_group_ptr([layer, plain], x.data_ptr(), [y.data_ptr(), y2.data_ptr()], 5, stream)
    assert st == binding.ERR_UNSUPPORTED
    assert binding.sync_status() == binding.OK
    for h in (layer, c2, plain):
        h.close()


@pytest.mark.parametrize("d", [1, 2, 4, 8])
@pytest.mark.parametrize("N,K", [(256, 1024), (520, 1000), (1000, 2048), (384, 640)])
def test_grouped_prefill_parity(N, K, d):
    """Per-group layers run the tcgen05 prefill GEMM above 64 tokens (d = 1, 2:
    per-(row, group) codeword-pair tables; d = 4, 8: direct sums)."""
    codes, A, B, layer = make(N, K, d, seed=7)
    assert layer.query(65)["kernel"] == binding.KERNEL_PREFILL
    assert layer.query(64)["kernel"] == binding.KERNEL_GROUPED
    Ms = (65, 200, 300)
    xall = synth.activations(7, 40, N + K, sum(Ms), K)
    yr, S = oracle.linear_grouped(xall, codes, A, B, GC)
    o = 0
    for M in Ms:
        res = oracle.compare(run(layer, xall[o:o + M]), yr[o:o + M], S[o:o + M])
        assert res["ok"], (M, res)
        o += M
    # forced at few tokens too
    res = oracle.compare(run(layer, xall[:9], binding.KERNEL_PREFILL), yr[:9], S[:9])
    assert res["ok"], res
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_grouped_prefill_integer_case_bit_exact(d):
    g = np.random.default_rng(77 + d)
    N, K = 256, 640
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    A = g.integers(-2, 3, size=(N, K // GC, d, d)).astype(np.float16)
    B = g.integers(-2, 3, size=(N, K // GC, d)).astype(np.float16)
    layer = binding.UniSVQLinear(codes, A, B, group_cols=GC)
    x = g.integers(-1, 2, size=(150, K)).astype(np.float32) * (g.random((150, K)) < 0.03)
    xb = synth.f32_to_bf16_bits(x)
    yr, _ = oracle.linear_grouped(xb, codes, A, B, GC)
    assert np.abs(yr).max() <= 256
    yg = run(layer, xb, binding.KERNEL_PREFILL)
    assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


def test_grouped_d8_group_call_runs_one_prefill_launch_per_layer():
    """d = 8 per-group layers run the prefill GEMM, but a group call of them
    takes one launch per layer (their maps fill the converters' shared
    memory); the outputs meet the oracle."""
    K = 512
    made = [synth.layer_inputs_grouped(8, 41, i, 0, N, K, 8) for i, N in enumerate((256, 128))]
    layers = [binding.UniSVQLinear(c, A, B, group_cols=GC) for c, A, B in made]
    assert layers[0].query(200)["kernel"] == binding.KERNEL_PREFILL
    q = binding.query_group(layers, 200)
    assert q["kernel"] == binding.KERNEL_PREFILL and q["launches"] == 2
    xb = synth.activations(8, 41, 200, 200, K)
    ys = binding.linear_group(layers, to_dev(xb))
    assert binding.sync_status() == binding.OK
    for (c, A, B), y in zip(made, ys):
        check(y.float().cpu().numpy().astype(np.float64), xb, c, A, B)
    for l in layers:
        l.close()


@pytest.mark.parametrize("d", [1, 2, 4])
def test_grouped_group_call_at_prefill_sizes(d):
    """Per-group layers that share x run one persistent prefill launch (each
    converter reading its tile's layer's maps): bit-identical to per-layer
    launches, and within the oracle bars."""
    K = 1024
    shapes = [(512, K), (256, K), (200, K)]
    made = [synth.layer_inputs_grouped(9, 42, i, 0, N, K_, d) for i, (N, K_) in enumerate(shapes)]
    layers = [binding.UniSVQLinear(c, A, B, group_cols=GC) for c, A, B in made]
    for M in (96, 300):
        q = binding.query_group(layers, M)
        assert q["kernel"] == binding.KERNEL_PREFILL and q["launches"] == 1
        xb = synth.activations(9, 42, M, M, K)
        x = to_dev(xb)
        ys = binding.linear_group(layers, x)
        assert binding.sync_status() == binding.OK
        for layer, (c, A, B), y in zip(layers, made, ys):
            yl = layer.forward(x, kernel=binding.KERNEL_PREFILL)
            assert binding.sync_status() == binding.OK
            assert np.array_equal(y.view(torch.int16).cpu().numpy(), yl.view(torch.int16).cpu().numpy())
            check(y.float().cpu().numpy().astype(np.float64), xb, c, A, B)
    for layer in layers:
        layer.close()


def test_grouped_pack_rejects_maps_that_do_not_fit():
    """d = 8 per-group maps take 18 KB per k-tile: a 28672-wide layer has no
    GEMV plan, so packing it is refused instead of every call failing."""
    N, K, d = 128, 28672, 8
    G = K // GC
    codes = np.zeros((N, K), dtype=np.uint8)
    A = np.zeros((N, G, d, d), dtype=np.float16)
    B = np.zeros((N, G, d), dtype=np.float16)
    with pytest.raises(binding.UnisvqError) as e:
        binding.UniSVQLinear(codes, A, B, group_cols=GC)
    assert e.value.status == binding.ERR_UNSUPPORTED
    # d = 4 at the same width packs and runs
    A4 = np.zeros((N, G, 4, 4), dtype=np.float16)
    B4 = np.ones((N, G, 4), dtype=np.float16)
    layer = binding.UniSVQLinear(codes, A4, B4, group_cols=GC)
    xb = synth.activations(10, 40, 0, 2, K)
    check(run(layer, xb), xb, codes, A4, B4)
    layer.close()
