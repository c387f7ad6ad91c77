"""GPU parity of libunisvq against the fp64 CPU oracle (needs an sm_103a GPU).

Bars: the fp32 dequantisation hook is bit-exact to RN_fp32 of the exact
codewords; layer outputs meet |y - y_ref| <= 2^-7 sum|w x| + 1e-6 per element
and a relative L2 error <= 4e-3 (oracle.compare); integer-valued cases are
bit-exact.
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


def to_dev(xbits: np.ndarray):
    return torch.from_numpy(np.ascontiguousarray(xbits).view(np.int16)).view(torch.bfloat16).cuda()


def run(layer, xbits, kernel=binding.KERNEL_AUTO):
    y = layer.forward(to_dev(xbits), kernel=kernel)
    st = binding.sync_status()
    assert st == binding.OK, binding.status_string(st)
    return y.float().cpu().numpy().astype(np.float64)


def check(yg, xbits, codes, A, B, rows=None):
    if rows is not None:
        yr, S = oracle.linear(xbits, codes[rows], A, B)
        yg = yg[:, rows]
    else:
        yr, S = oracle.linear(xbits, codes, A, B)
    res = oracle.compare(yg, yr, S)
    assert res["ok"], res
    return res


@pytest.mark.parametrize("d", [1, 2, 4, 8])
@pytest.mark.parametrize("N,K", [(200, 520), (128, 128), (300, 1024)])
def test_dequant_debug_bit_exact(d, N, K):
    codes, A, B = synth.layer_inputs(1, 10, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    W = layer.dequant_debug().cpu().numpy()
    assert binding.sync_status() == binding.OK
    Wref = oracle.dequant_f32(codes, A, B)
    assert np.array_equal(W.view(np.uint32), Wref.view(np.uint32))
    layer.close()


DECODE_SHAPES = [(256, 1024), (520, 1000), (130, 4096), (1024, 8192)]


DECODE_KERNELS = [binding.KERNEL_GEMV, binding.KERNEL_GEMV_ROWS, binding.KERNEL_SKINNY]


@pytest.mark.parametrize("kernel", DECODE_KERNELS)
@pytest.mark.parametrize("d", [1, 2, 4, 8])
@pytest.mark.parametrize("N,K", DECODE_SHAPES)
def test_decode_parity_small_M(kernel, d, N, K):
    if K % d:
        pytest.skip("K % d")
    codes, A, B = synth.layer_inputs(2, 20, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (1, 2, 3, 7, 8, 9, 16, 17, 31, 32, 64):
        xb = synth.activations(2, 20, 1000 * N + M, M, K)
        check(run(layer, xb, kernel), xb, codes, A, B)
    layer.close()


def test_skinny_one_tile_stages_parity():
    """12800 x 1024: 100 row blocks, so one-tile stages (three CTAs per SM)
    allow a K split of 4 against 3 and the planner takes them for the 16- and
    32-column accumulators (M = 3, 10); M = 16 and 17 mix in two-tile stages."""
    N, K, d = 12800, 1024, 2
    codes, A, B = synth.layer_inputs(6, 60, 0, 0, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (3, 10, 16, 17):
        xb = synth.activations(6, 60, M, M, K)
        check(run(layer, xb, binding.KERNEL_SKINNY), xb, codes, A, B)
    layer.close()


@pytest.mark.parametrize("kernel", DECODE_KERNELS)
def test_decode_many_token_groups(kernel):
    N, K, d = 384, 768, 2
    codes, A, B = synth.layer_inputs(3, 30, 0, 0, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (33, 64, 100, 130):
        xb = synth.activations(3, 30, M, M, K)
        check(run(layer, xb, kernel), xb, codes, A, B)
    layer.close()


@pytest.mark.parametrize("kernel", DECODE_KERNELS)
def test_integer_case_bit_exact(kernel):
    """Integer A (the printed D4 generator), integer B and small integer x:
    every intermediate is exact, so the GPU output must equal the oracle's."""
    d = 4
    A = np.array([[1, -1, 0, 0], [0, 1, -1, 0], [0, 0, 1, -1], [0, 0, 1, 1]], dtype=np.float16)
    B = np.array([1, -2, 0, 1], dtype=np.float16)
    N, K = 256, 512
    g = np.random.default_rng(11)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (1, 5, 16):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.05)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear(xb, codes, A, B)
        assert np.abs(yr).max() <= 256
        yg = run(layer, xb, kernel)
        assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


def test_sq_special_case_matches_scalar_dequant():
    """A = s I (d = 1 and d = 4): the layer is a 2-bit SQ GEMV (Eq. def:sq)."""
    for d in (1, 4):
        s, zp = 0.015625, 1.5
        A = (s * np.eye(d)).astype(np.float16)
        B = np.full(d, -s * zp).astype(np.float16)
        N, K = 256, 1024
        codes = synth.gen_codes(synth.rng(4, d), N, K)
        layer = binding.UniSVQLinear(codes, A, B)
        xb = synth.activations(4, 40, d, 4, K)
        check(run(layer, xb, binding.KERNEL_DECODE), xb, codes, A, B)
        layer.close()


def test_zero_tokens_is_noop_and_bad_pointers_rejected():
    N, K, d = 128, 256, 2
    codes, A, B = synth.layer_inputs(5, 50, 0, 0, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    x = torch.zeros((0, K), dtype=torch.bfloat16, device="cuda")
    y = layer(x)
    assert y.shape == (0, N)
    xb = torch.zeros((3, K + 8), dtype=torch.bfloat16, device="cuda")
    ybuf = torch.zeros((3, N), dtype=torch.bfloat16, device="cuda")
    st = layer.forward_ptr(xb.data_ptr() + 2, ybuf.data_ptr(), 3, torch.cuda.current_stream().cuda_stream)
    assert st == binding.ERR_INVALID_ARG
    st = layer.forward_ptr(ybuf.data_ptr(), ybuf.data_ptr(), 3, torch.cuda.current_stream().cuda_stream)
    assert st == binding.ERR_INVALID_ARG
    layer.close()


def test_outputs_do_not_touch_guard_bands():
    N, K, d, M = 130, 384, 2, 5
    codes, A, B = synth.layer_inputs(6, 60, 0, 0, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    xb = synth.activations(6, 60, 0, M, K)
    guard = 4096
    buf = torch.full((guard * 2 + M * N,), 12345.0, dtype=torch.bfloat16, device="cuda")
    fill = float(buf[0].item())
    y = buf[guard:guard + M * N].view(M, N)
    layer.forward(to_dev(xb), out=y)
    assert binding.sync_status() == binding.OK
    host = buf.float().cpu().numpy()
    assert (host[:guard] == fill).all() and (host[guard + M * N:] == fill).all()
    check(y.float().cpu().numpy().astype(np.float64), xb, codes, A, B)
    layer.close()


def test_clone_matches_original():
    N, K, d = 256, 512, 4
    codes, A, B = synth.layer_inputs(7, 70, 0, 0, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    twin = layer.clone()
    xb = synth.activations(7, 70, 0, 4, K)
    a = run(layer, xb)
    b = run(twin, xb)
    assert np.array_equal(a, b)
    twin.close()
    layer.close()


FULL_SHAPES = [(4096, 4096), (11008, 4096), (4096, 11008), (28672, 8192), (8192, 28672)]


@pytest.mark.parametrize("N,K,d", [(N, K, 2) for N, K in FULL_SHAPES] + [(28672, 8192, 4), (8192, 28672, 4)])
def test_full_size_decode_all_rows(N, K, d):
    """Config-sized layers (the Llama-2-7B and -70B projections, and the d = 4
    variant of the 70B crossover workload) at the decode batch sizes: every
    output row of every kernel that runs them against the oracle."""
    codes, A, B = synth.layer_inputs(0, 3, 0, N, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (1, 8, 16, 32):
        xb = synth.activations(0, 3, M, M, K)
        check(run(layer, xb), xb, codes, A, B)
        if M <= 16:
            check(run(layer, xb, binding.KERNEL_SKINNY), xb, codes, A, B)
        if M <= 8:
            check(run(layer, xb, binding.KERNEL_STREAM), xb, codes, A, B)
    layer.close()


# ---------------------------------------------------------------------------
# prefill (tcgen05) kernel
# ---------------------------------------------------------------------------

PREFILL_SHAPES = [(128, 128), (200, 520), (384, 1024), (1000, 2048)]


@pytest.mark.parametrize("d", [1, 2, 4, 8])
@pytest.mark.parametrize("N,K", PREFILL_SHAPES)
def test_prefill_parity(d, N, K):
    codes, A, B = synth.layer_inputs(8, 80, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (33, 64, 65, 128, 200, 256, 300, 777):
        xb = synth.activations(8, 80, 1000 * N + M, M, K)
        check(run(layer, xb, binding.KERNEL_PREFILL), xb, codes, A, B)
    layer.close()


@pytest.mark.parametrize("d", [1, 2, 4])
def test_prefill_group_one_launch(d):
    """Layers that share x (q/k/v-like, ragged N) in one persistent prefill
    launch: every tile computes exactly what the layer's own launch computes,
    so the outputs are bit-identical to per-layer calls and meet the oracle."""
    K = 1024
    shapes = [(520, K), (200, K), (1000, K), (128, K)]
    layers, data = [], []
    for i, (N, _) in enumerate(shapes):
        c, A, B = synth.layer_inputs(8, 85 + i, 0, 0, N, K, d)
        layers.append(binding.UniSVQLinear(c, A, B))
        data.append((c, A, B))
    for n in (2, 3, 4):
        q = binding.query_group(layers[:n], 300)
        assert q["kernel"] == binding.KERNEL_PREFILL and q["launches"] == 1
    for M in (65, 300, 777):
        xb = synth.activations(8, 85, M, M, K)
        x = to_dev(xb)
        got = binding.linear_group(layers, x, kernel=binding.KERNEL_PREFILL)
        assert binding.sync_status() == binding.OK
        for l, y, (c, A, B) in zip(layers, got, data):
            yl = l.forward(x, kernel=binding.KERNEL_PREFILL)
            assert binding.sync_status() == binding.OK
            assert np.array_equal(y.view(torch.int16).cpu().numpy(), yl.view(torch.int16).cpu().numpy())
            check(y.float().cpu().numpy().astype(np.float64), xb, c, A, B)
    for l in layers:
        l.close()


def test_prefill_group_falls_back_per_layer():
    """Mixed d (2 and 4) or a d = 8 layer: one prefill launch per layer."""
    K = 512
    mk = lambda i, N, d: binding.UniSVQLinear(*synth.layer_inputs(8, 90 + i, 0, 0, N, K, d))
    l2, l4, l8 = mk(0, 256, 2), mk(1, 384, 4), mk(2, 128, 8)
    for grp in ([l2, l4], [l2, l8]):
        q = binding.query_group(grp, 200)
        assert q["kernel"] == binding.KERNEL_PREFILL and q["launches"] == 2
    xb = synth.activations(8, 90, 200, 200, K)
    x = to_dev(xb)
    for grp in ([l2, l4], [l8, l2]):
        ys = binding.linear_group(grp, x)
        assert binding.sync_status() == binding.OK
        for l, y in zip(grp, ys):
            yl = l.forward(x, kernel=binding.KERNEL_PREFILL)
            assert np.array_equal(y.view(torch.int16).cpu().numpy(), yl.view(torch.int16).cpu().numpy())
    for l in (l2, l4, l8):
        l.close()


def test_d8_layers_dispatch_to_the_prefill_kernel():
    """d = 8 (the paper's ablation length): above 64 tokens the library picks
    the prefill GEMM, whose converters add two quad-table rows per vector
    (4^8 exact codewords would not fit in shared memory)."""
    d, N, K = 8, 300, 1024
    codes, A, B = synth.layer_inputs(8, 81, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    assert layer.query(200)["kernel"] == binding.KERNEL_PREFILL
    assert layer.query(64)["kernel"] != binding.KERNEL_PREFILL
    for M in (65, 200):
        xb = synth.activations(8, 81, M, M, K)
        check(run(layer, xb), xb, codes, A, B)
    layer.close()


def test_d8_prefill_integer_case_bit_exact():
    """Integer 8 x 8 A and B: every quad-table entry and every fp32 sum of two
    is an exact small integer, so the bf16 weight tile is exact and the output
    must equal the oracle's bit for bit."""
    d = 8
    A = (np.eye(d) - np.eye(d, k=-1) + np.eye(d, k=3)).astype(np.float16)
    B = np.array([1, -2, 0, 1, 3, -1, 0, 2], dtype=np.float16)
    N, K = 384, 1024
    g = np.random.default_rng(18)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (40, 65, 300):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.03)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear(xb, codes, A, B)
        assert np.abs(yr).max() <= 256
        yg = run(layer, xb, binding.KERNEL_PREFILL)
        assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


@pytest.mark.parametrize("kernel", DECODE_KERNELS)
def test_d8_integer_case_bit_exact(kernel):
    """Integer 8 x 8 A (unit lower bidiagonal with -1 below the diagonal),
    integer B and sparse integer x: exact at every step, so the output must
    equal the oracle's bit for bit."""
    d = 8
    A = (np.eye(d) - np.eye(d, k=-1)).astype(np.float16)
    B = np.array([1, -2, 0, 1, 3, -1, 0, 2], dtype=np.float16)
    N, K = 256, 512
    g = np.random.default_rng(17)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (1, 5, 16):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.05)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear(xb, codes, A, B)
        assert np.abs(yr).max() <= 256
        yg = run(layer, xb, kernel)
        assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


def test_prefill_integer_case_bit_exact():
    d = 4
    A = np.array([[1, -1, 0, 0], [0, 1, -1, 0], [0, 0, 1, -1], [0, 0, 1, 1]], dtype=np.float16)
    B = np.array([1, -2, 0, 1], dtype=np.float16)
    N, K = 256, 512
    g = np.random.default_rng(12)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (40, 300):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.05)
        xb = synth.f32_to_bf16_bits(x)
        yr, _ = oracle.linear(xb, codes, A, B)
        assert np.abs(yr).max() <= 256
        yg = run(layer, xb, binding.KERNEL_PREFILL)
        assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    layer.close()


def test_prefill_and_decode_agree_with_auto_dispatch():
    N, K, d = 512, 1024, 2
    codes, A, B = synth.layer_inputs(9, 90, 0, 0, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    assert layer.query(1)["kernel"] == binding.KERNEL_GEMV
    assert layer.query(16)["kernel"] == binding.KERNEL_GEMV
    assert layer.query(64)["kernel"] == binding.KERNEL_GEMV
    assert layer.query(2048)["kernel"] == binding.KERNEL_PREFILL
    xb = synth.activations(9, 90, 0, 96, K)
    check(run(layer, xb), xb, codes, A, B)
    layer.close()


def test_dispatch_picks_tcgen05_decode_for_large_launches():
    """The library's pick (unisvq_query / unisvq_query_group): the tcgen05
    skinny path (fold + streaming kernel: two launches) from 2^26 weights per
    launch, or from 2^25 weights over >= 64 row blocks or above 16 tokens; the
    GEMV otherwise. A launch pair takes 32 tokens where that needs fewer waves
    of row blocks (one CTA per SM) than two 16-token pairs (two per SM), else
    16."""
    big = binding.UniSVQLinear(*synth.layer_inputs(9, 91, 0, 0, 16384, 4096, 2))
    q = big.query(1)
    assert q["kernel"] == binding.KERNEL_SKINNY and q["launches"] == 2
    assert big.query(17)["launches"] == 2 and big.query(33)["launches"] == 4   # 32 tokens per pair
    small = binding.UniSVQLinear(*synth.layer_inputs(9, 91, 1, 0, 4096, 4096, 2))
    assert small.query(16)["kernel"] == binding.KERNEL_GEMV and small.query(16)["launches"] == 1
    tall = binding.UniSVQLinear(*synth.layer_inputs(9, 91, 2, 0, 4096, 11008, 2))   # 2^25.4 weights, 32 row blocks
    assert tall.query(1)["kernel"] == binding.KERNEL_GEMV and tall.query(16)["kernel"] == binding.KERNEL_GEMV
    assert tall.query(32)["kernel"] == binding.KERNEL_SKINNY and tall.query(32)["launches"] == 2
    wide = binding.UniSVQLinear(*synth.layer_inputs(9, 91, 3, 0, 11008, 4096, 2))
    pair = [wide, wide.clone()]            # 172 row blocks: 2 waves either way, so 16 tokens per pair
    assert binding.query_group(pair, 17)["launches"] == 4 and binding.query_group(pair, 32)["launches"] == 4
    xw = synth.activations(9, 91, 5, 20, 4096)
    cw, Aw, Bw = synth.layer_inputs(9, 91, 3, 0, 11008, 4096, 2)
    rows_w = np.unique(np.concatenate([synth.rng(9, 11008, 4096).choice(11008, 48, replace=False), [0, 11007]]))
    for yg in run_group(pair, xw):
        check(yg, xw, cw, Aw, Bw, rows=rows_w)
    for l in pair:
        l.close()
    tall.close()
    trio = [small, small.clone(), small.clone()]
    assert binding.query_group(trio, 1)["kernel"] == binding.KERNEL_SKINNY
    assert binding.query_group(trio[:1], 4)["kernel"] == binding.KERNEL_GEMV
    g4 = binding.query_group(trio, 4)
    assert g4["kernel"] == binding.KERNEL_SKINNY and g4["N"] == 3 * 4096 and g4["launches"] == 2
    xb = synth.activations(9, 91, 4, 4, 4096)
    codes, A, B = synth.layer_inputs(9, 91, 1, 0, 4096, 4096, 2)
    rows = np.unique(np.concatenate([np.sort(synth.rng(9, 4096, 4096).choice(4096, 32, replace=False)), [0, 4095]]))
    for yg in run_group(trio, xb):
        check(yg, xb, codes, A, B, rows=rows)
    for l in trio[1:]:
        l.close()
    small.close()
    big.close()


@pytest.mark.parametrize("N,K", [(4096, 4096), (1024, 4096), (14336, 4096), (4096, 14336)])
def test_full_size_prefill_all_rows(N, K):
    """Llama-3-8B-shaped projections at M = 2048 (the prefill workload), every row."""
    d = 2
    codes, A, B = synth.layer_inputs(0, 2, 0, N + K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    M = 2048
    xb = synth.activations(0, 2, K, M, K)
    check(run(layer, xb), xb, codes, A, B)
    layer.close()


@pytest.mark.parametrize("N,K,d", [(8192, 28672, 2), (28672, 8192, 2), (28672, 8192, 4)])
def test_full_size_prefill_70b_shapes(N, K, d):
    """Llama-2-70B down and gate/up shapes on the crossover sweep's prefill
    sizes (the d = 4 row is that sweep's variant), every row."""
    codes, A, B = synth.layer_inputs(0, 4, d, N + K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    for M in (64, 128, 512, 2048):
        xb = synth.activations(0, 4, K + M, M, K)
        check(run(layer, xb), xb, codes, A, B)
    layer.close()


# ---------------------------------------------------------------------------
# grouped call: several layers that read the same x
# ---------------------------------------------------------------------------
def run_group(layers, xbits, kernel=None):
    ys = binding.linear_group(layers, to_dev(xbits), kernel=kernel)
    st = binding.sync_status()
    assert st == binding.OK, binding.status_string(st)
    return [y.float().cpu().numpy().astype(np.float64) for y in ys]


GROUP_KERNELS = [None, binding.KERNEL_GEMV, binding.KERNEL_SKINNY]


@pytest.mark.parametrize("kernel", GROUP_KERNELS)
@pytest.mark.parametrize("K", [1000, 4096])
@pytest.mark.parametrize("M", [1, 3, 8, 9, 16, 17, 40])
def test_group_matches_oracle(kernel, K, M):
    """Layers of different N and d sharing x, in one call (the library's pick
    or a forced kernel): each output meets the tolerance against the oracle of
    its own layer."""
    specs = [(520, 2), (130, 4), (256, 1)]
    data = [synth.layer_inputs(7, 70, i, K, N, K, d) for i, (N, d) in enumerate(specs)]
    layers = [binding.UniSVQLinear(c, A, B) for c, A, B in data]
    xb = synth.activations(7, 70, M, M, K)
    for (c, A, B), yg in zip(data, run_group(layers, xb, kernel)):
        check(yg, xb, c, A, B)
    for l in layers:
        l.close()


@pytest.mark.parametrize("kernel", GROUP_KERNELS)
def test_group_integer_case_bit_exact(kernel):
    A = np.array([[1, -1, 0, 0], [0, 1, -1, 0], [0, 0, 1, -1], [0, 0, 1, 1]], dtype=np.float16)
    B = np.array([1, -2, 0, 1], dtype=np.float16)
    g = np.random.default_rng(13)
    K = 512
    codes = [g.integers(0, 4, size=(N, K), dtype=np.uint8) for N in (256, 384, 128, 130)]
    layers = [binding.UniSVQLinear(c, A, B) for c in codes]
    for M in (1, 7, 16):
        x = g.integers(-1, 2, size=(M, K)).astype(np.float32) * (g.random((M, K)) < 0.05)
        xb = synth.f32_to_bf16_bits(x)
        for c, yg in zip(codes, run_group(layers, xb, kernel)):
            yr, _ = oracle.linear(xb, c, A, B)
            assert np.array_equal(yg, yr), np.abs(yg - yr).max()
    for l in layers:
        l.close()


def test_group_rejects_mismatched_k_and_overlap():
    a = binding.UniSVQLinear(*synth.layer_inputs(3, 30, 0, 0, 256, 512, 2))
    b = binding.UniSVQLinear(*synth.layer_inputs(3, 30, 1, 0, 256, 1024, 2))
    x = torch.zeros((2, 512), dtype=torch.bfloat16, device="cuda")
    y0 = torch.zeros((2, 256), dtype=torch.bfloat16, device="cuda")
    y1 = torch.zeros((2, 256), dtype=torch.bfloat16, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    assert binding.linear_group_ptr([a, b], x.data_ptr(), [y0.data_ptr(), y1.data_ptr()], 2, s) == \
        binding.ERR_INVALID_ARG
    c = a.clone()
    assert binding.linear_group_ptr([a, c], x.data_ptr(), [y0.data_ptr(), y0.data_ptr()], 2, s) == \
        binding.ERR_INVALID_ARG
    assert binding.linear_group_ptr([a, c], x.data_ptr(), [y0.data_ptr(), y1.data_ptr()], 2, s) == binding.OK
    assert binding.sync_status() == binding.OK
    for l in (a, b, c):
        l.close()
