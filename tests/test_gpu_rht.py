"""The randomized Hadamard transform (Eq. def:hadamard) on the GPU against the
fp64 oracle: the rotation alone (every supported order family, including
the order-344 Paley factor of 11008 = 2^5 * 344, both sign placements, in
place and out of place), and the layer with the inverse
rotation around it (per-matrix and per-group layers, chunked token counts,
forced kernels, grouped calls)."""
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


def host(t):
    return t.float().cpu().numpy().astype(np.float64)


def signs(n, seed):
    return np.random.default_rng(seed).choice([-1.0, 1.0], size=n)


@pytest.mark.parametrize("n", [12, 20, 28, 64, 96, 344, 448, 688, 4096, 5120, 5504, 11008, 14336, 28672])
@pytest.mark.parametrize("signs_first", [1, 0])
def test_rotation_matches_oracle(n, signs_first):
    M = 3
    xb = synth.activations(7, 50, n, M, n)
    x = to_dev(xb)
    s = signs(n, n)
    sd = torch.from_numpy((s < 0).astype(np.uint8)).cuda()
    y = torch.empty_like(x)
    stream = torch.cuda.current_stream().cuda_stream
    assert binding.hadamard_ptr(x.data_ptr(), y.data_ptr(), M, n, sd.data_ptr(), signs_first, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    xf = oracle.bf16_bits_to_f64(xb)
    H = oracle.hadamard(n) / np.sqrt(n)
    ref = (xf * s) @ H if signs_first else (xf @ H) * s
    got = host(y)
    rms = np.sqrt(np.mean(ref ** 2))
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5 * rms), np.abs(got - ref).max()
    # in place gives the same bits
    z = x.clone()
    assert binding.hadamard_ptr(z.data_ptr(), z.data_ptr(), M, n, sd.data_ptr(), signs_first, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    assert torch.equal(z, y)


@pytest.mark.parametrize("n", [448, 11008])
def test_rotation_of_rows_not_16_byte_aligned(n):
    """Rows that start 2 bytes past a 16-byte boundary take the element-wise
    load path and give the same values as aligned rows."""
    M = 2
    xb = synth.activations(7, 55, n, M, n)
    buf = torch.zeros(M * n + 8, dtype=torch.bfloat16, device="cuda")
    x = buf[1:1 + M * n].view(M, n)
    x.copy_(to_dev(xb))
    s = signs(n, n + 1)
    sd = torch.from_numpy((s < 0).astype(np.uint8)).cuda()
    stream = torch.cuda.current_stream().cuda_stream
    y_al = torch.empty((M, n), dtype=torch.bfloat16, device="cuda")
    xa = to_dev(xb)
    assert binding.hadamard_ptr(xa.data_ptr(), y_al.data_ptr(), M, n, sd.data_ptr(), 1, stream) == binding.OK
    assert binding.hadamard_ptr(x.data_ptr(), x.data_ptr(), M, n, sd.data_ptr(), 1, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    assert torch.equal(x, y_al)


def test_rotation_without_signs_and_bad_orders():
    n, M = 256, 2
    xb = synth.activations(7, 51, 0, M, n)
    x = to_dev(xb)
    y = torch.empty_like(x)
    stream = torch.cuda.current_stream().cuda_stream
    assert binding.hadamard_ptr(x.data_ptr(), y.data_ptr(), M, n, 0, 1, stream) == binding.OK
    assert binding.sync_status() == binding.OK
    ref = oracle.bf16_bits_to_f64(xb) @ (oracle.hadamard(n) / 16.0)
    assert np.allclose(host(y), ref, rtol=2.0 ** -8, atol=1e-5)
    for bad in (36, 100, 172, 6880):
        xb2 = torch.zeros((1, bad), dtype=torch.bfloat16, device="cuda")
        yb2 = torch.zeros((1, bad), dtype=torch.bfloat16, device="cuda")
        assert binding.hadamard_ptr(xb2.data_ptr(), yb2.data_ptr(), 1, bad, 0, 1, stream) == binding.ERR_UNSUPPORTED
    assert binding.hadamard_ptr(x.data_ptr(), y.data_ptr(), 1, n, 0, 2, stream) == binding.ERR_INVALID_ARG


@pytest.mark.parametrize("N,K,d", [(4096, 4096, 2), (1792, 3584, 2), (640, 1280, 4), (768, 2560, 1),
                                   (11008, 4096, 2), (4096, 11008, 2)])
def test_layer_with_inverse_rht(N, K, d):
    codes, A, B = synth.layer_inputs(7, 52, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    s_U, s_V = signs(N, 1 + N), signs(K, 2 + K)
    layer.set_rht(s_V, s_U, max_tokens=64)
    Ms = (1, 5, 16, 70)
    xall = synth.activations(7, 52, N + K, sum(Ms), K)
    yr, S = oracle.linear_rht(xall, codes, A, B, s_U, s_V)
    o = 0
    for M in Ms:
        y = layer.forward(to_dev(xall[o:o + M]))
        assert binding.sync_status() == binding.OK
        res = oracle.compare(host(y), yr[o:o + M], S[o:o + M])
        assert res["ok"], (M, res)
        o += M
    info = layer.query(70)
    assert info["launches"] >= 2 * 2   # two chunks, an input and an output rotation each
    # a forced kernel keeps the rotations; removing them restores the plain layer
    x5 = to_dev(xall[:5])
    for kern in (binding.KERNEL_GEMV, binding.KERNEL_SKINNY):
        y = layer.forward(x5, kernel=kern)
        assert binding.sync_status() == binding.OK
        assert oracle.compare(host(y), yr[:5], S[:5])["ok"]
    layer.set_rht(None, None)
    y = layer.forward(x5)
    assert binding.sync_status() == binding.OK
    yp, Sp = oracle.linear(xall[:5], codes, A, B)
    assert oracle.compare(host(y), yp, Sp)["ok"]
    layer.close()


def test_grouped_layer_and_group_call_with_rht():
    K, d = 1024, 2
    shapes = [(512, K), (256, K)]
    made = [synth.layer_inputs_grouped(7, 53, i, 0, N, K_, d) for i, (N, K_) in enumerate(shapes)]
    layers = [binding.UniSVQLinear(c, A, B, group_cols=128) for c, A, B in made]
    sg = [(signs(N, 10 + i), signs(K, 20 + i)) for i, (N, _) in enumerate(shapes)]
    for layer, (s_U, s_V) in zip(layers, sg):
        layer.set_rht(s_V, s_U, max_tokens=8)
    M = 12
    xb = synth.activations(7, 53, 0, M, K)
    ys = binding.linear_group(layers, to_dev(xb))
    assert binding.sync_status() == binding.OK
    for (c, A, B), (s_U, s_V), y in zip(made, sg, ys):
        xt = oracle.rht_input(xb, s_V)
        yt, St = oracle.linear_grouped(xt, c, A, B, 128)
        N = c.shape[0]
        ref = oracle.rht_output(yt, s_U)
        Sref = St @ (np.abs(oracle.hadamard(N)) / np.sqrt(N))
        assert oracle.compare(host(y), ref, Sref)["ok"]
    for layer in layers:
        layer.close()


def test_set_rht_rejects_unsupported_widths_and_bad_signs():
    N, K = 4608, 4096      # 4608 = 2^9 * 9: no Hadamard order here
    codes = np.zeros((N, K), dtype=np.uint8)
    layer = binding.UniSVQLinear(codes, np.eye(2, dtype=np.float16), np.zeros(2, dtype=np.float16))
    with pytest.raises(binding.UnisvqError) as e:
        layer.set_rht(np.ones(K), np.ones(N))
    assert e.value.status == binding.ERR_UNSUPPORTED
    layer.close()
    layer = binding.UniSVQLinear(np.zeros((256, 512), dtype=np.uint8), np.eye(2, dtype=np.float16),
                                 np.zeros(2, dtype=np.float16))
    bad = np.zeros(512, dtype=np.uint8)
    bad[3] = 2
    with pytest.raises(binding.UnisvqError) as e:
        layer.set_rht(bad, np.zeros(256, dtype=np.uint8))
    assert e.value.status == binding.ERR_INVALID_ARG
    layer.close()


@pytest.mark.parametrize("M,Ns", [(1, (4096, 1024, 1024)), (16, (4096, 1024, 1024)), (40, (4096, 1024, 1024)),
                                  (5, (11008, 11008)), (16, (11008, 11008)), (3, (4096, 14336)),
                                  (7, (1024, 11008, 4096))])
def test_group_call_sharing_the_input_rotation(M, Ns):
    """Layers that share S_V (same input space) rotate x once and run as one
    group; each output still gets its own U S_U. The output rotations of
    widths with one H_m and cluster size run as one launch (4096 and 1024,
    11008 twice), the others one launch per width (4096 with 14336 = 2^9 * 28,
    11008 = 2^5 * 344 with powers of two)."""
    K, d = 4096, 2
    shapes = [(N, K) for N in Ns]
    made = [synth.layer_inputs(7, 54, i, 0, N, K_, d) for i, (N, K_) in enumerate(shapes)]
    layers = [binding.UniSVQLinear(c, A, B) for c, A, B in made]
    s_V = signs(K, 99)
    s_Us = [signs(N, 100 + i) for i, (N, _) in enumerate(shapes)]
    for layer, s_U in zip(layers, s_Us):
        layer.set_rht(s_V, s_U, max_tokens=16)
    xb = synth.activations(7, 54, M, M, K)
    ys = binding.linear_group(layers, to_dev(xb))
    assert binding.sync_status() == binding.OK
    for (c, A, B), s_U, y in zip(made, s_Us, ys):
        ref, S = oracle.linear_rht(xb, c, A, B, s_U, s_V)
        res = oracle.compare(host(y), ref, S)
        assert res["ok"], res
    for layer in layers:
        layer.close()


@pytest.mark.parametrize("N,K,d", [(4096, 4096, 2), (4096, 14336, 2), (1024, 5120, 4), (1024, 3072, 2),
                                   (1024, 2048, 8), (1792, 3584, 2), (512, 1536, 1)])
def test_input_rotation_fused_into_the_fold(N, K, d):
    """The tcgen05 decode path rotates x inside its fold kernel where K = 2^a m
    (m in 1, 12, 20, 28) splits into full slices of whole blocks (4096, 14336
    = 2^9 * 28, 5120 = 2^8 * 20, 3072 = 2^8 * 12, 2048 with d = 8); K = 3584
    and 1536 split into 7 and 6 slices and take the separate rotation. The
    layer matches the oracle for token counts inside one launch and across
    two."""
    codes, A, B = synth.layer_inputs(7, 56, N, K, N, K, d)
    layer = binding.UniSVQLinear(codes, A, B)
    s_U, s_V = signs(N, 3 + N), signs(K, 4 + K)
    layer.set_rht(s_V, s_U, max_tokens=8)
    Ms = (1, 7, 16, 33)
    xall = synth.activations(7, 56, N + K, sum(Ms), K)
    yr, S = oracle.linear_rht(xall, codes, A, B, s_U, s_V)
    o = 0
    for M in Ms:
        y = layer.forward(to_dev(xall[o:o + M]), kernel=binding.KERNEL_SKINNY)
        assert binding.sync_status() == binding.OK
        res = oracle.compare(host(y), yr[o:o + M], S[o:o + M])
        assert res["ok"], (M, res)
        o += M
    layer.close()


def test_fused_rotation_launch_counts():
    """Where the call resolves to the tcgen05 path, the RHT adds one launch
    (the output rotation): the fold kernel rotates the input."""
    K = 4096
    big = binding.UniSVQLinear(*synth.layer_inputs(7, 57, 0, 0, 14336, K, 2))
    big.set_rht(signs(K, 5), signs(14336, 6), max_tokens=8)
    assert big.query(5)["kernel"] == binding.KERNEL_SKINNY
    assert big.query(5)["launches"] == 2 + 1       # K split 2 or more: fused
    # 40 tokens: the 32-token launch does not split K (one CTA per row block
    # fills the GPU), so the separate rotations run, per chunk of 8 tokens
    assert big.query(40)["launches"] == 4 + 2 * 5
    xb = synth.activations(7, 57, 0, 5, K)
    y = big.forward(to_dev(xb))
    assert binding.sync_status() == binding.OK
    c, A, B = synth.layer_inputs(7, 57, 0, 0, 14336, K, 2)
    ref, S = oracle.linear_rht(xb, c, A, B, signs(14336, 6), signs(K, 5))
    assert oracle.compare(host(y), ref, S)["ok"]
    big.close()
    # a Llama-2-7B q/k/v group (3 x 4096 x 4096) sharing S_V: fold + decode + one output launch
    made = [synth.layer_inputs(7, 58, i, 0, 4096, K, 2) for i in range(3)]
    layers = [binding.UniSVQLinear(c, A, B) for c, A, B in made]
    s_V = signs(K, 7)
    s_Us = [signs(4096, 8 + i) for i in range(3)]
    for layer, s_U in zip(layers, s_Us):
        layer.set_rht(s_V, s_U, max_tokens=8)
    info = binding.query_group(layers, 16)
    assert info["kernel"] == binding.KERNEL_SKINNY and info["launches"] == 2 + 1
    xb = synth.activations(7, 58, 0, 16, K)
    ys = binding.linear_group(layers, to_dev(xb))
    assert binding.sync_status() == binding.OK
    for (c, A, B), s_U, y in zip(made, s_Us, ys):
        ref, S = oracle.linear_rht(xb, c, A, B, s_U, s_V)
        assert oracle.compare(host(y), ref, S)["ok"]
    for layer in layers:
        layer.close()
