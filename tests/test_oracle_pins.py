"""Pins of the CPU oracle to facts the paper and mathematics fix (no GPU).

Each pin is written as a function of the dequantisation / layer routine under
test, so `test_pins_catch_planted_mistakes` can run the same pins against
deliberately broken copies of the oracle and show each mistake is caught.
"""
import itertools
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_worked.json")


# --------------------------------------------------------------------------
# pin functions: each returns None on success, raises AssertionError otherwise
# --------------------------------------------------------------------------

def haar_orthogonal(d, seed):
    """Haar-distributed orthogonal matrix (QR of a Gaussian with sign fix)."""
    g = np.random.default_rng(seed)
    Q, R = np.linalg.qr(g.standard_normal((d, d)))
    return Q * np.sign(np.diag(R))


def pin_enumeration_moments(dequant_fn, d, seed=0, bits=2):
    """Eq. (def:affine), App. A.1: with A = sG (G orthogonal), B = -sG b 1,
    b = (2^bits-1)/2 and s = sqrt(12/(2^(2 bits)-1)), the 2^(bits d)
    codewords, each taken once (the uniform law on {0..2^bits-1}^d), have mean
    exactly 0 and covariance exactly I."""
    G = haar_orthogonal(d, seed)
    b = (2 ** bits - 1) / 2
    s = np.sqrt(12.0 / (2 ** (2 * bits) - 1))
    A = s * G
    B = -s * G @ (b * np.ones(d))
    pts = np.array(list(itertools.product(range(2 ** bits), repeat=d)), dtype=np.uint8)
    W = dequant_fn(pts, A, B)            # one codeword per row (K = d)
    mean = W.mean(axis=0)
    cov = (W - mean).T @ (W - mean) / W.shape[0]
    assert np.allclose(mean, 0.0, atol=1e-12), mean
    assert np.allclose(cov, np.eye(d), atol=1e-12), cov


def pin_sq_special_case(dequant_fn, d=4, seed=1):
    """Eq. (def:sq): with A = s I and B = -s zp 1 the grid is scalar
    quantisation. Re-quantising W_hat with the SQ rule must give back the
    codes (clamp inactive), and SQ dequantisation s (q - zp) must equal W_hat."""
    g = np.random.default_rng(seed)
    s, zp = 0.0625, 1.5
    codes = g.integers(0, 4, size=(7, 8 * d), dtype=np.uint8)
    W = dequant_fn(codes, s * np.eye(d), -s * zp * np.ones(d))
    q = np.clip(np.rint(W / s + zp), 0, 3)          # Phi_SQ quantiser
    assert np.array_equal(q.astype(np.uint8), codes)
    assert np.array_equal(W, s * (q - zp))           # Phi_SQ dequantiser


def pin_block_form(dequant_fn, d, seed=2):
    """Eq. (col:dequant) builds W^T by stacking, for each group i of d input
    columns, the block A W_int,i^T + B 1^T. Built here with exact rationals
    and explicit loops; it must equal the per-vector Eq. (def:unisvq) form."""
    g = np.random.default_rng(seed)
    N, K = 3, 3 * d
    A = g.integers(-3, 4, size=(d, d)).astype(np.float64) / 4
    B = g.integers(-3, 4, size=d).astype(np.float64) / 8
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    Af = [[Fraction(v) for v in row] for row in A]
    Bf = [Fraction(v) for v in B]
    WT = []                                            # rows of W^T (K of them)
    for i in range(K // d):
        Wi = [[int(codes[n, i * d + c]) for c in range(d)] for n in range(N)]  # W_int,i [N][d]
        for r in range(d):                             # block row r = (A W_int,i^T + B 1^T)[r]
            WT.append([sum(Af[r][c] * Wi[n][c] for c in range(d)) + Bf[r] for n in range(N)])
    Wref = np.array([[float(WT[k][n]) for k in range(K)] for n in range(N)])
    assert np.array_equal(dequant_fn(codes, A, B), Wref)


def pin_integer_layer_exact(linear_fn, seed=3):
    """The printed D4 generator (App. A.2) is an integer, non-symmetric A:
    with integer B and small integer x every product is an exact integer, so
    the layer output must equal exact integer arithmetic done with Python
    ints on the block form of Eq. (col:dequant)."""
    d = 4
    A = np.array([[1, -1, 0, 0], [0, 1, -1, 0], [0, 0, 1, -1], [0, 0, 1, 1]], dtype=np.float64)
    B = np.array([1, -2, 0, 3], dtype=np.float64)
    g = np.random.default_rng(seed)
    N, K, M = 5, 12, 3
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    x = g.integers(-5, 6, size=(M, K)).astype(np.float64)
    Ai = A.astype(int).tolist()
    Bi = B.astype(int).tolist()
    yref = np.zeros((M, N))
    for m in range(M):
        for n in range(N):
            acc = 0
            for i in range(K // d):
                for r in range(d):
                    w = sum(Ai[r][c] * int(codes[n, i * d + c]) for c in range(d)) + Bi[r]
                    acc += int(x[m, i * d + r]) * w
            yref[m, n] = acc
    y = linear_fn(x, codes, A, B)
    assert np.array_equal(y, yref), (y, yref)


def pin_golden(dequant_fn, linear_fn):
    """Hand-worked examples in tests/golden/hand_worked.json."""
    with open(GOLDEN) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        A = np.array(c["A"])
        B = np.array(c["B"])
        codes = np.array(c["codes"], dtype=np.uint8)
        x = np.array(c["x"])
        assert np.array_equal(dequant_fn(codes, A, B), np.array(c["W"])), c["name"]
        assert np.array_equal(linear_fn(x, codes, A, B), np.array(c["y"])), c["name"]


def pin_linearity(linear_fn, seed=4):
    """The layer is linear in x: y(a x1 + b x2) = a y(x1) + b y(x2)."""
    g = np.random.default_rng(seed)
    codes = g.integers(0, 4, size=(9, 16), dtype=np.uint8)
    A = g.standard_normal((2, 2))
    B = g.standard_normal(2)
    x1 = g.standard_normal((3, 16))
    x2 = g.standard_normal((3, 16))
    lhs = linear_fn(0.75 * x1 - 1.25 * x2, codes, A, B)
    rhs = 0.75 * linear_fn(x1, codes, A, B) - 1.25 * linear_fn(x2, codes, A, B)
    assert np.allclose(lhs, rhs, rtol=1e-12, atol=1e-12)


def oracle_linear_y(x, codes, A, B):
    return oracle.linear(np.asarray(x, dtype=np.float64), codes, A, B)[0]


# --------------------------------------------------------------------------
# the pins, applied to the oracle
# --------------------------------------------------------------------------

@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_enumeration_moments(d):
    pin_enumeration_moments(oracle.dequant, d)


def test_sq_special_case():
    pin_sq_special_case(oracle.dequant)


@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_block_form_matches_vector_form(d):
    pin_block_form(oracle.dequant, d)


def test_integer_layer_exact():
    pin_integer_layer_exact(oracle_linear_y)


def test_golden_hand_worked():
    pin_golden(oracle.dequant, oracle_linear_y)
    with open(GOLDEN) as f:
        for c in json.load(f)["cases"]:
            y, S = oracle.linear(np.array(c["x"]), np.array(c["codes"], dtype=np.uint8),
                                 np.array(c["A"]), np.array(c["B"]))
            assert np.array_equal(S, np.array(c["S"]))


def test_linearity():
    pin_linearity(oracle_linear_y)


@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_fold_identity(d):
    """Eq. (col:matmul) (fold onto activations) equals the direct form."""
    g = synth.rng(0, 99, d)
    codes = synth.gen_codes(g, 33, 64 * d)
    A, B = synth.gen_affine(g, d)
    x = synth.gen_activations(g, 5, 64 * d)
    y, S = oracle.linear(x, codes, A, B)
    yf = oracle.linear_folded(x, codes, A, B)
    assert np.allclose(yf, y, rtol=1e-11, atol=1e-11 * np.abs(S).max())


def test_codebook_is_dequant_of_every_index():
    """`codebook` row v is the dequantisation of the lattice point whose
    coordinate c is bit-field [2c+1:2c] of v."""
    for d in (1, 2, 4, 8):
        g = np.random.default_rng(d)
        A = g.standard_normal((d, d))
        B = g.standard_normal(d)
        v = np.arange(4 ** d)
        pts = np.stack([(v >> (2 * c)) & 3 for c in range(d)], axis=1).astype(np.uint8)
        cb = oracle.codebook(A, B)
        assert np.allclose(cb, oracle.dequant(pts, A, B), rtol=0, atol=1e-14 * np.abs(cb).max())


def test_dequant_f32_single_rounding():
    g = np.random.default_rng(5)
    codes = g.integers(0, 4, size=(4, 8), dtype=np.uint8)
    A, B = synth.gen_affine(g, 2)
    W = oracle.dequant(codes, A, B)
    W32 = oracle.dequant_f32(codes, A, B)
    assert W32.dtype == np.float32
    assert np.all(np.abs(W32.astype(np.float64) - W) <= np.abs(W) * 2.0 ** -24)


def test_compare_accepts_and_rejects():
    g = np.random.default_rng(6)
    y = g.standard_normal((4, 8))
    S = np.abs(y) + 1.0
    assert oracle.compare(y, y, S)["ok"]
    bad = y.copy()
    bad[1, 3] += 0.1 * S[1, 3]
    assert not oracle.compare(bad, y, S)["ok"]


# --------------------------------------------------------------------------
# planted mistakes: each broken oracle must fail at least one pin
# --------------------------------------------------------------------------

def _mut_dequant(kind):
    def f(codes, A, B):
        A = np.asarray(A, dtype=np.float64)
        B = np.asarray(B, dtype=np.float64)
        d = A.shape[0]
        N, K = codes.shape
        if kind == "transpose_A":
            A = A.T
        if kind == "drop_B":
            B = 0 * B
        if kind == "neg_B":
            B = -B
        Z = codes.reshape(N, K // d, d).astype(np.float64)
        if kind == "reverse_coords":
            Z = Z[..., ::-1]
        if kind == "vectors_along_output" and N % d == 0:
            Z = codes.T.reshape(K, N // d, d).astype(np.float64)
            W = (Z @ A.T + B).reshape(K, N).T
            return W
        W = Z @ A.T + B
        if kind == "scale_off":
            W = W * (1 + 2.0 ** -20)
        return W.reshape(N, K)
    return f


def _linear_from(dequant_fn):
    def f(x, codes, A, B):
        return np.asarray(x, dtype=np.float64) @ dequant_fn(codes, A, B).T
    return f


@pytest.mark.parametrize("kind", ["transpose_A", "drop_B", "neg_B", "reverse_coords",
                                  "vectors_along_output", "scale_off"])
def test_pins_catch_planted_mistakes(kind):
    dq = _mut_dequant(kind)
    lin = _linear_from(dq)
    checks = [
        lambda: pin_enumeration_moments(dq, 2),
        lambda: pin_enumeration_moments(dq, 4),
        lambda: pin_sq_special_case(dq),
        lambda: pin_block_form(dq, 2),
        lambda: pin_block_form(dq, 4),
        lambda: pin_integer_layer_exact(lin),
        lambda: pin_golden(dq, lin),
    ]
    failed = 0
    for chk in checks:
        try:
            chk()
        except (AssertionError, ValueError):
            failed += 1
    assert failed >= 1, f"planted mistake {kind!r} passed every pin"


def test_synth_code_probabilities():
    c = synth.gen_codes(synth.rng(0, 1), 512, 1024)
    p = np.bincount(c.ravel(), minlength=4) / c.size
    assert np.allclose(p, synth.CODE_PROBS, atol=3e-3)
    assert c.max() <= 3


def test_synth_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    v = np.random.default_rng(7).standard_normal(4096).astype(np.float32) * 37
    ours = synth.f32_to_bf16_bits(v)
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


# --------------------------------------------------------------------------
# per-(row, group) affine maps
# --------------------------------------------------------------------------

GROUPED_GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "grouped_hand_worked.json")


def test_grouped_golden_hand_worked():
    """The hand-worked per-group example: W, y and S exactly."""
    with open(GROUPED_GOLDEN) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        A = np.array(c["A"])
        B = np.array(c["B"])
        codes = np.array(c["codes"], dtype=np.uint8)
        x = np.array(c["x"])
        gc = c["group_cols"]
        assert np.array_equal(oracle.dequant_grouped(codes, A, B, gc), np.array(c["W"])), c["name"]
        y, S = oracle.linear_grouped(x, codes, A, B, gc)
        assert np.array_equal(y, np.array(c["y"])), c["name"]
        assert np.array_equal(S, np.array(c["S"])), c["name"]
        assert np.array_equal(oracle.linear_grouped_moments(x, codes, A, B, gc), np.array(c["y"])), c["name"]


@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_grouped_scalar_case_is_groupwise_uniform_quantisation(d):
    """A[n][g] = s[n][g] I, B[n][g] = b[n][g] 1: every weight is s z + b with
    the scale and offset of its row and 128-column group -- group-wise uniform
    2-bit dequantisation (per-row scale/offset broadcast along columns)."""
    g = np.random.default_rng(40 + d)
    N, K, gc = 5, 3 * 128 + 64, 128
    G = -(-K // gc)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    s = g.standard_normal((N, G))
    b = g.standard_normal((N, G))
    A = s[:, :, None, None] * np.eye(d)
    B = np.repeat(b[:, :, None], d, axis=2)
    s_col = np.repeat(s, gc, axis=1)[:, :K]
    b_col = np.repeat(b, gc, axis=1)[:, :K]
    expect = s_col * codes + b_col
    assert np.array_equal(oracle.dequant_grouped(codes, A, B, gc), expect)


@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_grouped_with_one_map_everywhere_is_the_per_matrix_layer(d):
    g = synth.rng(0, 98, d)
    N, K = 7, 2 * 128 + 8 * d
    codes = synth.gen_codes(g, N, K)
    A1, B1 = synth.gen_affine(g, d)
    G = -(-K // 128)
    A = np.broadcast_to(A1, (N, G, d, d))
    B = np.broadcast_to(B1, (N, G, d))
    assert np.array_equal(oracle.dequant_grouped(codes, A, B), oracle.dequant(codes, A1, B1))


@pytest.mark.parametrize("d", [1, 2, 4, 8])
def test_grouped_moment_form_matches_direct_form(d):
    """Exchanging the sums (codes meet the activations before A does) gives
    the same output, with a different non-symmetric A per row and group."""
    g = np.random.default_rng(70 + d)
    N, M, K = 6, 3, 2 * 128 + 16 * d
    G = -(-K // 128)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    A = g.standard_normal((N, G, d, d))
    B = g.standard_normal((N, G, d))
    x = g.standard_normal((M, K))
    y, S = oracle.linear_grouped(x, codes, A, B)
    ym = oracle.linear_grouped_moments(x, codes, A, B)
    assert np.allclose(ym, y, rtol=0, atol=1e-12 * S.max())


def test_grouped_linearity_and_row_chunks():
    g = np.random.default_rng(5)
    N, K, d = 11, 256, 2
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    A = g.standard_normal((N, 2, d, d))
    B = g.standard_normal((N, 2, d))
    x1 = g.standard_normal((2, K))
    x2 = g.standard_normal((2, K))
    f = lambda x, rc=256: oracle.linear_grouped(x, codes, A, B, 128, rc)[0]
    assert np.allclose(f(0.5 * x1 + 2 * x2), 0.5 * f(x1) + 2 * f(x2), rtol=1e-12, atol=1e-12)
    assert np.allclose(f(x1, 3), f(x1), rtol=1e-13, atol=1e-13)


# --------------------------------------------------------------------------
# randomized Hadamard transform, Eq. (def:hadamard)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("n", [1, 2, 8, 12, 20, 28, 64, 96, 112, 160, 344, 448, 688, 1024])
def test_hadamard_is_orthogonal_pm1(n):
    H = oracle.hadamard(n)
    assert H.shape == (n, n) and set(np.unique(H)) <= {-1, 1}
    assert np.array_equal(H @ H.T, n * np.eye(n, dtype=np.int64))


def test_sylvester_matches_scipy():
    scipy_linalg = pytest.importorskip("scipy.linalg")
    for n in (1, 2, 4, 64, 512):
        assert np.array_equal(oracle.hadamard(n), scipy_linalg.hadamard(n))


def test_hadamard_factor_of_model_widths():
    assert oracle.hadamard_factor(4096) == (4096, 1)
    assert oracle.hadamard_factor(14336) == (512, 28)
    assert oracle.hadamard_factor(28672) == (1024, 28)
    assert oracle.hadamard_factor(11008) == (32, 344)   # 2^5 * (7^3 + 1)
    assert oracle.hadamard_factor(11008 // 2 * 3) is None
    with pytest.raises(ValueError):
        oracle.hadamard(172)


# GF(343) and the order-344 Paley matrix: pinned to the field axioms, the
# character's defining property and H H^T = n I, not to the oracle's own output.

def gf343_field_ok(o) -> bool:
    """The modulus has no root in GF(7), and the multiplication table of the
    343 elements is that of a field: commutative, associative on a sample,
    distributive over the coefficient-wise sum, every nonzero row a
    permutation of the nonzero elements (inverses exist and are unique)."""
    r0, r1, r2 = o._GF343_T3
    if any((t ** 3 - (r0 + r1 * t + r2 * t * t)) % 7 == 0 for t in range(7)):
        return False
    e = np.arange(343)
    T = o.gf343_mul(e[:, None], e[None, :])
    if not np.array_equal(T, T.T) or np.any(T[0] != 0) or np.any(T[1] != e):
        return False
    if any(sorted(T[a, 1:]) != list(range(1, 343)) for a in range(1, 343)):
        return False
    g = np.random.default_rng(343)
    a, b, c = (g.integers(0, 343, size=2000) for _ in range(3))
    if not np.array_equal(T[T[a, b], c], T[a, T[b, c]]):
        return False
    add = lambda u, v: o.gf343_sub(u, o.gf343_sub(0, v))
    return bool(np.array_equal(T[a, add(b, c)], add(T[a, b], T[a, c])))


def paley344_ok(o) -> bool:
    """chi is multiplicative with 171 squares and chi(-1) = -1 (343 = 3 mod 4);
    the matrix is +-1, of Paley form (first row all +1, H - I antisymmetric)
    and H H^T = 344 I."""
    chi = o.gf343_quadratic_character()
    e = np.arange(343)
    T = o.gf343_mul(e[:, None], e[None, :])
    if not np.array_equal(chi[T], chi[:, None] * chi[None, :]):
        return False
    if (chi == 1).sum() != 171 or chi[o.gf343_sub(0, 1)] != -1:
        return False
    H = o.paley_hadamard(344)
    S = H - np.eye(344, dtype=np.int64)
    return bool(set(np.unique(H)) <= {-1, 1} and np.all(H[0] == 1) and np.array_equal(S, -S.T)
                and np.array_equal(H @ H.T, 344 * np.eye(344, dtype=np.int64)))


def test_gf343_is_a_field():
    assert gf343_field_ok(oracle)


def test_paley_344_is_hadamard():
    assert paley344_ok(oracle)


def test_hadamard_11008_is_sylvester_32_kron_paley_344():
    """Entries and orthogonality of sampled rows of the order-11008 matrix."""
    H = oracle.hadamard(11008)
    H344 = oracle.paley_hadamard(344)
    g = np.random.default_rng(11008)
    i, j = g.integers(0, 11008, size=(2, 3000))
    p, q, pp, qq = i // 344, i % 344, j // 344, j % 344
    syl = np.where(np.bitwise_count(p & pp) % 2 == 1, -1, 1)   # Sylvester: (-1)^popcount(p & p')
    assert np.array_equal(H[i, j], syl * H344[q, qq])
    rows = g.choice(11008, size=12, replace=False)
    G = H[rows] @ H[rows].T
    assert np.array_equal(G, 11008 * np.eye(12, dtype=np.int64))


def test_gf343_pins_catch_planted_mistakes(monkeypatch):
    # a reducible modulus (t^3 - t - 1 has the root 5 mod 7): a ring, not a field
    monkeypatch.setattr(oracle, "_GF343_T3", (1, 1, 0))
    assert not gf343_field_ok(oracle)
    assert not paley344_ok(oracle)
    monkeypatch.undo()
    # the integers mod 343 in place of the field: chi of Z/343 is no character
    monkeypatch.setattr(oracle, "gf343_mul", lambda a, b: (np.asarray(a) * np.asarray(b)) % 343)
    monkeypatch.setattr(oracle, "gf343_sub", lambda a, b: (np.asarray(a) - np.asarray(b)) % 343)
    assert not paley344_ok(oracle)
    monkeypatch.undo()
    # the t^4 reduction dropped (t^4 read as 0)
    real = oracle.gf343_mul

    def no_t4(a, b):
        a0, a1, a2 = oracle.gf343_digits(a)
        b0, b1, b2 = oracle.gf343_digits(b)
        p0, p1, p2, p3 = a0 * b0, a0 * b1 + a1 * b0, a0 * b2 + a1 * b1 + a2 * b0, a1 * b2 + a2 * b1
        return oracle.gf343_index(p0 + 2 * p3, p1, p2)
    monkeypatch.setattr(oracle, "gf343_mul", no_t4)
    assert not gf343_field_ok(oracle)
    monkeypatch.setattr(oracle, "gf343_mul", real)
    assert gf343_field_ok(oracle) and paley344_ok(oracle)


@pytest.mark.parametrize("N,K", [(24, 64), (56, 40), (16, 112), (344, 64), (24, 688)])
def test_rht_layer_undoes_the_weight_rotation(N, K):
    """Eq. (def:hadamard): if W_hat is exactly R(W) = U S_U W S_V V, the layer
    with the inverse transform around it returns x W^T. Checked with a dense W
    expressed through d = 1 codes and A = 1 (so W_hat is an integer matrix and
    R^-1(W_hat) is the W whose product we know)."""
    g = np.random.default_rng(N * K)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    A = np.ones((1, 1))
    B = np.zeros(1)
    s_U = g.choice([-1.0, 1.0], size=N)
    s_V = g.choice([-1.0, 1.0], size=K)
    W_hat = codes.astype(np.float64)
    # W with R(W) = W_hat: W = S_U U^T W_hat V^T S_V
    U = oracle.hadamard(N) / np.sqrt(N)
    V = oracle.hadamard(K) / np.sqrt(K)
    W = s_U[:, None] * (U.T @ W_hat @ V.T) * s_V[None, :]
    assert np.allclose(oracle.rht_weight(W, s_U, s_V), W_hat, atol=1e-12)
    x = g.standard_normal((3, K))
    y, S = oracle.linear_rht(x, codes, A, B, s_U, s_V)
    assert np.allclose(y, x @ W.T, rtol=0, atol=1e-11 * np.abs(x).sum())
    assert np.all(S >= 0)


def test_rht_input_output_are_inverse_rotations():
    g = np.random.default_rng(9)
    K = 448
    s = g.choice([-1.0, 1.0], size=K)
    x = g.standard_normal((2, K))
    xt = oracle.rht_input(x, s)
    assert np.allclose(np.linalg.norm(xt, axis=1), np.linalg.norm(x, axis=1), rtol=1e-13)
    # rht_output applies U then S; with U = V its transpose undoes rht_input
    V = oracle.hadamard(K) / np.sqrt(K)
    assert np.allclose((xt @ V.T) * s, x, atol=1e-12)



# --------------------------------------------------------------------------
# 3-bit codes (Sec. 5.2, Table tab:bitwidth): the lattice {0..7}^d
# --------------------------------------------------------------------------

@pytest.mark.parametrize("d", [1, 2, 4])
def test_enumeration_moments_3bit(d):
    pin_enumeration_moments(oracle.dequant, d, bits=3)


def test_codebook_3bit_is_dequant_of_every_index():
    """`codebook(A, B, bits=3)` row v is the dequantisation of the lattice
    point whose coordinate c is bit-field [3c+2:3c] of v."""
    for d in (1, 2, 4):
        g = np.random.default_rng(30 + d)
        A = g.standard_normal((d, d))
        B = g.standard_normal(d)
        v = np.arange(8 ** d)
        pts = np.stack([(v >> (3 * c)) & 7 for c in range(d)], axis=1).astype(np.uint8)
        cb = oracle.codebook(A, B, bits=3)
        assert cb.shape == (8 ** d, d)
        assert np.allclose(cb, oracle.dequant(pts, A, B), rtol=0, atol=1e-14 * np.abs(cb).max())


def test_3bit_scalar_case_is_uniform_3bit_dequantisation():
    """A = s I, B = -s zp 1 with codes 0..7: every weight is s (q - zp)."""
    g = np.random.default_rng(7)
    s_, zp = 0.03125, 3.5
    codes = g.integers(0, 8, size=(5, 64), dtype=np.uint8)
    W = oracle.dequant(codes, s_ * np.eye(2), -s_ * zp * np.ones(2))
    assert np.array_equal(W, s_ * (codes.astype(np.float64) - zp))


# --------------------------------------------------------------------------
# bf16 widening: every activation of the layer (the X of Eq. def:ptq_loss,
# Sec. 2.1, stored as bfloat16) reaches the oracle through bf16_bits_to_f64
# --------------------------------------------------------------------------

# (bit pattern, value written out by hand from the bfloat16 format: sign bit,
# 8 exponent bits with bias 127, 7 fraction bits)
BF16_CASES = [
    (0x3F80, 1.0),
    (0xBF80, -1.0),
    (0xC0A0, -5.0),                      # 1 10000001 0100000: -(1 + 1/4) * 2^2
    (0x4049, 3.140625),                  # 0 10000000 1001001: (1 + 73/128) * 2
    (0x3F81, 1.0 + 2.0 ** -7),           # the next bf16 above 1
    (0x0080, 2.0 ** -126),               # smallest normal
    (0x0001, 2.0 ** -133),               # smallest subnormal: 2^-126 * 2^-7
    (0x807F, -(127 / 128) * 2.0 ** -126),  # largest negative subnormal
    (0x7F7F, (2.0 - 2.0 ** -7) * 2.0 ** 127),  # largest finite
    (0x7F80, float("inf")),
    (0xFF80, float("-inf")),
    (0x0000, 0.0),
]


def bf16_by_definition(b: int) -> float:
    """IEEE-style bfloat16 value of a 16-bit pattern, from its fields."""
    sign = -1.0 if b >> 15 else 1.0
    e = (b >> 7) & 0xFF
    f = b & 0x7F
    if e == 0xFF:
        return sign * float("inf") if f == 0 else float("nan")
    if e == 0:
        return sign * (f / 128.0) * 2.0 ** -126
    return sign * (1.0 + f / 128.0) * 2.0 ** (e - 127)


def pin_bf16_widening(widen_fn):
    bits = np.array([b for b, _ in BF16_CASES], dtype=np.uint16)
    got = widen_fn(bits)
    for (b, v), g in zip(BF16_CASES, got):
        assert g == v, (hex(b), g, v)
        assert bf16_by_definition(b) == v, hex(b)
    # -0.0 keeps its sign
    z = widen_fn(np.array([0x8000], dtype=np.uint16))[0]
    assert z == 0.0 and np.signbit(z)
    # every finite pattern against the field definition (all 65536 patterns)
    allb = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    w = widen_fn(allb)
    e = (allb.astype(np.int64) >> 7) & 0xFF
    fin = e != 0xFF
    ref = np.array([bf16_by_definition(int(b)) for b in allb[fin][::97]])
    assert np.array_equal(w[fin][::97], ref)
    nan_pat = (e == 0xFF) & ((allb & 0x7F) != 0)
    assert np.all(np.isnan(w[nan_pat]))


def test_bf16_widening_pinned():
    pin_bf16_widening(oracle.bf16_bits_to_f64)


@pytest.mark.parametrize("kind", ["as_fp16", "byteswap", "shift15", "drop_sign"])
def test_bf16_pin_catches_planted_mistakes(kind):
    def widen(bits):
        b = np.ascontiguousarray(bits, dtype=np.uint16)
        if kind == "as_fp16":
            return b.view(np.float16).astype(np.float64)
        if kind == "byteswap":
            b = b.byteswap()
        if kind == "drop_sign":
            b = b & 0x7FFF
        sh = 15 if kind == "shift15" else 16
        return (b.astype(np.uint32) << sh).view(np.float32).astype(np.float64)
    with pytest.raises(AssertionError):
        pin_bf16_widening(widen)
