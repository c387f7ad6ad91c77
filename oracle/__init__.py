"""CPU oracle for the UniSVQ linear layer (TEST INFRASTRUCTURE ONLY).

Plain, slow, fp64 NumPy restatement of what the inference-time UniSVQ linear
layer computes. Only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline
legs of `bench.py` may import it; the product library never does, and this
package imports nothing from the product.

Every function cites the passage of the paper it follows:

* Eq. (def:unisvq), Sec. 3.1 -- one length-d weight vector is the affine image
  A z + B of an integer lattice point z (coordinates in {0,1,2,3} for 2 bits).
* Eq. (col:dequant), Sec. 3.2.3 -- the dequantised W^T stacks, for each group i
  of d input columns, the block A W_int,i^T + B 1^T: the vectors run along the
  input dimension and one (A, B) serves the whole weight matrix.
* Eq. (col:matmul), Sec. 3.2.3 -- Y = X W^T = sum_i (X_i A) W_int,i^T
  + sum_i (X_i B) 1^T (the fold of the affine onto the activations).
* Eq. (def:ptq_loss), Sec. 2.1 -- the layer output is Y = X W^T with X tokens x
  inputs and W outputs x inputs.

`dequant`, `linear` and `linear_folded` take integer codes of any width:
2-bit codes z in {0..3} and the 3-bit variant z in {0..7} (Sec. 5.2, Table
tab:bitwidth: only the integer vectors widen).

Inputs are exactly widened to fp64 (bf16 activations, fp16 affine). Where the
paper fixes no rounding, the oracle keeps everything exact in fp64 and rounds
once at the very end (`dequant_f32`).

The RHT functions (`hadamard`, `rht_weight`, `rht_input`, `rht_output`,
`linear_rht`) restate Eq. (def:hadamard): the weights are rotated before
quantisation, so at inference the activations are rotated on the way in and
the outputs on the way out.

The per-(row, group) functions (`dequant_grouped`, `linear_grouped`,
`linear_grouped_moments`) restate Eq. (def:unisvq) with one (A, B) per output
row and group of input columns; the paper itself uses one per matrix.

Pins (tests/test_oracle_pins.py): exhaustive codebook enumeration with the
orthogonal initial grid (mean 0, covariance I, App. A.1), the scalar
quantisation special case (Eq. def:sq), an integer-matrix case checked against
exact Python integers, the hand-worked example in tests/golden/, linearity in
x, agreement of Eq. (col:dequant) with Eq. (def:unisvq), and the fold
identity of Eq. (col:matmul); for the per-group functions, the hand-worked
example in tests/golden/grouped_hand_worked.json, group-wise uniform scalar
quantisation (A = s I), reduction to the per-matrix oracle when all groups
share one map, and the exchange-of-sums identity; for the RHT functions,
H H^T = n I for every order built, Sylvester's matrix against SciPy's and
against its closed form (-1)^popcount(p & p'), the field axioms of GF(343)
and the multiplicativity of its quadratic character (with planted mistakes
caught: a reducible modulus, the ring Z/343, a dropped reduction term), and
the undo identity: the RHT layer applied to W_hat = R(W) returns x W^T; for the
bf16 widening that every activation passes through, hand-chosen bit patterns
(signed zero, subnormals, the largest finite value, infinities) against the
IEEE bfloat16 definition. No function here is "parity unpinned".
"""
from __future__ import annotations

import numpy as np

# Tolerances for comparing a layer output against the oracle (per element and
# over the whole tensor); see `compare`.
ABS_REL_BOUND = 2.0 ** -7
ABS_FLOOR = 1e-6
REL_L2_BOUND = 4e-3


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    with np.errstate(invalid="ignore"):   # signalling-NaN patterns stay NaN
        return b.view(np.float32).astype(np.float64)


def as_f64(a) -> np.ndarray:
    """Exact widening of fp16 / fp32 / fp64 arrays to float64."""
    return np.asarray(a).astype(np.float64)


def _check(codes: np.ndarray, A: np.ndarray, B: np.ndarray):
    d = A.shape[0]
    if A.shape != (d, d) or B.shape != (d,):
        raise ValueError("A must be d x d and B length d")
    if codes.ndim != 2 or codes.shape[1] % d:
        raise ValueError("codes must be [N][K] with K a multiple of d")
    return d


def codebook(A, B, bits: int = 2) -> np.ndarray:
    """All 2^(bits d) codewords, row v = A z(v) + B with z_c(v) the bit-field
    [bits (c+1) - 1 : bits c] of v.

    Eq. (def:unisvq) evaluated on every point of {0..2^bits - 1}^d (2-bit codes
    by default; 3-bit codes only widen the lattice, Sec. 5.2).
    """
    d = np.asarray(A).shape[0]
    v = np.arange(2 ** (bits * d))
    mask = (1 << bits) - 1
    Z = np.stack([(v >> (bits * c)) & mask for c in range(d)], axis=1).astype(np.float64)
    return Z @ as_f64(A).T + as_f64(B)


def dequant(codes: np.ndarray, A, B) -> np.ndarray:
    """Dequantised weights W_hat [N][K] in fp64.

    Eq. (def:unisvq) applied to every vector: for output row n and input group
    g (columns g*d .. g*d+d-1), W_hat[n, g*d + r] = sum_c A[r, c] z[n, g*d + c]
    + B[r], the column-vector form of the blocks of Eq. (col:dequant).
    """
    d = _check(codes, np.asarray(A), np.asarray(B))
    N, K = codes.shape
    Z = codes.reshape(N, K // d, d).astype(np.float64)
    W = Z @ as_f64(A).T + as_f64(B)
    return W.reshape(N, K)


def dequant_f32(codes: np.ndarray, A, B) -> np.ndarray:
    """RN-to-fp32 of the exact fp64 dequantised weights (a single rounding)."""
    return dequant(codes, A, B).astype(np.float32)


def linear(x: np.ndarray, codes: np.ndarray, A, B, row_chunk: int = 4096):
    """Layer output y = x W_hat^T and the tolerance scale S = |x| |W_hat|^T.

    Eq. (def:ptq_loss): Y = X W^T with X [M][K] and W [N][K]. `x` is either
    bf16 bits (uint16) or a float array. Rows of W are dequantised in chunks so
    large layers never hold a full fp64 W.
    Returns (y, S), both float64 [M][N].
    """
    xf = bf16_bits_to_f64(x) if x.dtype == np.uint16 else as_f64(x)
    M = xf.shape[0]
    N = codes.shape[0]
    y = np.empty((M, N))
    S = np.empty((M, N))
    ax = np.abs(xf)
    for r0 in range(0, N, row_chunk):
        W = dequant(codes[r0:r0 + row_chunk], A, B)
        y[:, r0:r0 + W.shape[0]] = xf @ W.T
        S[:, r0:r0 + W.shape[0]] = ax @ np.abs(W).T
    return y, S


def linear_folded(x: np.ndarray, codes: np.ndarray, A, B) -> np.ndarray:
    """Eq. (col:matmul): y = sum_i (X_i A) W_int,i^T + sum_i (X_i B) 1^T.

    X_i is the [M][d] slice of inputs i*d .. i*d+d-1 and W_int,i the matching
    [N][d] slice of the integer codes. fp64 throughout.
    """
    d = _check(codes, np.asarray(A), np.asarray(B))
    xf = bf16_bits_to_f64(x) if x.dtype == np.uint16 else as_f64(x)
    M, K = xf.shape
    Xi = xf.reshape(M, K // d, d)
    XA = (Xi @ as_f64(A)).reshape(M, K)          # the row vectors X_i A
    XB = (Xi @ as_f64(B)).sum(axis=1)            # sum_i X_i B, one scalar per token
    return XA @ codes.astype(np.float64).T + XB[:, None]


def _check_grouped(codes: np.ndarray, A: np.ndarray, B: np.ndarray, group_cols: int):
    N, K = codes.shape
    d = A.shape[-1]
    G = -(-K // group_cols)
    if A.shape != (N, G, d, d) or B.shape != (N, G, d):
        raise ValueError("A must be [N][G][d][d] and B [N][G][d], G = ceil(K / group_cols)")
    if K % d or group_cols % d:
        raise ValueError("K and group_cols must be multiples of d")
    return N, K, d, G


def dequant_grouped(codes: np.ndarray, A, B, group_cols: int = 128) -> np.ndarray:
    """Dequantised weights [N][K] in fp64 with one affine map per (output row,
    group of `group_cols` input columns).

    Eq. (def:unisvq) applied to every vector, each with the (A, B) of its own
    row n and column group g = k // group_cols (per-row, per-group granularity,
    finer than the paper's one map per matrix). A is [N][G][d][d], B [N][G][d],
    G = ceil(K / group_cols); group_cols is a multiple of d, so a vector never
    straddles two groups: W_hat[n, k] = sum_c A[n, g, r, c] z[n, k - r + c]
    + B[n, g, r] with r = k mod d.
    """
    A = as_f64(A)
    B = as_f64(B)
    N, K, d, G = _check_grouped(codes, A, B, group_cols)
    Z = codes.reshape(N, K // d, d).astype(np.float64)
    g_of_vec = (np.arange(K // d) * d) // group_cols          # group of each vector
    W = np.einsum("nvrc,nvc->nvr", A[:, g_of_vec], Z) + B[:, g_of_vec]
    return W.reshape(N, K)


def linear_grouped(x: np.ndarray, codes: np.ndarray, A, B, group_cols: int = 128, row_chunk: int = 256):
    """Layer output y = x W_hat^T and tolerance scale S = |x| |W_hat|^T for
    per-(row, group) affine maps (`dequant_grouped`); Eq. (def:ptq_loss).
    Returns (y, S), both float64 [M][N].
    """
    xf = bf16_bits_to_f64(x) if x.dtype == np.uint16 else as_f64(x)
    A = np.asarray(A)
    B = np.asarray(B)
    M = xf.shape[0]
    N = codes.shape[0]
    y = np.empty((M, N))
    S = np.empty((M, N))
    ax = np.abs(xf)
    for r0 in range(0, N, row_chunk):
        r1 = min(N, r0 + row_chunk)
        W = dequant_grouped(codes[r0:r1], A[r0:r1], B[r0:r1], group_cols)
        y[:, r0:r1] = xf @ W.T
        S[:, r0:r1] = ax @ np.abs(W).T
    return y, S


def linear_grouped_moments(x: np.ndarray, codes: np.ndarray, A, B, group_cols: int = 128) -> np.ndarray:
    """The same output contracted before the affine map is applied: for row n
    and group g, S_rc = sum_v x[v d + r] z[n, v d + c] over the group's
    vectors v and X_r = sum_v x[v d + r]; then
    y[n] = sum_g sum_{r,c} A[n, g, r, c] S_rc + sum_g sum_r B[n, g, r] X_r.

    This is Eq. (def:unisvq) summed over a group with the order of the sums
    exchanged (x_v . (A z_v + B) = sum_{r,c} A_rc x_vr z_vc + sum_r B_r x_vr),
    the form in which the codes meet the activations before A does. fp64.
    """
    A = as_f64(A)
    B = as_f64(B)
    xf = bf16_bits_to_f64(x) if x.dtype == np.uint16 else as_f64(x)
    N, K, d, G = _check_grouped(codes, A, B, group_cols)
    M = xf.shape[0]
    y = np.zeros((M, N))
    for g in range(G):
        k0, k1 = g * group_cols, min(K, (g + 1) * group_cols)
        xg = xf[:, k0:k1].reshape(M, -1, d)                   # [M][V][r]
        zg = codes[:, k0:k1].reshape(N, -1, d).astype(np.float64)   # [N][V][c]
        Smom = np.einsum("mvr,nvc->mnrc", xg, zg)
        X = xg.sum(axis=1)                                    # [M][r]
        y += np.einsum("mnrc,nrc->mn", Smom, A[:, g]) + X @ B[:, g].T
    return y


# ---------------------------------------------------------------------------
# Randomized Hadamard transform around the layer, Eq. (def:hadamard), Sec. 3.2.1
# ---------------------------------------------------------------------------

def _quadratic_character(q: int) -> np.ndarray:
    """chi(a) for a in 0..q-1, q prime: 0 at 0, +1 on quadratic residues, -1 otherwise."""
    chi = -np.ones(q, dtype=np.int64)
    chi[0] = 0
    chi[(np.arange(1, q) ** 2) % q] = 1
    return chi


# GF(343) = GF(7)[t] / (t^3 - c(t)): t^3 is replaced by the coefficients below
# (c0, c1, c2), here t^3 = 2. t^3 - 2 is irreducible over GF(7) because it has
# no root there (2 is not a cube mod 7), so the quotient is a field.
_GF343_T3 = (2, 0, 0)


def gf343_digits(e):
    """Element e in 0..342 of GF(343) as its coefficients (c0, c1, c2) of
    c0 + c1 t + c2 t^2, with e = c0 + 7 c1 + 49 c2 (works elementwise on arrays)."""
    e = np.asarray(e)
    return e % 7, (e // 7) % 7, e // 49


def gf343_index(c0, c1, c2):
    return (np.asarray(c0) % 7) + 7 * (np.asarray(c1) % 7) + 49 * (np.asarray(c2) % 7)


def gf343_sub(a, b):
    """a - b in GF(343): coefficient-wise mod 7."""
    a0, a1, a2 = gf343_digits(a)
    b0, b1, b2 = gf343_digits(b)
    return gf343_index(a0 - b0, a1 - b1, a2 - b2)


def gf343_mul(a, b):
    """a b in GF(343): the polynomial product, with t^3 and t^4 = t t^3 reduced
    through _GF343_T3."""
    a = gf343_digits(a)
    b = gf343_digits(b)
    p = [0, 0, 0, 0, 0]
    for i in range(3):
        for j in range(3):
            p[i + j] = p[i + j] + a[i] * b[j]
    r0, r1, r2 = _GF343_T3
    # t^3 = r0 + r1 t + r2 t^2; t^4 = r0 t + r1 t^2 + r2 t^3
    c = [p[0], p[1], p[2]]
    t4 = [0, r0, r1]            # t^4 without its t^3 term r2 t^3
    for k in range(3):
        c[k] = c[k] + p[3] * (r0, r1, r2)[k] + p[4] * t4[k]
    c = [c[k] + p[4] * r2 * (r0, r1, r2)[k] for k in range(3)]
    return gf343_index(c[0], c[1], c[2])


def gf343_quadratic_character() -> np.ndarray:
    """chi(e) for e in 0..342: 0 at 0, +1 on the nonzero squares of GF(343), -1 otherwise."""
    e = np.arange(1, 343)
    chi = -np.ones(343, dtype=np.int64)
    chi[0] = 0
    chi[gf343_mul(e, e)] = 1
    return chi


def paley_hadamard(m: int) -> np.ndarray:
    """A +-1 Hadamard matrix of order m in {12, 20, 28, 344} (Paley's constructions).

    Order q + 1 with q = 11, 19 (prime) or 343 = 7^3 (q = 3 mod 4): with the
    Jacobsthal matrix Q[i][j] = chi(e_j - e_i) over the field of order q (for
    343, e_i is the field element of index i, `gf343_digits`),
    H = I + [[0, 1^T], [-1, Q]].
    Order 2(q + 1) with q = 13 (q = 1 mod 4, prime): with the symmetric
    conference matrix C = [[0, 1^T], [1, Q]], H = [[C + I, C - I], [C - I, -C - I]].
    """
    if m in (12, 20, 344):
        q = m - 1
        idx = np.arange(q)
        if q == 343:
            Q = gf343_quadratic_character()[gf343_sub(idx[None, :], idx[:, None])]
        else:
            Q = _quadratic_character(q)[(idx[None, :] - idx[:, None]) % q]
        S = np.zeros((m, m), dtype=np.int64)
        S[0, 1:] = 1
        S[1:, 0] = -1
        S[1:, 1:] = Q
        return np.eye(m, dtype=np.int64) + S
    if m == 28:
        q = 13
        chi = _quadratic_character(q)
        Q = chi[(np.arange(q)[None, :] - np.arange(q)[:, None]) % q]
        C = np.zeros((q + 1, q + 1), dtype=np.int64)
        C[0, 1:] = 1
        C[1:, 0] = 1
        C[1:, 1:] = Q
        I = np.eye(q + 1, dtype=np.int64)
        return np.block([[C + I, C - I], [C - I, -C - I]])
    raise ValueError("Paley order must be 12, 20, 28 or 344")


def hadamard_factor(n: int):
    """(2^a, m) with n = 2^a m and m in {1, 12, 20, 28, 344} (the largest such m), or None."""
    for m in (344, 28, 20, 12, 1):
        if n % m == 0:
            p = n // m
            if p & (p - 1) == 0:
                return p, m
    return None


def hadamard(n: int) -> np.ndarray:
    """+-1 Hadamard matrix of order n = 2^a m: Sylvester's H_{2^a} (H_1 = [1],
    H_{2k} = [[H_k, H_k], [H_k, -H_k]]) Kronecker H_m (Paley, m > 1), so entry
    [(p, q), (p', q')] at index p m + q is H_{2^a}[p][p'] H_m[q][q']."""
    f = hadamard_factor(n)
    if f is None:
        raise ValueError(f"no Hadamard matrix of order {n} is built (n = 2^a m, m in 1, 12, 20, 28, 344)")
    p, m = f
    H = np.ones((1, 1), dtype=np.int64)
    while H.shape[0] < p:
        H = np.block([[H, H], [H, -H]])
    return H if m == 1 else np.kron(H, paley_hadamard(m))


def rht_weight(W: np.ndarray, s_U, s_V) -> np.ndarray:
    """Eq. (def:hadamard): R(W) = U S_U W S_V V with U = H_N / sqrt(N), V = H_K / sqrt(K)
    (orthogonal) and S_U, S_V the diagonal +-1 matrices of the sign vectors. fp64."""
    W = as_f64(W)
    N, K = W.shape
    U = hadamard(N) / np.sqrt(N)
    V = hadamard(K) / np.sqrt(K)
    return U @ (as_f64(s_U)[:, None] * W * as_f64(s_V)[None, :]) @ V


def rht_input(x: np.ndarray, s_V) -> np.ndarray:
    """The activations the quantised R(W) multiplies: x S_V V (row vectors). fp64."""
    xf = bf16_bits_to_f64(x) if x.dtype == np.uint16 else as_f64(x)
    K = xf.shape[1]
    return (xf * as_f64(s_V)[None, :]) @ (hadamard(K) / np.sqrt(K))


def rht_output(yt: np.ndarray, s_U) -> np.ndarray:
    """The layer output from that of R(W): yt U S_U (row vectors). fp64."""
    yt = as_f64(yt)
    N = yt.shape[1]
    return (yt @ (hadamard(N) / np.sqrt(N))) * as_f64(s_U)[None, :]


def linear_rht(x: np.ndarray, codes: np.ndarray, A, B, s_U, s_V, row_chunk: int = 4096):
    """y = x W^T for W = S_U U^T W_hat V^T S_V, the weight whose RHT (Eq.
    def:hadamard) was quantised to W_hat: y = ((x S_V V) W_hat^T) U S_U.

    Returns (y, S) with S = S_t |U|: S_t = |x S_V V| |W_hat|^T bounds the error
    of the inner layer element by element, and the output transform mixes those
    bounds with weights |U| = 1 / sqrt(N).
    """
    xt = rht_input(x, s_V)
    yt, St = linear(xt, codes, A, B, row_chunk)
    N = codes.shape[0]
    return rht_output(yt, s_U), St @ (np.abs(hadamard(N)) / np.sqrt(N))


def compare(y: np.ndarray, y_ref: np.ndarray, S: np.ndarray) -> dict:
    """Check a layer output against the oracle.

    Per element |y - y_ref| <= 2^-7 * S + 1e-6 (S = sum_k |W_hat x|), and the
    relative L2 error over the tensor must not exceed 4e-3.
    """
    y = np.asarray(y, dtype=np.float64)
    err = np.abs(y - y_ref)
    bound = ABS_REL_BOUND * S + ABS_FLOOR
    ratio = np.max(err / bound) if err.size else 0.0
    nref = np.linalg.norm(y_ref)
    rel_l2 = float(np.linalg.norm(y - y_ref) / nref) if nref > 0 else float(np.linalg.norm(y - y_ref))
    finite = bool(np.all(np.isfinite(y)))
    return {
        "max_err_over_bound": float(ratio),
        "rel_l2": rel_l2,
        "finite": finite,
        "ok": finite and ratio <= 1.0 and rel_l2 <= REL_L2_BOUND,
    }
