"""Host-side tests of libunisvq that need no GPU: exports, layout, validation."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "unisvq.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(unisvq_[a-z_0-9]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert "unisvq_linear" in names and "unisvq_pack" in names
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/unisvq.h but not exported"
    from paper_2606_10520_gb300 import binding
    assert sorted(binding.EXPORTS) == names


def decode_layout(packed: np.ndarray, N: int, K: int) -> np.ndarray:
    """Independent reader of the packed layout, written from include/unisvq.h."""
    Np = -(-N // 128) * 128
    Kp = -(-K // 128) * 128
    KT = Kp // 128
    # word (rb, kt, u, g, t, slot) with slot = 2h + q holds row 128rb + 16u + 8q + g
    words = packed.view("<u4").reshape(Np // 128, KT, 8, 8, 4, 4)
    out = np.full((Np, Kp), 255, dtype=np.int64)
    for rb in range(Np // 128):
        for kt in range(KT):
            for u in range(8):
                for g in range(8):
                    for t in range(4):
                        for slot in range(4):
                            h, q = slot >> 1, slot & 1
                            r = 128 * rb + 16 * u + 8 * q + g
                            w = int(words[rb, kt, u, g, t, slot])
                            for s in range(4):
                                for b in range(4):
                                    k = 128 * kt + 64 * h + 16 * t + 4 * s + b
                                    out[r, k] = (w >> (8 * b + 2 * s)) & 3
    return out


@pytest.mark.parametrize("N,K", [(16, 128), (37, 200), (130, 260), (8, 4)])
def test_pack_host_layout_roundtrip(lib, N, K):
    from paper_2606_10520_gb300 import binding
    g = np.random.default_rng(N * 1000 + K)
    codes = g.integers(0, 4, size=(N, K), dtype=np.uint8)
    packed = binding.pack_host(codes)
    assert packed.nbytes == binding.packed_code_bytes(N, K)
    assert packed.nbytes == (-(-N // 128)) * (-(-K // 128)) * 4096
    full = decode_layout(packed, N, K)
    assert not (full == 255).any(), "some (row, col) never written"
    assert np.array_equal(full[:N, :K], codes)
    assert (full[N:, :] == 0).all() and (full[:, K:] == 0).all(), "padding must be code 0"


def test_packed_bytes_is_quarter_byte_per_weight(lib):
    from paper_2606_10520_gb300 import binding
    for N, K in [(4096, 4096), (11008, 4096), (28672, 8192)]:
        assert binding.packed_code_bytes(N, K) == N * K // 4


def test_status_strings(lib):
    from paper_2606_10520_gb300 import binding
    for s in range(6):
        assert isinstance(binding.status_string(s), str) and binding.status_string(s)


def _pack_status(lib, codes, A, B, N, K, d):
    h = ctypes.c_void_p()
    return lib.unisvq_pack(codes.ctypes.data if codes is not None else None,
                           A.ctypes.data if A is not None else None,
                           B.ctypes.data if B is not None else None, N, K, d, None, ctypes.byref(h))


def test_pack_rejects_bad_arguments_before_touching_the_gpu(lib):
    from paper_2606_10520_gb300 import binding
    codes = np.zeros((4, 8), dtype=np.uint8)
    A = np.eye(2, dtype=np.float16).view(np.uint16)
    B = np.zeros(2, dtype=np.float16).view(np.uint16)
    assert _pack_status(lib, None, A, B, 4, 8, 2) == binding.ERR_INVALID_ARG
    assert _pack_status(lib, codes, A, B, 4, 8, 3) == binding.ERR_UNSUPPORTED
    assert _pack_status(lib, codes, A, B, 4, 7, 2) == binding.ERR_INVALID_ARG     # K % d
    assert _pack_status(lib, codes, A, B, 0, 8, 2) == binding.ERR_INVALID_ARG
    bad = codes.copy()
    bad[1, 3] = 4
    assert _pack_status(lib, bad, A, B, 4, 8, 2) == binding.ERR_INVALID_ARG
    Anan = np.array([[np.nan, 0], [0, 1]], dtype=np.float16).view(np.uint16)
    assert _pack_status(lib, codes, Anan, B, 4, 8, 2) == binding.ERR_INVALID_ARG


def test_pack_takes_the_paper_vector_lengths_only(lib):
    """d in {1, 2, 4, 8}: the lengths the paper evaluates (d = 8 in its vector
    length ablation); anything else is UNSUPPORTED, and K must be a multiple of d."""
    from paper_2606_10520_gb300 import binding
    codes = np.zeros((4, 24), dtype=np.uint8)
    A8 = np.eye(8, dtype=np.float16).view(np.uint16)
    B8 = np.zeros(8, dtype=np.float16).view(np.uint16)
    A8nan = A8.copy()
    A8nan[7, 7] = np.array([np.inf], dtype=np.float16).view(np.uint16)[0]
    for d in (3, 5, 6, 16):
        assert _pack_status(lib, codes, A8, B8, 4, 24, d) == binding.ERR_UNSUPPORTED
    assert _pack_status(lib, codes, A8, B8, 4, 20, 8) == binding.ERR_INVALID_ARG      # K % 8
    assert _pack_status(lib, codes, A8nan, B8, 4, 24, 8) == binding.ERR_INVALID_ARG   # A[7][7] = inf


def test_linear_rejects_bad_arguments(lib):
    from paper_2606_10520_gb300 import binding
    assert lib.unisvq_linear(None, None, None, 1, None) == binding.ERR_INVALID_ARG
    assert lib.unisvq_destroy(None) == binding.OK
    info = binding.Info()
    assert lib.unisvq_query(None, 1, ctypes.byref(info)) == binding.ERR_INVALID_ARG
    hs = (ctypes.c_void_p * 2)(None, None)
    ys = (ctypes.c_void_p * 2)(None, None)
    assert lib.unisvq_linear_group(None, 1, None, ys, 1, None) == binding.ERR_INVALID_ARG
    assert lib.unisvq_linear_group(hs, 0, None, ys, 1, None) == binding.ERR_INVALID_ARG
    assert lib.unisvq_linear_group(hs, binding.MAX_GROUP + 1, None, ys, 1, None) == binding.ERR_INVALID_ARG
    assert lib.unisvq_linear_group(hs, 2, None, ys, 1, None) == binding.ERR_INVALID_ARG   # null handles


def test_version(lib):
    assert lib.unisvq_version() >= 100


def _pack_grouped_status(lib, codes, A, B, N, K, d, gc):
    h = ctypes.c_void_p()
    return lib.unisvq_pack_grouped(codes.ctypes.data if codes is not None else None,
                                   A.ctypes.data if A is not None else None,
                                   B.ctypes.data if B is not None else None, N, K, d, gc, None, ctypes.byref(h))


def test_pack_grouped_rejects_bad_arguments_before_touching_the_gpu(lib):
    from paper_2606_10520_gb300 import binding
    N, K, d = 4, 256, 2
    G = K // 128
    codes = np.zeros((N, K), dtype=np.uint8)
    A = np.zeros((N, G, d, d), dtype=np.float16).view(np.uint16)
    B = np.zeros((N, G, d), dtype=np.float16).view(np.uint16)
    assert _pack_grouped_status(lib, None, A, B, N, K, d, 128) == binding.ERR_INVALID_ARG
    assert _pack_grouped_status(lib, codes, A, B, N, K, 3, 128) == binding.ERR_UNSUPPORTED
    assert _pack_grouped_status(lib, codes, A, B, N, K, d, 64) == binding.ERR_UNSUPPORTED
    assert _pack_grouped_status(lib, codes, A, B, N, 255, d, 128) == binding.ERR_INVALID_ARG   # K % d
    bad = codes.copy()
    bad[2, 100] = 7
    assert _pack_grouped_status(lib, bad, A, B, N, K, d, 128) == binding.ERR_INVALID_ARG
    Ainf = A.copy()
    Ainf[3, 1, 1, 0] = np.array([np.inf], dtype=np.float16).view(np.uint16)[0]
    assert _pack_grouped_status(lib, codes, Ainf, B, N, K, d, 128) == binding.ERR_INVALID_ARG
    Bnan = B.copy()
    Bnan[0, 0, 1] = np.array([np.nan], dtype=np.float16).view(np.uint16)[0]
    assert _pack_grouped_status(lib, codes, A, Bnan, N, K, d, 128) == binding.ERR_INVALID_ARG


def test_pack_bits_rejects_bad_widths_and_codes(lib):
    from paper_2606_10520_gb300 import binding
    codes = np.zeros((4, 16), dtype=np.uint8)
    A = np.eye(2, dtype=np.float16).view(np.uint16)
    B = np.zeros(2, dtype=np.float16).view(np.uint16)
    A8 = np.eye(8, dtype=np.float16).view(np.uint16)
    B8 = np.zeros(8, dtype=np.float16).view(np.uint16)
    h = ctypes.c_void_p()
    st = lambda c, a, b, d, bits: lib.unisvq_pack_bits(c.ctypes.data, a.ctypes.data, b.ctypes.data, 4, 16, d, bits,
                                                        None, ctypes.byref(h))
    assert st(codes, A, B, 2, 4) == binding.ERR_UNSUPPORTED
    assert st(codes, A, B, 2, 1) == binding.ERR_UNSUPPORTED
    assert st(codes, A8, B8, 8, 3) == binding.ERR_UNSUPPORTED      # 8^8 codewords
    bad = codes.copy()
    bad[1, 5] = 8
    assert st(bad, A, B, 2, 3) == binding.ERR_INVALID_ARG          # code >= 2^3
    bad[1, 5] = 4
    assert st(bad, A, B, 2, 2) == binding.ERR_INVALID_ARG          # code >= 2^2


# ---------------------------------------------------------------------------
# Prefill tables (unisvq_prefill_table_host), rebuilt independently: exact
# fp64 codewords, rounded once to bf16 (round to nearest even, written here)
# or fp32 (numpy's conversion), in the word layout include/unisvq.h states.
# ---------------------------------------------------------------------------

def _bf16_rne_bits(x):
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                         # x = m 2^e, 0.5 <= |m| < 1
    y = np.ldexp(np.rint(m * 256.0), e - 8)    # 8 significant bits, ties to even
    return (y.astype(np.float32).view(np.uint32) >> 16).astype(np.uint32)


def _f32_bits(x):
    return np.asarray(x, dtype=np.float64).astype(np.float32).view(np.uint32)


def _expected_table(A, B, d, bits):
    A = A.astype(np.float64)
    B = B.astype(np.float64)
    zmax = (1 << bits) - 1

    def cw(z):   # z [..., d] -> A z + B, exact in fp64
        return np.asarray(z, dtype=np.float64) @ A.T + B

    if d <= 2:
        n = 1 << (2 * bits)
        v = np.arange(n)
        lo, hi = v & zmax, v >> bits
        if d == 2:
            w = cw(np.stack([lo, hi], axis=-1))
            w0, w1 = w[:, 0], w[:, 1]
        else:
            w0, w1 = cw(lo[:, None])[:, 0], cw(hi[:, None])[:, 0]
        return _bf16_rne_bits(w0) | (_bf16_rne_bits(w1) << 16)
    if d == 4 and bits == 2:
        v = np.arange(256)
        w = cw(np.stack([(v >> (2 * c)) & 3 for c in range(4)], axis=-1))
        t = np.zeros(512, dtype=np.uint32)
        t[0::2] = _bf16_rne_bits(w[:, 0]) | (_bf16_rne_bits(w[:, 1]) << 16)
        t[1::2] = _bf16_rne_bits(w[:, 2]) | (_bf16_rne_bits(w[:, 3]) << 16)
        return t
    if d == 4 and bits == 3:
        t = np.zeros(512, dtype=np.uint32)
        for p in range(2):
            for v in range(64):
                for r in range(4):
                    val = A[r, 2 * p] * (v & 7) + A[r, 2 * p + 1] * (v >> 3) + (B[r] if p == 0 else 0.0)
                    t[256 * p + 4 * v + r] = _f32_bits(val)
        return t
    t = np.zeros(4096, dtype=np.uint32)   # d = 8, bits = 2
    for q in range(2):
        for v in range(256):
            z = np.array([(v >> (2 * c)) & 3 for c in range(4)], dtype=np.float64)
            for r in range(8):
                val = A[r, 4 * q:4 * q + 4] @ z + (B[r] if q == 0 else 0.0)
                h = (r // 4) ^ ((v >> 2) & 1)
                t[2048 * q + 8 * v + 4 * h + r % 4] = _f32_bits(val)
    return t


@pytest.mark.parametrize("d,bits", [(1, 2), (2, 2), (4, 2), (8, 2), (1, 3), (2, 3), (4, 3)])
def test_prefill_tables_match_an_independent_build(lib, d, bits):
    from paper_2606_10520_gb300 import binding
    g = np.random.default_rng(100 * d + bits)
    for trial in range(3):
        A = (g.standard_normal((d, d)) * (0.5 if trial else 3.0)).astype(np.float16)
        B = g.standard_normal(d).astype(np.float16)
        got = binding.prefill_table_host(A, B, d, bits)
        want = _expected_table(A, B, d, bits)
        assert got.shape == want.shape
        assert np.array_equal(got, want), (d, bits, np.flatnonzero(got != want)[:8])


def test_prefill_table_rejects_bad_arguments(lib):
    from paper_2606_10520_gb300 import binding
    A = np.ascontiguousarray(np.eye(4, dtype=np.float16).reshape(-1)).view(np.uint16)
    B = np.zeros(4, dtype=np.float16).view(np.uint16)
    w = ctypes.c_size_t(0)
    call = lambda d, bits, a=A: lib.unisvq_prefill_table_host(a.ctypes.data, B.ctypes.data, d, bits, None, 0,
                                                              ctypes.byref(w))
    assert call(4, 2) == binding.OK and w.value == 512
    for d, bits in ((3, 2), (4, 4), (8, 3), (0, 2)):
        assert call(d, bits) == binding.ERR_INVALID_ARG
    bad = A.copy()
    bad[5] = 0x7E00   # fp16 NaN
    assert call(4, 2, bad) == binding.ERR_INVALID_ARG
    out = np.zeros(8, dtype=np.uint32)
    assert lib.unisvq_prefill_table_host(A.ctypes.data, B.ctypes.data, 4, 2, out.ctypes.data, out.size,
                                         ctypes.byref(w)) == binding.ERR_INVALID_ARG   # too small
