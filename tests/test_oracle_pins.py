"""Pins of the oracle against things other than itself (CPU only).

Each test checks one oracle function against the paper's printed numbers, a
published test vector, a library routine (numpy / scipy), brute force on small
inputs, or an invariant the paper states -- chosen so that a dropped term, a
wrong sign or index, or a transposed operand in the oracle fails one of them.
"""
import math
import os

import numpy as np
import pytest
import scipy.linalg

import gen
import oracle
from oracle import accounting as acc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
D = 128


def _golden(name):
    out = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            parts = line.split()
            out[parts[0]] = float(parts[1]) if len(parts) > 1 else parts[0]
    return out


# ---- scalar helpers ----------------------------------------------------------

def test_splitmix64_published_vector():
    want = [int(l, 16) for l in open(os.path.join(GOLDEN, "splitmix64_seed0.txt")) if l.startswith("0x")]
    gamma = 0x9E3779B97F4A7C15
    got = [oracle.splitmix64((n * gamma) & (2**64 - 1)) for n in range(3)]
    assert got == want


def test_fp16_from_double_matches_numpy():
    rng = np.random.default_rng(1)
    xs = np.concatenate([
        rng.standard_normal(20000) * 10.0 ** rng.integers(-9, 5, 20000),
        np.array([0.0, -0.0, 1.0, 1 + 2**-11, 1 + 3 * 2**-11, 2**-24, 2**-25, 2**-25 * (1 + 2**-30), 3 * 2**-26,
                  2**-14, 2**-14 - 2**-25, 65504.0 - 1e-9, 65503.0, 65519.99, -65519.0, 1e-30, 6.1e-5]),
    ])
    xs = xs[np.abs(xs) < 65520]
    want = xs.astype(np.float16).view(np.uint16)
    got = np.array([oracle.fp16_from_double(x) for x in xs], np.uint16)
    assert np.array_equal(got, want)
    # saturation (D4 reading): beyond the fp16 range the oracle clamps to +-65504
    assert oracle.fp16_from_double(1e9) == 0x7BFF and oracle.fp16_from_double(-70000.0) == 0xFBFF


def test_fp16_and_bf16_decoding_match_numpy():
    h = np.arange(65536, dtype=np.uint16)
    f = h.view(np.float16).astype(np.float64)
    ok = np.isfinite(f)
    got = np.array([oracle.fp16_to_double(int(x)) for x in h[ok][::7]])
    assert np.array_equal(got, f[ok][::7])
    b = np.arange(0, 65536, 13, dtype=np.uint16)
    b = b[(b & 0x7F80) != 0x7F80]  # drop inf / NaN patterns
    fb = (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    ok = np.isfinite(fb)
    got = np.array([oracle.bf16_to_double(int(x)) for x in b[ok]])
    assert np.array_equal(got, fb[ok])


def test_wht_is_sylvester_hadamard():
    H = scipy.linalg.hadamard(D).astype(np.float64)
    rng = np.random.default_rng(2)
    for _ in range(5):
        v = rng.integers(-1000, 1000, D).astype(np.float64)  # integer sums: exact in both
        assert np.array_equal(oracle.wht128(v), H @ v)
        assert np.array_equal(oracle.wht128(oracle.wht128(v)), D * v)  # H H = D I
    e0 = np.zeros(D)
    e0[0] = 1.0
    assert np.array_equal(oracle.wht128(np.ones(D)), D * e0)  # H 1 = D e_0


def test_signs_are_a_pm1_pattern_of_both_signs():
    s = oracle.signs(11)
    assert set(np.unique(s)) == {-1.0, 1.0}
    assert not np.array_equal(s, oracle.signs(12))


# ---- shapes and byte accounting (Appendix A.1 worked example, Eq. 9, Eq. 11) -

def test_paper_worked_example():
    g = _golden("paper_worked_example.txt")
    S, Dg, H, W, k = int(g["S"]), int(g["D"]), int(g["H"]), int(g["W"]), int(g["k"])
    assert k == S // 128  # k = S/128 (Section 4.1)
    m_full = acc.paper_m_full(S, H, Dg)
    m_base = acc.paper_m_base(S, H, Dg, W, k, int(g["b_a"]), int(g["b_gamma"]))
    assert round(m_full / 1e6, 1) == g["m_full_mb"]
    assert round(m_base / 1e6, 2) == g["m_base_mb"]
    assert round(100 * m_base / m_full, 1) == g["m_base_pct"]
    remaining = g["theta"] * m_full - m_base
    assert round(remaining / 1e6, 2) == g["remaining_mb"]
    P = S - W
    assert 2 * H * P == int(g["token_sides"])
    # The printed N follows from Eq. 9 with the mean of the two residual costs
    # c_K = D/4 + 4 and c_V = D/4 + 5 (reading R11 of the byte accounting) ...
    b_res = (acc.paper_c_k(Dg) + acc.paper_c_v(Dg)) / 2
    N = acc.paper_n_residuals(g["theta"], m_full, m_base, b_res)
    assert N == int(g["n_residuals"])
    # ... and it is also the largest N whose split floor(N/2) keys + rest values fits.
    nk, nv = acc.paper_split(N)
    assert nk * acc.paper_c_k(Dg) + nv * acc.paper_c_v(Dg) <= remaining
    nk2, nv2 = acc.paper_split(N + 1)
    assert nk2 * acc.paper_c_k(Dg) + nv2 * acc.paper_c_v(Dg) > remaining
    # Appendix E.1 quotes 17.3 % residual density at this operating point.
    dens = 100 * N / (2 * H * P)
    assert math.floor(dens * 10) / 10 == g["density_pct"]


def test_unit_shape_formula():
    # anchors 2 % incl. the window (k = 82 for the 4096-token case), 10 % residual slots
    assert oracle.unit_shape(4096, 0.02, 0.1, 0.1, 32) == (82, 409, 409)
    assert oracle.unit_shape(32768, 0.02, 0.1, 0.1, 32) == (656, 3276, 3276)
    assert oracle.unit_shape(131072, 0.02, 0.1, 0.1, 32) == (2622, 13107, 13107)
    assert oracle.unit_shape(20, 0.02, 0.1, 0.1, 32) == (20, 0, 0)  # S < W: all anchors
    assert oracle.unit_shape(100, 0.02, 1.0, 0.5, 32) == (32, 68, 50)  # slots capped at S - k


def test_format_bytes_ratio_near_20x():
    for S in (4096, 32768, 131072):
        k, nk, nv = oracle.unit_shape(S, 0.02, 0.1, 0.1, 32)
        b = acc.decode_read_bytes(S, k, nk, nv, G=0)
        assert 19.5 < 512 * S / b < 20.2


# ---- quantizer: hand-computed examples ----------------------------------------

def _pack(codes):
    out = np.zeros(32, np.uint8)
    for j, c in enumerate(codes):
        out[j // 4] |= np.uint8(c << (2 * (j % 4)))
    return out


def test_quantizer_without_rotation_hand_example():
    # r = (-1, 0, 1, 2, -1, 0, 1, 2, ...): min = -1, scale = (2 - (-1)) / 3 = 1, code = r + 1
    r = np.tile([-1.0, 0.0, 1.0, 2.0], D // 4)
    codes, sc, mn = oracle.quantize_residual(r, rot_seed=5, rotate=False)
    assert sc == 0x3C00 and mn == 0xBC00  # fp16(1.0), fp16(-1.0)
    assert np.array_equal(codes, _pack([0, 1, 2, 3] * (D // 4)))
    # byte 0 holds codes of coordinates 0..3 in bits 0-1, 2-3, 4-5, 6-7
    assert codes[0] == 0b11100100


def test_quantizer_with_rotation_recovers_designed_codes():
    # Design the rotated vector v* = min + c * scale with min = -0.75, scale = 0.5
    # (both exact in fp16), then build r = s o (H v*) / 128 so that H (s o r) = v*.
    rng = np.random.default_rng(3)
    c = rng.integers(0, 4, D)
    c[5], c[77] = 0, 3  # make min and max attained
    v = -0.75 + 0.5 * c
    s = oracle.signs(99)
    H = scipy.linalg.hadamard(D).astype(np.float64)
    r = s * (H @ v) / D
    codes, sc, mn = oracle.quantize_residual(r, rot_seed=99, rotate=True)
    assert sc == np.float16(0.5).view(np.uint16) and mn == np.float16(-0.75).view(np.uint16)
    assert np.array_equal(codes, _pack(c))


def test_quantizer_degenerate_constant_residual():
    codes, sc, mn = oracle.quantize_residual(np.full(D, 0.3), rot_seed=1, rotate=False)
    assert sc == 0 and not codes.any()
    assert mn == np.float16(0.3).view(np.uint16)


# ---- encode: invariants and brute force ----------------------------------------

PAR = dict(f_a=0.02, f_rk=0.1, f_rv=0.1, W=32, seed=7, rot_seed=11)


@pytest.fixture(scope="module")
def tiny():
    S = 4096
    K, V = gen.clustered_batch(1, 1, [S], seed=42)
    units = oracle.encode(K, V, [S], 1, **PAR)
    return K[0, 0], V[0, 0], units[0]


def test_anchor_selection(tiny):
    K, V, u = tiny
    S, W = u.S, PAR["W"]
    assert u.k == 82 and len(np.unique(u.anchor_pos)) == u.k and np.all(np.diff(u.anchor_pos) > 0)
    assert np.array_equal(u.anchor_pos[-W:], np.arange(S - W, S))
    # the other k - W anchors are the positions of [0, S - W) with the smallest hash
    base = PAR["seed"] ^ (0 << 40) ^ (0 << 32)
    h = np.array([oracle.splitmix64(base ^ p) for p in range(S - W)], dtype=np.uint64)
    want = np.sort(np.argsort(h, kind="stable")[: u.k - W])
    assert np.array_equal(u.anchor_pos[:-W], want)
    # anchor rows are the input rows, bit for bit
    assert np.array_equal(u.anchor_k, K[u.anchor_pos]) and np.array_equal(u.anchor_v, V[u.anchor_pos])


@pytest.mark.parametrize("side", ["k", "v"])
def test_assignment_is_argmax_abs_cosine(tiny, side):
    K, V, u = tiny
    X = gen.bf16_to_f64(K if side == "k" else V)
    XA = X[u.anchor_pos]
    idx = u.idx_k if side == "k" else u.idx_v
    c = np.abs(X @ XA.T) / np.linalg.norm(XA, axis=1)[None, :]  # Eq. 1 up to the common 1/||x_i||
    non = np.setdiff1d(np.arange(u.S), u.anchor_pos)
    chosen = c[non, idx[non]]
    assert np.all(chosen >= c[non].max(axis=1) * (1 - 1e-12))
    assert np.array_equal(idx[u.anchor_pos], np.arange(u.k))


@pytest.mark.parametrize("side", ["k", "v"])
def test_gamma_is_least_squares_coefficient(tiny, side):
    K, V, u = tiny
    X = gen.bf16_to_f64(K if side == "k" else V)
    idx, gam = (u.idx_k, u.gam_k) if side == "k" else (u.idx_v, u.gam_v)
    non = np.setdiff1d(np.arange(u.S), u.anchor_pos)[::17]
    g_ls = np.array([np.linalg.lstsq(X[u.anchor_pos[idx[i]]][:, None], X[i], rcond=None)[0][0] for i in non])
    assert np.array_equal(gam[non], gen.fp16_bits(g_ls))  # Eq. 2, rounded once to fp16
    xa = X[u.anchor_pos[idx[non]]]
    r = X[non] - g_ls[:, None] * xa
    assert np.max(np.abs(np.sum(r * xa, axis=1)) / np.sum(xa * xa, axis=1)) < 1e-12  # r orthogonal to x_a
    assert np.all(gam[u.anchor_pos] == 0x3C00)  # anchors carry gamma = 1 on themselves


@pytest.mark.parametrize("side", ["k", "v"])
def test_slots_are_the_largest_residual_energies(tiny, side):
    K, V, u = tiny
    X = gen.bf16_to_f64(K if side == "k" else V)
    idx, gam, res, n = (u.idx_k, u.gam_k, u.res_k, u.nk) if side == "k" else (u.idx_v, u.gam_v, u.res_v, u.nv)
    g = gam.view(np.float16).astype(np.float64)
    e = np.sum((X - g[:, None] * X[u.anchor_pos[idx]]) ** 2, axis=1)
    non = np.setdiff1d(np.arange(u.S), u.anchor_pos)
    order = non[np.lexsort((non, -e[non]))]
    assert n == 409 and np.array_equal(res, np.sort(order[:n]))


@pytest.mark.parametrize("side", ["k", "v"])
def test_reconstruction_invariants(tiny, side):
    K, V, u = tiny
    X = gen.bf16_to_f64(K if side == "k" else V)
    Xh = oracle.reconstruct(u, side, PAR["rot_seed"])
    idx, gam, res = (u.idx_k, u.gam_k, u.res_k) if side == "k" else (u.idx_v, u.gam_v, u.res_v)
    # anchors reconstruct exactly
    assert np.array_equal(Xh[u.anchor_pos], X[u.anchor_pos])
    # a token without a residual lies on the span of its anchor: x^ = gamma x_a exactly
    g = gam.view(np.float16).astype(np.float64)
    plain = np.setdiff1d(np.setdiff1d(np.arange(u.S), u.anchor_pos), res)
    assert np.array_equal(Xh[plain], g[plain, None] * X[u.anchor_pos[idx[plain]]])
    # its error is exactly its residual norm; stored residuals cut the error on average
    r = X - g[:, None] * X[u.anchor_pos[idx]]
    err = np.linalg.norm(X - Xh, axis=1)
    rn = np.linalg.norm(r, axis=1)
    assert np.allclose(err[plain], rn[plain], rtol=1e-12)
    assert np.mean(err[res] / rn[res]) < 0.5


def test_residual_dequant_matches_dense_hadamard(tiny):
    _, _, u = tiny
    s = oracle.signs(PAR["rot_seed"])
    H = scipy.linalg.hadamard(D).astype(np.float64)
    g = u.gam_k.view(np.float16).astype(np.float64)
    base = g[:, None] * gen.bf16_to_f64(u.anchor_k)[u.idx_k]
    Xh = oracle.reconstruct(u, "k", PAR["rot_seed"])
    for t in range(0, u.nk, 37):
        codes = np.array([(u.codes_k[t, j // 4] >> (2 * (j % 4))) & 3 for j in range(D)], np.float64)
        chat = u.min_k[t:t + 1].view(np.float16).astype(np.float64)[0] + codes * \
            u.scale_k[t:t + 1].view(np.float16).astype(np.float64)[0]
        rt = s * (H @ chat) / D  # Eq. 14: r~ = U^T C^-1(q), U = H diag(s) / sqrt(D)
        i = u.res_k[t]
        assert np.allclose(Xh[i], base[i] + rt, rtol=0, atol=1e-12)


# ---- attention: brute force, factorised identity, special cases, Theorem 1 ----

def _softmax_attend(Kh, Vh, q, sm_scale):
    l = sm_scale * (Kh @ q)
    a = np.exp(l - l.max())
    a /= a.sum()
    return a @ Vh, a


@pytest.mark.parametrize("sm_scale", [1.0, 1 / math.sqrt(D)])
def test_attend_matches_dense_bruteforce(tiny, sm_scale):
    _, _, u = tiny
    q = gen.queries(1, 5)
    out = oracle.attend([u], q, 1, sm_scale, PAR["rot_seed"])[0, 0]
    Kh = oracle.reconstruct(u, "k", PAR["rot_seed"])
    Vh = oracle.reconstruct(u, "v", PAR["rot_seed"])
    y, _ = _softmax_attend(Kh, Vh, gen.bf16_to_f64(q[0]), sm_scale)
    assert np.allclose(out, y, rtol=0, atol=1e-12)


@pytest.mark.parametrize("G", [1, 4, 8])
def test_factorized_equals_definition(tiny, G):
    _, _, u = tiny
    q = gen.queries(G, 6)
    out = oracle.attend([u], q, G, 1.0, PAR["rot_seed"])[0]
    f = oracle.attend_factorized(u, q, G, 1.0, PAR["rot_seed"])
    assert np.allclose(out, f, rtol=0, atol=1e-12)


@pytest.mark.parametrize("S", [1, 2, 31, 32, 33, 64, 65, 127])
def test_small_contexts_bruteforce(S):
    K, V = gen.clustered_batch(1, 1, [S], seed=S)
    u = oracle.encode(K, V, [S], 1, 0.02, 0.5, 0.5, 32, 3, 11)[0]
    q = gen.queries(2, S)
    out = oracle.attend([u], q, 2, 1.0, 11)[0]
    Kh, Vh = oracle.reconstruct(u, "k", 11), oracle.reconstruct(u, "v", 11)
    for g in range(2):
        y, _ = _softmax_attend(Kh, Vh, gen.bf16_to_f64(q[g]), 1.0)
        assert np.allclose(out[g], y, rtol=0, atol=1e-12)
    if S <= 32:  # every position is an anchor: plain softmax attention over the input rows
        for g in range(2):
            y, _ = _softmax_attend(gen.bf16_to_f64(K[0, 0]), gen.bf16_to_f64(V[0, 0]), gen.bf16_to_f64(q[g]), 1.0)
            assert np.allclose(out[g], y, rtol=0, atol=1e-13)
    if S == 1:
        assert np.array_equal(out[0], gen.bf16_to_f64(V[0, 0, 0]))


@pytest.mark.parametrize("sm_scale", [1.0, 1 / math.sqrt(D)])
def test_theorem1_output_error_bound(tiny, sm_scale):
    K, V, u = tiny
    Kx, Vx = gen.bf16_to_f64(K), gen.bf16_to_f64(V)
    Kh, Vh = oracle.reconstruct(u, "k", PAR["rot_seed"]), oracle.reconstruct(u, "v", PAR["rot_seed"])
    for t in range(4):
        q = gen.bf16_to_f64(gen.queries(1, 100 + t)[0])
        y, _ = _softmax_attend(Kx, Vx, q, sm_scale)
        yh, ah = _softmax_attend(Kh, Vh, q, sm_scale)
        E_V = np.sum(ah * np.linalg.norm(Vx - Vh, axis=1))
        mu = sm_scale * np.linalg.norm(q) * np.max(np.linalg.norm(Kx - Kh, axis=1))
        E_K = 2 * np.max(np.linalg.norm(Vx, axis=1)) * np.tanh(mu)
        assert np.linalg.norm(y - yh) <= E_V + E_K


def test_zero_and_parallel_vectors():
    S = 200
    K, V = gen.clustered_batch(1, 1, [S], seed=9)
    K = K.copy()
    V = V.copy()
    K[0, 0, 10] = 0  # zero key: no direction, gamma 0
    V[0, 0, 11] = 0
    # a negative multiple of the last (anchor) row: gamma must come out negative
    K[0, 0, 12] = gen.bf16_bits(-2.0 * gen.bf16_to_f64(K[0, 0, S - 1]))
    u = oracle.encode(K, V, [S], 1, 0.02, 0.1, 0.1, 32, 3, 11)[0]
    assert u.gam_k[10] == 0 and u.gam_v[11] == 0
    assert u.idx_k[12] == u.k - 1 and u.gam_k[12] == np.float16(-2.0).view(np.uint16)


# ---- exact dense suffix (Appendix E.1, E.2): one softmax over prefix and suffix ----

def _suffix_rows(n, seed, scale=1.0):
    """bf16 bits [n][128] of clustered rows (a generated token's key or value)."""
    K, V = gen.clustered_batch(1, 1, [max(n, 1)], seed=seed)
    if scale != 1.0:
        K = gen.bf16_bits(gen.bf16_to_f64(K) * scale)
    return K[0, 0, :n], V[0, 0, :n]


@pytest.mark.parametrize("n_suf", [1, 5, 70])
@pytest.mark.parametrize("sm_scale", [1.0, 1 / math.sqrt(D)])
def test_suffix_attend_matches_dense_bruteforce(tiny, n_suf, sm_scale):
    """The compressed positions, rebuilt per Eq. 3, followed by the exact suffix rows, under one
    softmax: equal to a dense softmax over the concatenated rows."""
    _, _, u = tiny
    ks, vs = _suffix_rows(n_suf, 900 + n_suf)
    q = gen.queries(2, 77)
    out = oracle.attend_suffix([u], q, 2, 1, sm_scale, PAR["rot_seed"], ks[None], vs[None], [n_suf])[0]
    Kh = np.concatenate([oracle.reconstruct(u, "k", PAR["rot_seed"]), gen.bf16_to_f64(ks)])
    Vh = np.concatenate([oracle.reconstruct(u, "v", PAR["rot_seed"]), gen.bf16_to_f64(vs)])
    for g in range(2):
        y, _ = _softmax_attend(Kh, Vh, gen.bf16_to_f64(q[g]), sm_scale)
        assert np.allclose(out[g], y, rtol=0, atol=1e-12)


def test_suffix_rows_past_the_length_are_ignored_and_empty_suffix_is_plain_attend(tiny):
    _, _, u = tiny
    ks, vs = _suffix_rows(40, 901)
    q = gen.queries(4, 78)
    plain = oracle.attend([u], q, 4, 1.0, PAR["rot_seed"])
    empty = oracle.attend_suffix([u], q, 4, 1, 1.0, PAR["rot_seed"], ks[None], vs[None], [0])
    assert np.array_equal(plain, empty)
    short = oracle.attend_suffix([u], q, 4, 1, 1.0, PAR["rot_seed"], ks[None, :10], vs[None, :10], [10])
    garbage = ks.copy()
    garbage[10:] = 0x7F80  # +inf rows past the length must never be read
    cut = oracle.attend_suffix([u], q, 4, 1, 1.0, PAR["rot_seed"], garbage[None], vs[None], [10])
    assert np.array_equal(short, cut)


def test_suffix_all_anchor_prefix_is_plain_softmax_over_the_input_rows():
    """Every compressed position an anchor (S <= W): prefix and suffix are both exact, so the
    result is textbook softmax attention over the input rows followed by the suffix rows; a suffix
    whose logits dwarf the prefix's takes almost all the weight."""
    S = 24
    K, V = gen.clustered_batch(1, 1, [S], seed=5)
    u = oracle.encode(K, V, [S], 1, 0.02, 0.1, 0.1, 32, 3, 11)[0]
    for scale in (1.0, 8.0):
        ks, vs = _suffix_rows(9, 902, scale)
        q = gen.queries(1, 79)
        out = oracle.attend_suffix([u], q, 1, 1, 1.0, 11, ks[None], vs[None], [9])[0, 0]
        Kx = np.concatenate([gen.bf16_to_f64(K[0, 0]), gen.bf16_to_f64(ks)])
        Vx = np.concatenate([gen.bf16_to_f64(V[0, 0]), gen.bf16_to_f64(vs)])
        y, a = _softmax_attend(Kx, Vx, gen.bf16_to_f64(q[0]), 1.0)
        assert np.allclose(out, y, rtol=0, atol=1e-13)
    assert a[S:].sum() > 0.99  # the scaled suffix dominates


def test_suffix_lengths_follow_requests_in_a_batch():
    """Unit u = b*H + h takes request b's length: two requests, two KV heads, lengths 3 and 0."""
    S, H = 300, 2
    K, V = gen.clustered_batch(2, H, [S, S], seed=8)
    units = oracle.encode(K, V, [S, S], H, 0.02, 0.1, 0.1, 32, 3, 11)
    ks = np.zeros((4, 6, D), np.uint16)
    vs = np.zeros((4, 6, D), np.uint16)
    for u in range(4):
        ks[u], vs[u] = _suffix_rows(6, 910 + u)
    q = gen.queries(4 * 2, 80)
    out = oracle.attend_suffix(units, q, 2, H, 1.0, 11, ks, vs, [3, 0])
    plain = oracle.attend(units, q, 2, 1.0, 11)
    for u in range(4):
        ref = oracle.attend_suffix([units[u]], q.reshape(4, 2, D)[u], 2, 1, 1.0, 11, ks[u:u + 1, :3], vs[u:u + 1, :3],
                                   [3]) if u < 2 else plain[u:u + 1]
        assert np.array_equal(out[u:u + 1], ref)


# ---- Lloyd-Max codec (Section 3.1, Appendix A.1 "Codebook"; distortion Eq. 13) ----

# Max (1960): the four-level minimum-MSE quantizer of a unit Gaussian has levels +-0.4528,
# +-1.5104 and thresholds 0, +-0.9816; the codec takes the levels to 8 significant bits.
LM_LEVELS = np.array([-1.5078125, -0.453125, 0.453125, 1.5078125])


def test_lloyd_levels_are_the_gaussian_lloyd_max_quantizer():
    """The table is within 0.5 % of Max's levels, and those levels are the centroids of the unit
    Gaussian over their own midpoint decision regions (the Lloyd condition), to 1e-3."""
    import scipy.stats as st
    assert np.allclose(LM_LEVELS, [-1.5104, -0.4528, 0.4528, 1.5104], rtol=5e-3)
    t = 0.5 * (0.4528 + 1.5104)
    for lo, hi, level in ((0.0, t, 0.4528), (t, np.inf, 1.5104)):
        centroid = (st.norm.pdf(lo) - st.norm.pdf(hi)) / (st.norm.cdf(hi) - st.norm.cdf(lo))
        assert abs(centroid - level) < 1e-3


def test_lloyd_quantizer_without_rotation_hand_example():
    # 48 coordinates of +-1.5 sigma and 80 of +-0.5 sigma: the RMS is exactly sigma = 0.75
    # (fp16-exact); +-1.5 lies beyond the outer threshold, +-0.5 inside it
    t = np.array([1.5] * 24 + [-1.5] * 24 + [0.5] * 40 + [-0.5] * 40)
    rng = np.random.default_rng(4)
    perm = rng.permutation(D)
    r = 0.75 * t[perm]
    codes, sc, mn = oracle.quantize_residual(r, rot_seed=5, rotate=False, lloyd=True)
    assert sc == np.float16(0.75).view(np.uint16) and mn == 0
    expect = np.where(t[perm] > 1, 3, np.where(t[perm] > 0, 2, np.where(t[perm] > -1, 1, 0)))
    assert np.array_equal(codes, _pack(expect))
    out = oracle.dequantize_residual(codes, sc, mn, rot_seed=5, rotate=False, lloyd=True)
    assert np.array_equal(out, 0.75 * LM_LEVELS[expect])


def test_lloyd_quantizer_with_rotation_matches_a_dense_hadamard():
    """Codes of the rotated vector v = H (s o r) by the decision regions of v / fp16(RMS(v)), and
    the record dequantized as s o (H (scale L[code])) / 128 with a dense Hadamard matrix."""
    rng = np.random.default_rng(6)
    s = oracle.signs(21)
    H = scipy.linalg.hadamard(D).astype(np.float64)
    for _ in range(20):
        r = rng.standard_normal(D) * rng.uniform(0.01, 3.0)
        codes, sc, mn = oracle.quantize_residual(r, rot_seed=21, rotate=True, lloyd=True)
        v = H @ (s * r)
        scale = float(np.float16(np.sqrt(np.sum(v * v) / D)))
        assert sc == np.float16(scale).view(np.uint16) and mn == 0
        x = v / scale
        expect = np.where(x < -0.98046875, 0, np.where(x < 0, 1, np.where(x < 0.98046875, 2, 3)))
        assert np.array_equal(codes, _pack(expect))
        out = oracle.dequantize_residual(codes, sc, mn, rot_seed=21, rotate=True, lloyd=True)
        assert np.allclose(out, s * (H @ (scale * LM_LEVELS[expect])) / D, rtol=0, atol=1e-13)


def test_lloyd_zero_residual():
    codes, sc, mn = oracle.quantize_residual(np.zeros(D), rot_seed=1, rotate=True, lloyd=True)
    assert sc == 0 and mn == 0
    assert np.array_equal(codes, _pack([2] * D))
    assert not oracle.dequantize_residual(codes, sc, mn, 1, True, True).any()


def test_eta_of_each_codec_on_gaussian_residuals():
    """Eq. 13 on rotated Gaussian residuals: the Lloyd-Max codec leaves about the Gaussian
    four-level minimum MSE (0.1175, here from numerical integration of its own levels and
    thresholds; the per-token RMS scale brings it slightly lower), the uniform min/max codec about
    twice as much."""
    import scipy.integrate as si
    import scipy.stats as st
    T = 0.98046875
    mse = 2 * sum(si.quad(lambda x, L=L: (x - L) ** 2 * st.norm.pdf(x), lo, hi)[0]
                  for lo, hi, L in ((0, T, 0.453125), (T, np.inf, 1.5078125)))
    assert abs(mse - 0.1175) < 1e-3
    R = np.random.default_rng(0).standard_normal((2000, D))
    e_lm = oracle.eta(R, 11, True, True)
    e_un = oracle.eta(R, 11, True, False)
    assert abs(e_lm - mse) < 0.005
    assert 1.8 * e_lm < e_un < 0.3


# ---- RoPE at decode (Section 3.2: keys kept pre-RoPE, turned to their positions) ----

def _rope_complex(X, pos, base):
    """Rotate-half RoPE as complex multiplication: z_j = x_j + i x_{j+64} times e^{i p theta_j}."""
    X = np.atleast_2d(np.asarray(X, np.float64))
    th = base ** (-2.0 * np.arange(64) / 128.0)
    z = (X[:, :64] + 1j * X[:, 64:]) * np.exp(1j * np.asarray(pos, np.float64)[:, None] * th[None, :])
    return np.concatenate([z.real, z.imag], axis=1)


@pytest.mark.parametrize("base", [10000.0, 500000.0])
def test_rope_turn_is_the_complex_rotation(base):
    rng = np.random.default_rng(8)
    for p in (0, 1, 7, 4095, 131071, 1 << 20):
        x = rng.standard_normal(D)
        y = oracle.rope(x, p, base)
        assert np.allclose(y, _rope_complex(x, [p], base)[0], rtol=0, atol=1e-9)
        assert abs(np.linalg.norm(y) - np.linalg.norm(x)) < 1e-12  # a rotation


@pytest.mark.parametrize("base", [10000.0, 500000.0])
def test_rope_attend_matches_dense_bruteforce(tiny, base):
    """Each reconstructed (pre-RoPE) key turned to its position, then Eq. 4 softmax: equal to a
    dense softmax over the complex-rotated rows; positions from a permutation (stored order)."""
    _, _, u = tiny
    q = gen.queries(2, 81)
    Kh = oracle.reconstruct(u, "k", PAR["rot_seed"])
    Vh = oracle.reconstruct(u, "v", PAR["rot_seed"])
    for pos in (np.arange(u.S, dtype=np.int32), np.random.default_rng(3).permutation(u.S).astype(np.int32)):
        u.pos = pos
        out = oracle.attend([u], q, 2, 1.0, PAR["rot_seed"], rope_theta=base)[0]
        Kr = _rope_complex(Kh, pos, base)
        for g in range(2):
            y, _ = _softmax_attend(Kr, Vh, gen.bf16_to_f64(q[g]), 1.0)
            assert np.allclose(out[g], y, rtol=0, atol=1e-10)
    u.pos = np.arange(u.S, dtype=np.int32)


@pytest.mark.parametrize("base", [10000.0, 500000.0])
def test_rope_with_suffix_matches_dense_bruteforce(tiny, base):
    """RoPE at decode with a dense suffix (Section 3.2; Appendix E.2): the compressed keys turned to
    their stored positions and suffix token t turned to position S + t, after the request's S
    compressed tokens, all in one softmax: equal to a dense softmax over the complex-rotated rows."""
    _, _, u = tiny
    n_suf = 37
    ks, vs = _suffix_rows(n_suf, 930)
    q = gen.queries(2, 83)
    pos = np.random.default_rng(5).permutation(u.S).astype(np.int32)
    u.pos = pos
    try:
        out = oracle.attend_suffix([u], q, 2, 1, 1.0, PAR["rot_seed"], ks[None], vs[None], [n_suf],
                                   rope_theta=base)[0]
    finally:
        u.pos = np.arange(u.S, dtype=np.int32)
    Kr = np.concatenate([_rope_complex(oracle.reconstruct(u, "k", PAR["rot_seed"]), pos, base),
                         _rope_complex(gen.bf16_to_f64(ks), u.S + np.arange(n_suf), base)])
    Vh = np.concatenate([oracle.reconstruct(u, "v", PAR["rot_seed"]), gen.bf16_to_f64(vs)])
    for g in range(2):
        y, _ = _softmax_attend(Kr, Vh, gen.bf16_to_f64(q[g]), 1.0)
        assert np.allclose(out[g], y, rtol=0, atol=1e-10)


def test_rope_at_position_zero_is_plain_attention(tiny):
    _, _, u = tiny
    q = gen.queries(4, 82)
    plain = oracle.attend([u], q, 4, 1.0, PAR["rot_seed"])
    u.pos = np.zeros(u.S, np.int32)
    zero = oracle.attend([u], q, 4, 1.0, PAR["rot_seed"], rope_theta=500000.0)
    u.pos = np.arange(u.S, dtype=np.int32)
    assert np.array_equal(plain, zero)
    moved = oracle.attend([u], q, 4, 1.0, PAR["rot_seed"], rope_theta=500000.0)
    assert not np.allclose(plain, moved, rtol=0, atol=1e-6)
