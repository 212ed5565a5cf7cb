"""Pins of the oracle's full selection (Algorithm 1; Section 3.2-3.4, Appendix A.2) against
things other than itself (CPU only): libm, numpy/scipy brute force, a finite-difference
check of the first-order error each utility prices, the paper's worked example, and the
special case that reduces to the plain encoder."""
import math
import os

import numpy as np
import pytest
import scipy.special

import gen
import oracle

D = 128
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _f64(b):
    return gen.bf16_to_f64(b)


def _obs_queries(K, m, seed):
    """Observation rows near a few of the unit's keys (any bf16 rows serve the pins)."""
    rng = np.random.default_rng(seed)
    t = rng.integers(0, K.shape[0], size=m)
    return gen.bf16_bits(0.25 * _f64(K[t]) + rng.standard_normal((m, D)))


def _alpha(K, Q):
    """Exact attention of the rows of Q over K (Eq. 4 with 1/sqrt(D)), by scipy."""
    return scipy.special.softmax(_f64(Q) @ _f64(K).T / math.sqrt(D), axis=1)


def test_exp_matches_libm():
    rng = np.random.default_rng(3)
    xs = np.concatenate([-rng.uniform(0, 700, 5000), -rng.uniform(0, 2, 5000), [0.0, -1e-300, -700.0]])
    for x in xs:
        got, want = oracle.exp_neg(float(x)), math.exp(float(x))
        assert abs(got - want) <= np.spacing(want), (x, got, want)
    assert oracle.exp_neg(0.0) == 1.0 and oracle.exp_neg(-700.5) == 0.0


@pytest.mark.parametrize("S,W,m,kappa", [(200, 16, 8, 7), (97, 32, 64, 7), (150, 8, 16, 1), (40, 0, 4, 3)])
def test_selector_scores_brute_force(S, W, m, kappa):
    K, _ = gen.clustered_kv(S, 11, 0)
    Q = _obs_queries(K, m, 5)
    got = oracle.selector_scores(K, Q, W, kappa)
    P = S - min(W, S)
    mean = _alpha(K, Q).mean(axis=0)[:P]
    want = np.convolve(mean, np.ones(kappa), mode="same") / kappa  # zero padding, divisor kappa
    assert got.shape == (P,)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-300)


def test_budget_reproduces_the_worked_example():
    g = {}
    for line in open(os.path.join(GOLDEN, "paper_worked_example.txt")):
        if line.strip() and not line.startswith("#"):
            a, b = line.split()
            g[a] = float(b)
    N = oracle.budget_n(g["theta"], int(g["S"]), int(g["H"]), int(g["W"]), int(g["k"]))
    assert N == int(g["n_residuals"])
    assert oracle.budget_n(0.0, 32768, 8, 32, 256) == 0  # no budget left after the fixed bytes


def _unit_with_anchors(S, W, f_a, seed):
    """A plainly encoded unit (anchors, indices, coefficients) and its dense rows."""
    K, V = gen.clustered_batch(1, 1, [S], seed=seed)
    u = oracle.encode(K, V, [S], 1, f_a, 0.0, 0.0, W, 9, 10)[0]
    return u, K[0, 0], V[0, 0]


def _brute_utilities(u, K, V, Q):
    a = _alpha(K, Q)
    y = a @ _f64(V)
    gk = np.asarray(u.gam_k).view(np.float16).astype(np.float64)
    gv = np.asarray(u.gam_v).view(np.float16).astype(np.float64)
    rk = _f64(K) - gk[:, None] * _f64(u.anchor_k)[u.idx_k]
    rv = _f64(V) - gv[:, None] * _f64(u.anchor_v)[u.idx_v]
    dk = (_f64(Q) @ rk.T) ** 2 / D  # [m][S]
    cv = ((_f64(V)[None, :, :] - y[:, None, :]) ** 2).sum(axis=2)  # [m][S]
    uk = (a ** 2 * dk * cv).mean(axis=0)
    uv = (a ** 2).mean(axis=0) * (rv ** 2).sum(axis=1)
    return uk, uv, a, y, rk, rv


def test_utilities_brute_force():
    u, K, V = _unit_with_anchors(300, 16, 0.1, 4)
    Q = _obs_queries(K, 32, 6)
    uk, uv = oracle.utilities(u, K, V, Q)
    bk, bv, *_ = _brute_utilities(u, K, V, Q)
    non = np.setdiff1d(np.arange(u.S), u.anchor_pos)
    np.testing.assert_allclose(uk[non], bk[non], rtol=1e-11)
    np.testing.assert_allclose(uv[non], bv[non], rtol=1e-11)
    assert np.all(uk[u.anchor_pos] == -1.0) and np.all(uv[u.anchor_pos] == -1.0)


def test_utilities_price_the_first_order_output_error():
    """With one observation row, dropping token t's key residual moves the exact output by
    alpha_t ds_t (V_t - y) to first order (Eq. 5 with one perturbed logit: the token's own
    weight moves by alpha_t (1 - alpha_t) ds_t and every other weight by -alpha_u alpha_t ds_t),
    so ||dy||^2 = u^K_t; dropping its value residual moves it by -alpha_t r^V_t, so
    ||dy||^2 = u^V_t.  Checked by finite differences of the exact attention."""
    u, K, V = _unit_with_anchors(260, 16, 0.1, 8)
    Q = _obs_queries(K, 1, 2)
    uk, uv = oracle.utilities(u, K, V, Q)
    _, _, a, y, rk, rv = _brute_utilities(u, K, V, Q)
    Kf, Vf, q = _f64(K), _f64(V), _f64(Q)[0]
    non = np.setdiff1d(np.arange(u.S), u.anchor_pos)
    t_sel = non[np.argsort(-uk[non])[:5]]
    eps = 1e-6
    for t in t_sel:
        K2 = Kf.copy()
        K2[t] -= eps * rk[t]
        a2 = scipy.special.softmax(K2 @ q / math.sqrt(D))
        dy = (a2 @ Vf - y[0]) / eps
        assert abs(dy @ dy - uk[t]) <= 1e-4 * uk[t], t
        V2 = Vf.copy()
        V2[t] -= eps * rv[t]
        dyv = (a[0] @ V2 - y[0]) / eps
        assert abs(dyv @ dyv - uv[t]) <= 1e-6 * uv[t], t


def _select_case(lens, H, G, W, f_a, theta, rho, kappa, seed=3):
    B = len(lens)
    K, V = gen.clustered_batch(B, H, lens, seed=seed)
    m = W * G
    Q = np.zeros((B, H, m, D), np.uint16)
    for b in range(B):
        for h in range(H):
            Q[b, h] = _obs_queries(K[b, h, :lens[b]], m, 100 * b + h)
    units = oracle.encode_select(K, V, Q, lens, H, f_a, W, theta, rho, kappa, 17, 18)
    return K, V, Q, units


def _hash_rank(P, b, h, seed=17):
    base = seed ^ (b << 40) ^ (h << 32)
    keys = np.array([oracle.splitmix64(base ^ p) for p in range(P)], dtype=np.uint64)
    return np.argsort(keys, kind="stable")


@pytest.mark.parametrize("lens,H,G", [([700, 451], 2, 2), ([520], 3, 4)])
def test_select_anchors_and_pooled_residuals(lens, H, G):
    W, f_a, theta, rho, kappa = 16, 0.06, 0.11, 0.7, 7
    K, V, Q, units = _select_case(lens, H, G, W, f_a, theta, rho, kappa)
    for b, S in enumerate(lens):
        k = units[b * H].k
        w = min(W, S)
        n_s = math.floor(np.float32(rho).item() * (k - w))
        cands = [[], []]
        for h in range(H):
            u = units[b * H + h]
            Kh, Vh, Qh = K[b, h, :S], V[b, h, :S], Q[b, h]
            # anchors: the window, the top n_s selector scores, then the sampling hash order
            P = S - w
            mean = _alpha(Kh, Qh).mean(axis=0)[:P]
            sc = np.convolve(mean, np.ones(kappa), mode="same") / kappa
            top = np.lexsort((np.arange(P), -sc))[:n_s]
            rest = [p for p in _hash_rank(P, b, h) if p not in set(top.tolist())][:k - w - n_s]
            want = np.sort(np.concatenate([top, rest, np.arange(P, S)])).astype(np.int32)
            assert np.array_equal(u.anchor_pos, want), (b, h)
            bk, bv, *_ = _brute_utilities(u, Kh, Vh, Qh)
            non = np.setdiff1d(np.arange(S), u.anchor_pos)
            for side, arr in ((0, bk), (1, bv)):
                cands[side] += [(-arr[t], h, t) for t in non]
        N = oracle.budget_n(np.float32(theta).item(), S, H, W, k)
        for side, n in ((0, N // 2), (1, N - N // 2)):
            order = sorted(cands[side])
            n = min(n, len(order))
            chosen = {(h, t) for _, h, t in order[:n]}
            # utilities equal only within rounding could order differently: require a clear margin
            if n < len(order):
                assert order[n - 1][0] < order[n][0] * (1 - 1e-9) or order[n - 1][0] == order[n][0]
            got = set()
            for h in range(H):
                u = units[b * H + h]
                res = u.res_k if side == 0 else u.res_v
                assert np.all(np.diff(res) > 0)
                got |= {(h, int(t)) for t in res}
            assert got == chosen, (b, side)


def test_select_codes_are_the_pinned_quantizer_of_the_residual():
    K, V, Q, units = _select_case([300], 2, 2, 16, 0.1, 0.2, 0.7, 7)
    for h, u in enumerate(units):
        for side, X, A, idx, gam, res, codes, sc, mn in (
                ("k", K[0, h], u.anchor_k, u.idx_k, u.gam_k, u.res_k, u.codes_k, u.scale_k, u.min_k),
                ("v", V[0, h], u.anchor_v, u.idx_v, u.gam_v, u.res_v, u.codes_v, u.scale_v, u.min_v)):
            g = np.asarray(gam).view(np.float16).astype(np.float64)
            for i, t in enumerate(res[:20]):
                r = _f64(X[t]) - g[t] * _f64(A[idx[t]])
                c, s_, m_ = oracle.quantize_residual(r, 18)
                assert np.array_equal(c, codes[i]) and s_ == sc[i] and m_ == mn[i], (side, t)


def test_select_without_scored_anchors_and_with_every_residual_is_the_plain_encoder():
    """rho = 0 keeps the window plus the sampled anchors of the plain encoder, and a budget
    above every candidate gives every non-anchor both residuals: the plain encoder with
    residual fractions 1 must then produce the same cache."""
    lens, H, G, W, f_a = [333, 129], 2, 2, 16, 0.1
    K, V = gen.clustered_batch(len(lens), H, lens, seed=5)
    Q = np.zeros((len(lens), H, W * G, D), np.uint16)
    for b in range(len(lens)):
        for h in range(H):
            Q[b, h] = _obs_queries(K[b, h, :lens[b]], W * G, b + 7 * h)
    sel = oracle.encode_select(K, V, Q, lens, H, f_a, W, 1.0, 0.0, 7, 17, 18)
    plain = oracle.encode(K, V, lens, H, f_a, 1.0, 1.0, W, 17, 18)
    for a, b in zip(sel, plain):
        for f in ("anchor_pos", "anchor_k", "anchor_v", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
                  "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v"):
            assert np.array_equal(np.asarray(getattr(a, f)), np.asarray(getattr(b, f))), f
