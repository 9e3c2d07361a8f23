"""Pins for the fp64 CPU oracle: each check ties it to something other than itself.

Sources of truth used here: published SplitMix64 outputs, the closed form of
the Box-Muller transform, distribution tests, finite differences of a tiny
linear-layer loss, an independent (factored) algebraic route to the projected
gradient, the identity projection, a reparametrisation identity for the
Adafactor scaling, and brute-force sorting.
"""
import math

import numpy as np
import pytest
import scipy.stats

from oracle import bergson_oracle as orc

RNG = np.random.default_rng(20261202)


# --- generator --------------------------------------------------------------

def test_splitmix64_published_outputs():
    # First outputs of SplitMix64 seeded with 0 (Steele, Lea and Flood 2014;
    # the reference C code distributed with xoshiro/xoroshiro by Vigna).
    want = [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F,
            0xF88BB8A8724C81EC, 0x1B39896A51A8749B]
    got = [int(x) for x in orc.splitmix64_sequence(0, 5)]
    assert got == want


def test_box_muller_closed_form():
    # z_{2p}^2 + z_{2p+1}^2 = -2 ln u1 and atan2(z_{2p+1}, z_{2p}) = 2 pi u2 (mod 2 pi)
    seed = 77
    n = 4096
    z = orc.gaussian_counter(seed, n)
    p = np.arange(n // 2, dtype=np.uint64)
    s = np.uint64(seed)
    h1 = orc.mix64(s ^ orc.mix64(np.uint64(2) * p))
    h2 = orc.mix64(s ^ orc.mix64(np.uint64(2) * p + np.uint64(1)))
    u1 = ((h1 >> np.uint64(11)) + np.uint64(1)).astype(np.float64) / 2.0 ** 53
    u2 = (h2 >> np.uint64(11)).astype(np.float64) / 2.0 ** 53
    ze, zo = z[0::2], z[1::2]
    np.testing.assert_allclose(ze * ze + zo * zo, -2.0 * np.log(u1), rtol=1e-12, atol=1e-14)
    ang = np.mod(np.arctan2(zo, ze), 2.0 * np.pi)
    d = np.abs(ang - 2.0 * np.pi * u2)
    d = np.minimum(d, 2.0 * np.pi - d)
    assert d.max() < 1e-9


def test_gaussian_moments_and_ks():
    z = orc.gaussian_counter(12345, 1_000_000)
    n = z.size
    assert abs(z.mean()) < 5.0 / math.sqrt(n)
    assert abs(z.var() - 1.0) < 5.0 * math.sqrt(2.0 / n)
    assert scipy.stats.kstest(z, "norm").pvalue > 1e-4
    # neighbouring counters (same Box-Muller pair and across pairs) uncorrelated
    assert abs(np.corrcoef(z[0::2], z[1::2])[0, 1]) < 5.0 / math.sqrt(n / 2)
    assert abs(np.corrcoef(z[:-1], z[1:])[0, 1]) < 5.0 / math.sqrt(n)


def test_seeds_give_independent_streams():
    a = orc.gaussian_counter(1, 200_000)
    b = orc.gaussian_counter(2, 200_000)
    assert abs(np.corrcoef(a, b)[0, 1]) < 5.0 / math.sqrt(a.size)


def test_projection_scaling_preserves_norm_in_expectation():
    # Johnson-Lindenstrauss: E ||P^T x||^2 = ||x||^2 when P_ij ~ N(0, 1/k).
    d, k, trials = 96, 16, 400
    x = RNG.standard_normal(d)
    vals = np.array([np.sum((orc.projection_matrix(s, d, k).T @ x) ** 2) for s in range(trials)])
    ratio = vals / np.sum(x * x)          # ~ chi^2_k / k, mean 1, var 2/k
    assert abs(ratio.mean() - 1.0) < 5.0 * math.sqrt(2.0 / k / trials)


def test_projection_layout_is_counter_row_major():
    d, k, seed = 24, 16, 9
    P = orc.projection_matrix(seed, d, k)
    z = orc.gaussian_counter(seed, d * k)
    i, j = 5, 11
    assert P[i, j] == float(np.float32(z[i * k + j] / math.sqrt(k)))


# --- per-example gradient ---------------------------------------------------

def _tiny_loss(W, a, u, m):
    # L = sum_t m_t (u_t . y_t + 0.5 ||y_t||^2), y_t = W a_t
    y = a @ W.T
    return float(np.sum(m[:, None] * (u * y + 0.5 * y * y)))


@pytest.mark.parametrize("d_in,d_out", [(4, 6), (7, 5)])
def test_gradient_matches_finite_differences(d_in, d_out):
    T = 9
    W = RNG.standard_normal((d_out, d_in))
    a = RNG.standard_normal((T, d_in))
    u = RNG.standard_normal((T, d_out))
    m = (RNG.random(T) > 0.3).astype(np.float64)
    g = u + a @ W.T                      # dL/dy_t for unmasked tokens
    grad = orc.per_example_gradient(a, g, m)
    assert grad.shape == (d_out, d_in)
    h = 1e-6
    fd = np.zeros_like(W)
    for i in range(d_out):
        for j in range(d_in):
            Wp = W.copy(); Wp[i, j] += h
            Wm = W.copy(); Wm[i, j] -= h
            fd[i, j] = (_tiny_loss(Wp, a, u, m) - _tiny_loss(Wm, a, u, m)) / (2 * h)
    assert np.max(np.abs(grad - fd)) / np.max(np.abs(fd)) < 1e-7


def test_masked_tokens_contribute_nothing_even_if_nonfinite():
    T, d_in, d_out = 12, 5, 3
    a = RNG.standard_normal((T, d_in))
    g = RNG.standard_normal((T, d_out))
    m = np.ones(T, np.uint8); m[[2, 7, 11]] = 0
    a2, g2 = a.copy(), g.copy()
    a2[2] = np.nan; g2[7] = np.inf; a2[11] = 1e30
    keep = m.astype(bool)
    want = g[keep].T @ a[keep]
    np.testing.assert_allclose(orc.per_example_gradient(a2, g2, m), want, rtol=1e-14)


# --- normalisation + projection ---------------------------------------------

def _layer(B, T, d_in, d_out, k_in, k_out, rc, kind=orc.PROJ_GAUSSIAN, seed=0):
    A = RNG.standard_normal((B, T, d_in)).astype(np.float32)
    G = RNG.standard_normal((B, T, d_out)).astype(np.float32)
    r = RNG.uniform(0.5, 2.0, d_out) if rc else None
    c = RNG.uniform(0.5, 2.0, d_in) if rc else None
    s_in, s_out = orc.module_seeds(seed, 0)
    return orc.Layer(A, G, k_in, k_out, s_in, s_out, r, c, 0, kind)


def test_factored_identity_equals_explicit_path():
    # sum_t (P_out'^T g_t)(P_in'^T a_t)^T with P' = diag(s) P: a different route
    # to P_out^T (W / sqrt(r c^T)) P_in that never forms W.
    B, T = 3, 20
    L = _layer(B, T, 24, 40, 16, 8, rc=True)
    mask = (RNG.random((B, T)) > 0.25).astype(np.uint8)
    explicit = orc.project_module(L, mask)
    P_in = orc.projection_matrix(L.seed_in, L.d_in, L.k_in) / np.sqrt(L.c)[:, None]
    P_out = orc.projection_matrix(L.seed_out, L.d_out, L.k_out) / np.sqrt(L.r)[:, None]
    for b in range(B):
        at = L.A[b].astype(np.float64) @ P_in        # [T, k_in]
        gt = L.G[b].astype(np.float64) @ P_out       # [T, k_out]
        acc = np.zeros((L.k_out, L.k_in))
        for t in range(T):
            if mask[b, t]:
                acc += np.outer(gt[t], at[t])
        np.testing.assert_allclose(explicit[b], acc.reshape(-1), rtol=1e-12, atol=1e-12)


def test_identity_projection_reproduces_normalised_gradient():
    B, T, d_in, d_out = 2, 7, 16, 32
    L = _layer(B, T, d_in, d_out, d_in, d_out, rc=True, kind=orc.PROJ_IDENTITY)
    out = orc.project_module(L, None)
    for b in range(B):
        W = np.zeros((d_out, d_in))
        for t in range(T):
            for i in range(d_out):
                for j in range(d_in):
                    W[i, j] += float(L.G[b, t, i]) * float(L.A[b, t, j]) / math.sqrt(L.r[i] * L.c[j])
        # block layout: row-major, k_out (= d_out) major
        np.testing.assert_allclose(out[b].reshape(d_out, d_in), W, rtol=1e-12, atol=1e-12)


def test_adafactor_equals_reparametrised_inputs():
    # dividing W by sqrt(r_i c_j) equals the gradient of inputs a/sqrt(c) and
    # output-gradients g/sqrt(r) with no normalisation.
    B, T = 2, 11
    L = _layer(B, T, 24, 40, 16, 16, rc=True)
    base = orc.project_module(L, None)
    L2 = orc.Layer(L.A / np.sqrt(L.c), L.G / np.sqrt(L.r), L.k_in, L.k_out, L.seed_in, L.seed_out)
    np.testing.assert_allclose(base, orc.project_module(L2, None), rtol=1e-12, atol=1e-12)


def test_adafactor_uniform_moments_scale_by_closed_form():
    L = _layer(2, 9, 24, 40, 16, 16, rc=False)
    plain = orc.project_module(L, None)
    L.r = np.full(L.d_out, 4.0)
    L.c = np.full(L.d_in, 0.25)
    tol = 1e-12 * np.abs(plain).max()
    np.testing.assert_allclose(orc.project_module(L, None), plain / math.sqrt(4.0 * 0.25), rtol=0, atol=tol)
    L.r = np.full(L.d_out, 9.0)
    L.c = np.full(L.d_in, 4.0)
    np.testing.assert_allclose(orc.project_module(L, None), plain / 6.0, rtol=0, atol=tol)


def test_projection_inner_products_unbiased():
    # E <P_out^T W P_in, P_out^T V P_in> = <W, V> over independent seeds.
    d_in, d_out, k = 12, 10, 16
    W = RNG.standard_normal((d_out, d_in))
    V = W + 0.5 * RNG.standard_normal((d_out, d_in))
    trials = 600
    acc = []
    for s in range(trials):
        Pi = orc.projection_matrix(2 * s, d_in, k)
        Po = orc.projection_matrix(2 * s + 1, d_out, k)
        acc.append(np.sum(orc.double_sided_projection(W, Po, Pi) * orc.double_sided_projection(V, Po, Pi)))
    acc = np.array(acc)
    want = np.sum(W * V)
    assert abs(acc.mean() - want) < 5.0 * acc.std() / math.sqrt(trials)


def test_modules_land_at_their_column_offsets():
    B, T = 2, 5
    L0 = _layer(B, T, 16, 8, 16, 16, rc=False)
    L1 = _layer(B, T, 8, 24, 16, 16, rc=False, seed=3)
    L1.col_offset = 256 + 32          # gap of 32 untouched columns
    L1.G = np.zeros_like(L1.G)        # zero gradient -> zero block
    out = orc.project_grads([L0, L1], None, ld_out=256 + 32 + 256 + 16)
    np.testing.assert_array_equal(out[:, 256:]  , 0.0)
    np.testing.assert_allclose(out[:, :256], orc.project_module(L0, None), rtol=0, atol=0)


# --- store + scores ---------------------------------------------------------

def test_unit_normalize_and_store():
    X = RNG.standard_normal((6, 300))
    X[3] = 0.0
    rows, norms = orc.unit_normalize(X)
    n = np.linalg.norm(rows, axis=1)
    np.testing.assert_allclose(n[[0, 1, 2, 4, 5]], 1.0, atol=1e-14)
    assert n[3] == 0.0 and norms[3] == 0.0
    np.testing.assert_allclose(norms, np.linalg.norm(X, axis=1), rtol=1e-14)
    store, _ = orc.build_store(X)
    assert store.dtype == np.float16
    sn = np.linalg.norm(store.astype(np.float64), axis=1)
    np.testing.assert_allclose(sn[[0, 1, 2, 4, 5]], 1.0, atol=1e-3)


def test_scores_symmetric_with_self_top1():
    X = RNG.standard_normal((8, 256))
    store, _ = orc.build_store(X)
    S = orc.cosine_scores(store, store.astype(np.float64))
    np.testing.assert_allclose(S, S.T, atol=2e-3)
    np.testing.assert_allclose(np.diag(S), 1.0, atol=1e-3)
    val, idx = orc.topk_rows(S, 4)
    np.testing.assert_array_equal(idx[:, 0], np.arange(8))


def test_scores_are_cosines():
    store, _ = orc.build_store(RNG.standard_normal((5, 64)))
    q = RNG.standard_normal((3, 64))
    S = orc.cosine_scores(store, q)
    np.testing.assert_allclose(orc.cosine_scores(store, 7.5 * q), S, rtol=1e-13)
    s64 = store.astype(np.float64)
    for i in range(3):
        for n in range(5):
            cos = np.dot(q[i], s64[n]) / np.linalg.norm(q[i])
            assert abs(S[i, n] - cos) < 1e-13


def test_topk_matches_sorted_with_ties():
    S = np.round(RNG.standard_normal((4, 40)), 1)   # many exact ties
    S[1, 5] = S[1, 30] = 9.0                          # tie at the top
    val, idx = orc.topk_rows(S, 7)
    for q in range(4):
        want = sorted(range(40), key=lambda n: (-S[q, n], n))[:7]
        assert list(idx[q]) == want
        assert list(val[q]) == [S[q, n] for n in want]
    with pytest.raises(ValueError):
        orc.topk_rows(S, 41)


# --- on-the-fly scores -------------------------------------------------------

def test_onthefly_scores_definitions():
    X = RNG.standard_normal((5, 40))
    Y = RNG.standard_normal((3, 40))
    X[2] = 0.0
    S = orc.onthefly_scores(X, Y, unit=True)
    D = orc.onthefly_scores(X, Y, unit=False)
    for b in range(5):
        for q in range(3):
            dot = sum(float(X[b, i]) * float(Y[q, i]) for i in range(40))
            assert abs(D[b, q] - dot) < 1e-12
            nx = math.sqrt(sum(float(v) ** 2 for v in X[b]))
            ny = math.sqrt(sum(float(v) ** 2 for v in Y[q]))
            assert abs(S[b, q] - (dot / (nx * ny) if nx > 0 else 0.0)) < 1e-12
    np.testing.assert_array_equal(S[2], 0.0)
    # cosine: invariant to positive row/query scaling, bounded by 1, self-score 1
    np.testing.assert_allclose(orc.onthefly_scores(3.0 * X, 0.5 * Y), S, atol=1e-14)
    assert np.all(np.abs(S) <= 1 + 1e-12)
    np.testing.assert_allclose(np.diag(orc.onthefly_scores(Y, Y)), 1.0, atol=1e-14)
    # agrees with the store path up to the fp16 rounding of the rows
    store, _ = orc.build_store(X)
    np.testing.assert_allclose(orc.cosine_scores(store, Y).T, S, atol=2e-3)


# --- per-token scores ---------------------------------------------------------

def test_token_scores_sum_to_sequence_score():
    B, T = 2, 9
    L0 = _layer(B, T, 24, 16, 16, 16, rc=True)
    L1 = _layer(B, T, 16, 40, 16, 16, rc=True, seed=5)
    L1.col_offset = 256
    mask = (RNG.random((B, T)) > 0.3).astype(np.uint8)
    Qr = RNG.standard_normal((3, 512))
    tok = orc.token_scores([L0, L1], mask, Qr)
    seq = orc.project_grads([L0, L1], mask, 512)          # sums tokens before projecting
    np.testing.assert_allclose(tok.sum(axis=2), Qr @ seq.T, rtol=1e-11, atol=1e-11)
    assert np.all(tok[:, mask == 0] == 0.0)


def test_token_score_equals_single_token_sequence():
    B, T = 1, 6
    L = _layer(B, T, 24, 16, 16, 16, rc=False)
    Qr = RNG.standard_normal((2, 256))
    tok = orc.token_scores([L], None, Qr)
    for t in range(T):
        m = np.zeros((1, T), np.uint8)
        m[0, t] = 1
        np.testing.assert_allclose(tok[:, 0, t], Qr @ orc.project_grads([L], m, 256)[0], rtol=1e-11)


def test_token_scores_identity_closed_form():
    # P = I, no moments: s[q, b, t] = g_t^T Q_q a_t
    B, T, d_in, d_out = 1, 4, 16, 32
    L = _layer(B, T, d_in, d_out, d_in, d_out, rc=False, kind=orc.PROJ_IDENTITY)
    Qr = RNG.standard_normal((2, d_out * d_in))
    tok = orc.token_scores([L], None, Qr)
    for q in range(2):
        Qm = Qr[q].reshape(d_out, d_in)
        for t in range(T):
            g = L.G[0, t].astype(np.float64)
            a = L.A[0, t].astype(np.float64)
            want = sum(g[i] * Qm[i, j] * a[j] for i in range(d_out) for j in range(d_in))
            assert abs(tok[q, 0, t] - want) < 1e-10 * max(1.0, abs(want))


# --- query aggregation --------------------------------------------------------

def test_aggregate_rows_closed_forms():
    r = RNG.standard_normal(30)
    X = np.stack([r, 2 * r, 5 * r, RNG.standard_normal(30), RNG.standard_normal(30)])
    offs = [0, 3, 3, 5]                                   # groups: 3 rows, empty, 2 rows
    mean_n = orc.aggregate_rows(X, offs, orc.AGG_MEAN, True)
    np.testing.assert_allclose(mean_n[0], r / np.linalg.norm(r), atol=1e-14)   # same direction
    np.testing.assert_array_equal(mean_n[1], 0.0)
    sum_raw = orc.aggregate_rows(X, offs, orc.AGG_SUM, False)
    np.testing.assert_allclose(sum_raw[0], 8 * r, atol=1e-13)
    np.testing.assert_allclose(sum_raw[2], X[3] + X[4], atol=1e-14)
    mean_raw = orc.aggregate_rows(X, offs, orc.AGG_MEAN, False)
    np.testing.assert_allclose(mean_raw[2], 0.5 * (X[3] + X[4]), atol=1e-14)
    # scores of a mean-aggregated query are the mean of the members' scores
    store, _ = orc.build_store(RNG.standard_normal((7, 30)))
    S_members = store.astype(np.float64) @ orc.unit_normalize(X[3:5])[0].T
    np.testing.assert_allclose(store.astype(np.float64) @ mean_n[2], S_members.mean(axis=1), atol=1e-13)


# --- empirical-Fisher preconditioner ------------------------------------------

def test_fisher_fit_mix_power_apply():
    n, K = 40, 12
    X = RNG.standard_normal((n, K)) @ np.diag(np.linspace(0.2, 3.0, K))
    R = orc.fisher_fit(X)
    want = np.zeros((K, K))
    for i in range(n):
        want += np.outer(X[i], X[i])
    np.testing.assert_allclose(R, want / n, atol=1e-13)
    assert np.all(np.linalg.eigvalsh(R) > 0)
    R2 = orc.fisher_fit(RNG.standard_normal((n, K)))
    Rm = orc.fisher_mix(R, R2, 0.25, 0.1)
    np.testing.assert_allclose(Rm, 0.25 * R + 0.75 * R2 + 0.1 * np.trace(0.25 * R + 0.75 * R2) / K * np.eye(K),
                               atol=1e-13)
    M = orc.fisher_power(Rm, -0.5)
    np.testing.assert_allclose(M @ Rm @ M, np.eye(K), atol=1e-10)       # whitening
    np.testing.assert_allclose(M, M.T, atol=1e-12)
    Minv = orc.fisher_power(Rm, -1.0)
    np.testing.assert_allclose(Minv @ Rm, np.eye(K), atol=1e-10)
    # preconditioned rows are whitened: their Fisher under M is the identity
    Xp = orc.precondition_rows(X, orc.fisher_power(orc.fisher_mix(R, None, 1.0, 0.0), -0.5))
    np.testing.assert_allclose(orc.fisher_fit(Xp), np.eye(K), atol=1e-10)


# --- bias gradients -----------------------------------------------------------

def test_bias_gradient_finite_differences_and_augmented_input():
    T, d_in, d_out = 8, 5, 4
    W = RNG.standard_normal((d_out, d_in))
    bias = RNG.standard_normal(d_out)
    a = RNG.standard_normal((T, d_in))
    u = RNG.standard_normal((T, d_out))
    m = (RNG.random(T) > 0.3).astype(np.float64)

    def loss(bv):
        y = a @ W.T + bv
        return float(np.sum(m[:, None] * (u * y + 0.5 * y * y)))
    g = u + a @ W.T + bias                       # dL/dy_t
    gb = orc.bias_gradient(g, m)
    h = 1e-6
    fd = np.array([(loss(bias + h * np.eye(d_out)[i]) - loss(bias - h * np.eye(d_out)[i])) / (2 * h)
                   for i in range(d_out)])
    assert np.max(np.abs(gb - fd)) / np.max(np.abs(fd)) < 1e-7
    # the bias is the weight of a constant-one input feature
    a_aug = np.concatenate([a, np.ones((T, 1))], axis=1)
    np.testing.assert_allclose(orc.per_example_gradient(a_aug, g, m)[:, -1], gb, rtol=1e-13)


def test_projected_bias_identity_and_offsets():
    B, T, d = 2, 6, 16
    L = _layer(B, T, d, d, d, d, rc=True, kind=orc.PROJ_IDENTITY)
    L.bias_col_offset = d * d
    out = orc.project_grads([L], None)
    assert out.shape == (B, d * d + d)
    for b in range(B):
        want = L.G[b].astype(np.float64).sum(axis=0) / np.sqrt(L.r)
        np.testing.assert_allclose(out[b, d * d:], want, rtol=1e-12)
