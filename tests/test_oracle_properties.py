"""Property tests of the oracle over random small shapes (host only): the
factored route to the projected gradient equals the explicit definition for
every projection kind, a unit-normalised row stays unit, top-k and bottom-k
equal Python's sorted() with the tie rules, and the per-token scores add up
to the per-sequence inner product."""
import numpy as np
import pytest

from oracle import bergson_oracle as orc

hyp = pytest.importorskip("hypothesis")
st = pytest.importorskip("hypothesis.strategies")

SETTINGS = hyp.settings(max_examples=60, deadline=None, derandomize=True)


def _layer(rng, B, T, d_in, d_out, k_in, k_out, kind, rc, seed):
    A = rng.standard_normal((B, T, d_in))
    G = rng.standard_normal((B, T, d_out))
    r = rng.uniform(0.5, 2.0, d_out) if rc else None
    c = rng.uniform(0.5, 2.0, d_in) if rc else None
    s_in, s_out = orc.module_seeds(seed, 0)
    return orc.Layer(A, G, k_in, k_out, s_in, s_out, r, c, 0, kind)


@SETTINGS
@hyp.given(B=st.integers(1, 3), T=st.integers(0, 12), d_in=st.integers(1, 12),
           d_out=st.integers(1, 12), k_in=st.sampled_from([1, 2, 5, 16]),
           k_out=st.sampled_from([1, 3, 16]), rc=st.booleans(),
           kind=st.sampled_from([orc.PROJ_GAUSSIAN, orc.PROJ_RADEMACHER, orc.PROJ_UNIFORM]),
           seed=st.integers(0, 2**32))
def test_factored_route_equals_explicit_definition(B, T, d_in, d_out, k_in, k_out, rc, kind, seed):
    rng = np.random.default_rng(seed)
    L = _layer(rng, B, T, d_in, d_out, k_in, k_out, kind, rc, seed)
    mask = (rng.random((B, T)) > 0.3).astype(np.uint8)
    got = orc.project_module(L, mask)
    s_in = 1.0 / np.sqrt(L.c) if rc else np.ones(d_in)
    s_out = 1.0 / np.sqrt(L.r) if rc else np.ones(d_out)
    P_in = orc.projection_matrix(L.seed_in, d_in, k_in, kind) * s_in[:, None]
    P_out = orc.projection_matrix(L.seed_out, d_out, k_out, kind) * s_out[:, None]
    for b in range(B):
        acc = np.zeros((k_out, k_in))
        for t in range(T):
            if mask[b, t]:
                acc += np.outer(L.G[b, t] @ P_out, L.A[b, t] @ P_in)
        scale = max(1.0, np.abs(acc).max())
        np.testing.assert_allclose(got[b], acc.reshape(-1), rtol=0, atol=1e-11 * scale)


@SETTINGS
@hyp.given(n=st.integers(1, 30), K=st.integers(1, 40), seed=st.integers(0, 2**32))
def test_unit_rows_and_fp16_store(n, K, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((n, K)) * rng.uniform(0.01, 100.0)
    x[rng.random(n) < 0.2] = 0.0
    rows, norms = orc.unit_normalize(x)
    nz = norms > 0
    np.testing.assert_allclose(np.linalg.norm(rows[nz], axis=1), 1.0, rtol=1e-12)
    assert np.all(rows[~nz] == 0.0)
    store, _ = orc.build_store(x)
    assert store.dtype == np.float16
    np.testing.assert_allclose(np.linalg.norm(store[nz].astype(np.float64), axis=1), 1.0,
                               atol=1e-3)


@SETTINGS
@hyp.given(Q=st.integers(1, 4), N=st.integers(1, 40), data=st.data())
def test_topk_and_bottomk_match_sorted(Q, N, data):
    k = data.draw(st.integers(1, N))
    vals = data.draw(st.lists(st.integers(-3, 3), min_size=Q * N, max_size=Q * N))
    S = np.array(vals, dtype=np.float64).reshape(Q, N) / 2.0      # many exact ties
    tv, ti = orc.topk_rows(S, k)
    bv, bi = orc.bottomk_rows(S, k)
    for q in range(Q):
        assert list(ti[q]) == sorted(range(N), key=lambda n: (-S[q, n], n))[:k]
        assert list(bi[q]) == sorted(range(N), key=lambda n: (S[q, n], n))[:k]
        assert list(tv[q]) == [S[q, n] for n in ti[q]]
        assert list(bv[q]) == [S[q, n] for n in bi[q]]


@SETTINGS
@hyp.given(B=st.integers(1, 2), T=st.integers(1, 8), d=st.integers(2, 8),
           seed=st.integers(0, 2**32))
def test_token_scores_sum_to_the_sequence_inner_product(B, T, d, seed):
    rng = np.random.default_rng(seed)
    L = _layer(rng, B, T, d, d + 1, 16, 16, orc.PROJ_GAUSSIAN, True, seed)
    mask = (rng.random((B, T)) > 0.25).astype(np.uint8)
    queries = rng.standard_normal((2, 256))
    per_token = orc.token_scores([L], mask, queries)              # [Q, B, T]
    rows = orc.project_grads([L], mask, 256)                      # [B, 256]
    np.testing.assert_allclose(per_token.sum(axis=2), queries @ rows.T, rtol=1e-9, atol=1e-9)
    assert np.all(per_token[:, mask == 0] == 0.0)
