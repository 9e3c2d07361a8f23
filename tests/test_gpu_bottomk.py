"""GPU parity of the bottom-k query (Bergson Sec. 3.1: the k most and least
influential training items) against the fp64 oracle's exact bottom-k.

Bar as for the top-k: scores within 1e-3 absolute, index sets exact except
among scores within 1e-4 of the k-th, order (score ascending, index
ascending).  Cases: ragged N and K, Q = 1 and Q = 129 (two query groups),
bottomk = N, the two-pass path with a prefix threshold (Q > 128 on a large
store), exact ties, planted anti-neighbours, and the identity with the top-k
of the negated queries (bitwise).
"""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import check_topk, np32

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _store_from_rows(rows: torch.Tensor) -> torch.Tensor:
    N, K = rows.shape
    store = torch.empty((N, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(rows.to(DEV), N, K, True, store, 0)
    return store


def _query(entry, store, queries, k):
    N, K = store.shape
    Q = queries.shape[0]
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(N, K, Q, k), DEV)
    s = torch.empty((Q, k), dtype=torch.float32, device=DEV)
    i = torch.empty((Q, k), dtype=torch.int64, device=DEV)
    entry(store, N, K, queries, k, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(s), i.cpu().numpy()


def _check_bottomk(s, i, S, k):
    # the bottom-k of S is the top-k of -S with the same tie rule
    check_topk(-s.astype(np.float64), i, -S, k)
    assert np.all(np.diff(s, axis=1) >= 0), "scores not ascending"


@pytest.mark.parametrize("N,K,Q,k", [(5000, 520, 200, 17), (40, 64, 1, 40), (777, 128, 129, 5),
                                      (3000, 1024, 64, 100)])
def test_bottomk_random(N, K, Q, k):
    g = wl.generator(N * 3 + K, "cpu")
    store = _store_from_rows(torch.randn((N, K), generator=g))
    queries = torch.randn((Q, K), generator=g)
    s, i = _query(bg.bergson_score_bottomk, store, queries.to(DEV), k)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    _check_bottomk(s, i, S, k)
    want_s, _ = orc.bottomk_rows(S, k)
    np.testing.assert_allclose(s, want_s, rtol=0, atol=1e-3)


@pytest.mark.parametrize("Q,k", [(130, 5), (40, 3)])
def test_bottomk_prefix_threshold_pass(Q, k):
    # Q > 128 on a store of >= 8 x 128 x k rows takes the prefix pass, whose
    # scores (against -q) seed the full pass; Q = 40 is the single-pass path.
    N, K = 30_000, 256
    g = wl.generator(Q * 11 + k, "cpu")
    rows = torch.randn((N, K), generator=g)
    queries = torch.randn((Q, K), generator=g)
    rows[100:100 + Q] = -queries + 0.3 * torch.randn((Q, K), generator=g)   # strong prefix hits
    rows[N - 300:N - 300 + 20] = -2.0 * queries[:20] + torch.randn((20, K), generator=g)
    store = _store_from_rows(rows)
    s, i = _query(bg.bergson_score_bottomk, store, queries.to(DEV), k)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    _check_bottomk(s, i, S, k)


def test_bottomk_equals_topk_of_negated_queries_bitwise():
    N, K, Q, k = 9000, 384, 33, 25
    g = wl.generator(77, "cpu")
    store = _store_from_rows(torch.randn((N, K), generator=g))
    queries = torch.randn((Q, K), generator=g).to(DEV)
    bs, bi = _query(bg.bergson_score_bottomk, store, queries, k)
    ts, ti = _query(bg.bergson_score_topk, store, -queries, k)
    np.testing.assert_array_equal(bi, ti)
    np.testing.assert_array_equal(bs, -ts)


def test_bottomk_ties_prefer_lower_index():
    g = wl.generator(5, "cpu")
    base = torch.randn((50, 256), generator=g)
    rows = torch.cat([base, -base[:10]], 0)         # rows 50..59 are the opposites of rows 0..9
    rows = torch.cat([rows, -base[:10]], 0)         # rows 60..69 duplicate rows 50..59
    store = _store_from_rows(rows)
    s, i = _query(bg.bergson_score_bottomk, store, base[:10].clone().to(DEV), 2)
    for r in range(10):
        assert set(i[r].tolist()) == {50 + r, 60 + r}
        assert i[r, 0] == 50 + r                     # equal scores: lower index first
        assert s[r, 0] == s[r, 1]
    np.testing.assert_allclose(s, -1.0, atol=1e-3)


def test_bottomk_planted_anti_neighbours_exact_set():
    N, K, Q, per = 60_000, 1024, 48, 100
    g = wl.generator(31, "cpu")
    rows = torch.randn((N, K), generator=g)
    queries = torch.randn((Q, K), generator=g)
    pos = wl.planted_positions(N, Q, per, seed=32)
    rows[pos.reshape(-1)] = wl.planted_rows(-queries, per, seed=33)
    store = _store_from_rows(rows)
    s, i = _query(bg.bergson_score_bottomk, store, queries.to(DEV), per)
    for q in range(Q):
        assert set(i[q].tolist()) == set(pos[q].tolist())
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    _check_bottomk(s, i, S, per)
