"""GPU parity of the two-SM scorer (more than 128 queries: clusters of two
CTAs, one tcgen05 MMA of M = 256 per pair, each CTA loading half of every
store tile; one query tile per CTA up to 256 queries, two above) against the
fp64 oracle.

Cases: the smallest pair counts (Q = 129: one query on the odd CTA; Q = 257:
the odd CTA's second query tile and most of the even CTA's are empty), ragged query counts, stores whose
last tile leaves the odd CTA's half partly or wholly past N, K not a
multiple of 64, topk 1 to 100, the prefix-threshold path with ties across
the prefix boundary, planted neighbours with known exact sets, the bottom-k
search, and agreement with the single-CTA kernel on the queries both serve.
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


def _store(rows: torch.Tensor) -> torch.Tensor:
    N, K = rows.shape
    st = torch.empty((N, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(rows.to(DEV), N, K, True, st, 0)
    return st


def _query(store, queries, k, entry=None):
    entry = entry or bg.bergson_score_topk
    N, K = store.shape
    Q = queries.shape[0]
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(N, K, Q, k), DEV)
    s = torch.empty((Q, k), dtype=torch.float32, device=DEV)
    i = torch.empty((Q, k), dtype=torch.int64, device=DEV)
    entry(store, N, K, queries, k, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(s), i.cpu().numpy()


@pytest.mark.parametrize("N,K,Q,topk", [
    (10_100, 1024, 129, 17),     # one query tile per CTA; the odd CTA holds one query
    (5_020, 520, 256, 5),        # one query tile per CTA, both full
    (10_100, 1024, 257, 17),     # last tile: 100 rows, the odd CTA's half empty
    (5_020, 520, 600, 1),        # K % 64 != 0, ragged query groups
    (7_000 + 200, 256, 1024, 100),   # last tile 200 rows: the odd CTA's half partly valid
    (300, 64, 511, 300),         # topk = N
    (20_000, 1024, 1300, 10),    # three pair groups: a ring of three paced producers
])
def test_pair_scorer_random(N, K, Q, topk):
    g = wl.generator(N + 7 * Q + K, "cpu")
    store = _store(torch.randn((N, K), generator=g))
    queries = torch.randn((Q, K), generator=g)
    s, i = _query(store, queries.to(DEV), topk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(s, i, S, topk)


def test_pair_scorer_prefix_threshold_pass():
    # N >= 8 x 128 x topk and Q > 128: prefix pass first, then the full pass
    # from its k-th scores; exact ties straddle the prefix boundary.
    N, K, Q, topk = 30_000, 256, 300, 3
    g = wl.generator(1234, "cpu")
    rows = torch.randn((N, K), generator=g)
    queries = torch.randn((Q, K), generator=g)
    rows[N - 5:] = rows[:5]
    queries[:5] = rows[:5]
    rows[100:100 + Q] = queries + 0.3 * torch.randn((Q, K), generator=g)
    store = _store(rows)
    s, i = _query(store, queries.to(DEV), topk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(s, i, S, topk)
    for r in range(5):
        assert set(i[r, :2].tolist()) == {r, N - 5 + r}


def test_pair_scorer_planted_neighbours_exact_set():
    N, K, Q, per = 60_000, 1024, 300, 100
    g = wl.generator(61, "cpu")
    rows = torch.randn((N, K), generator=g)
    queries = torch.randn((Q, K), generator=g)
    pos = wl.planted_positions(N, Q, per, seed=62)
    rows[pos.reshape(-1)] = wl.planted_rows(queries, per, seed=63)
    store = _store(rows)
    s, i = _query(store, queries.to(DEV), per)
    for q in range(Q):
        assert set(i[q].tolist()) == set(pos[q].tolist())
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(s, i, S, per)


@pytest.mark.parametrize("Q", [200, 400])
def test_pair_scorer_bottomk(Q):
    N, K, k = 9_000, 384, 10
    g = wl.generator(71, "cpu")
    store = _store(torch.randn((N, K), generator=g))
    queries = torch.randn((Q, K), generator=g)
    s, i = _query(store, queries.to(DEV), k, bg.bergson_score_bottomk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(-s.astype(np.float64), i, -S, k)
    ts, ti = _query(store, (-queries).to(DEV), k)
    np.testing.assert_array_equal(i, ti)
    np.testing.assert_array_equal(s, -ts)


@pytest.mark.parametrize("q_small,q_big", [(128, 129), (128, 257)])
def test_pair_and_single_cta_kernels_agree(q_small, q_big):
    # Q = 128 runs on the single-CTA kernel, Q = 129 on pairs with one query
    # tile per CTA and Q = 257 on pairs with two; the shared queries get the
    # same rows and (to fp32 summation order) the same scores.
    N, K = 20_000, 512
    g = wl.generator(81, "cpu")
    store = _store(torch.randn((N, K), generator=g))
    queries = torch.randn((q_big, K), generator=g).to(DEV)
    s1, i1 = _query(store, queries[:q_small].contiguous(), 20)
    s2, i2 = _query(store, queries, 20)
    np.testing.assert_allclose(s2[:q_small], s1, rtol=0, atol=2e-6)
    gap = np.abs(s1[:, :, None] - s1[:, None, :]) + np.eye(20)[None] * 1.0
    clear = gap.min(axis=2) > 1e-5          # entries without a near-tie partner
    assert np.all(i2[:q_small][clear] == i1[clear])


def test_pair_scorer_prefix_cut_to_whole_tile_rounds():
    # Q = 1024, topk = 100: the 12,800-row prefix is cut to one round of store
    # tiles over the CTAs of a query group; strong neighbours sit just inside and
    # just past the cut, and exact ties straddle it.
    N, K, Q, topk = 110_000, 128, 1024, 100
    g = wl.generator(91, "cpu")
    rows = torch.randn((N, K), generator=g)
    queries = torch.randn((Q, K), generator=g)
    for q in range(0, Q, 16):
        rows[9_000 + q] = queries[q] * 3.0 + torch.randn((K,), generator=g)
        rows[12_000 + q] = queries[q] * 3.0 + torch.randn((K,), generator=g)
    rows[13_500:13_510] = rows[9_700:9_710]
    store = _store(rows)
    s, i = _query(store, queries.to(DEV), topk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    sample = np.r_[0:1024:16, 1:64]
    check_topk(s[sample], i[sample], S[sample], topk)
    for q in range(0, Q, 16):
        assert {9_000 + q, 12_000 + q} <= set(i[q].tolist())
