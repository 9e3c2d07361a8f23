"""Exact top-k over a store scored chunk by chunk, and streamed from host memory.

Sec. 3.1: gradient stores are persisted to disk and queried with exact top-k,
so a store may be much larger than device memory.  A running [Q, k] result
merged chunk after chunk must be exactly the single-pass result: the same
rows, bit-identical scores (every score is computed the same way whatever
chunk holds its row) and the same order, ties included.  The single-pass
result is itself held to the fp64 oracle by the parity tests; here it is
also checked against the oracle directly.
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


def _store(rows):
    N, K = rows.shape
    st = torch.empty((N, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(rows.to(DEV), N, K, True, st, 0)
    return st


def _single(store, queries, topk, least=False):
    N, K = store.shape
    Q = queries.shape[0]
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(N, K, Q, topk), DEV)
    s = torch.empty((Q, topk), dtype=torch.float32, device=DEV)
    i = torch.empty((Q, topk), dtype=torch.int64, device=DEV)
    fn = bg.bergson_score_bottomk if least else bg.bergson_score_topk
    fn(store, N, K, queries, topk, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(s), i.cpu().numpy()


def _chunked(store, queries, topk, bounds, order, least=False):
    N, K = store.shape
    Q = queries.shape[0]
    ws = bg.workspace_tensor(bg.bergson_score_topk_update_workspace(K, Q, topk), DEV)
    s = torch.full((Q, topk), float("nan"), dtype=torch.float32, device=DEV)
    i = torch.full((Q, topk), -7, dtype=torch.int64, device=DEV)
    for n, c in enumerate(order):
        r0, r1 = bounds[c], bounds[c + 1]
        bg.bergson_score_topk_update(store[r0:r1], r1 - r0, K, r0, queries, topk, n == 0, s, i, ws,
                                     least=least)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(s), i.cpu().numpy()


def _rows_with_duplicates(N, K, seed):
    g = wl.generator(seed, "cpu")
    X = torch.randn((N, K), generator=g)
    X[N - 5] = X[3]           # exact duplicates far apart: equal scores, order by index
    X[N // 2] = X[10]
    return X


@pytest.mark.parametrize("Q,topk", [(5, 20), (200, 16), (300, 50)])
def test_chunks_in_any_order_equal_the_single_pass(Q, topk):
    N, K = 50_003, 256
    X = _rows_with_duplicates(N, K, 60 + Q)
    store = _store(X)
    g = wl.generator(61, "cpu")
    queries = torch.randn((Q, K), generator=g).to(DEV)
    want_s, want_i = _single(store, queries, topk)
    # a chunk smaller than topk, ragged sizes, chunk edges next to the duplicates
    bounds = [0, 4, 11, 11 + topk // 2, 13_000, 25_001, 25_002, 40_000, N]
    for order in (list(range(len(bounds) - 1)), [5, 0, 7, 2, 1, 6, 3, 4]):
        got_s, got_i = _chunked(store, queries, topk, bounds, order)
        np.testing.assert_array_equal(got_i, want_i)
        np.testing.assert_array_equal(got_s.view(np.uint32), want_s.view(np.uint32))
    S = orc.cosine_scores(store.cpu().numpy(), queries.cpu().numpy().astype(np.float64))
    check_topk(want_s[:8], want_i[:8], S[:8], topk)


@pytest.mark.parametrize("Q", [7, 260])
def test_bottomk_chunks_equal_the_single_pass(Q):
    N, K, k = 30_000, 192, 12
    X = _rows_with_duplicates(N, K, 70 + Q)
    store = _store(X)
    queries = wl.gaussian_rows(Q, K, seed=71).to(DEV)
    want_s, want_i = _single(store, queries, k, least=True)
    bounds = [0, 9_999, 10_000, 10_005, N]
    got_s, got_i = _chunked(store, queries, k, bounds, [2, 0, 3, 1], least=True)
    np.testing.assert_array_equal(got_i, want_i)
    np.testing.assert_array_equal(got_s.view(np.uint32), want_s.view(np.uint32))
    assert np.all(np.diff(got_s, axis=1) >= 0)


def test_planted_neighbours_across_chunk_edges():
    N, K, Q, topk = 40_000, 512, 6, 30
    g = wl.generator(80, "cpu")
    queries = torch.randn((Q, K), generator=g)
    X = torch.randn((N, K), generator=g)
    planted = wl.planted_rows(queries, topk, seed=81)
    # every query's planted rows straddle an edge of the 10,000-row chunks:
    # query q takes rows e - 45 + 3 j + q // 3 (j < 30) around edge e = 10,000 (q % 3 + 1)
    pos = np.stack([10_000 * (q % 3 + 1) - 45 + 3 * np.arange(topk) + q // 3 for q in range(Q)])
    assert len(np.unique(pos)) == pos.size
    X[torch.from_numpy(pos.reshape(-1))] = planted
    store = _store(X)
    want_s, want_i = _single(store, queries.to(DEV), topk)
    bounds = list(range(0, N + 1, 10_000))
    got_s, got_i = _chunked(store, queries.to(DEV), topk, bounds, [3, 1, 0, 2])
    np.testing.assert_array_equal(got_i, want_i)
    np.testing.assert_array_equal(got_s.view(np.uint32), want_s.view(np.uint32))
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(got_s, got_i, S, topk)
    for q in range(Q):
        assert set(pos[q].tolist()) == set(got_i[q].tolist())


def test_prefix_pass_in_the_first_chunk_then_updates():
    # first chunk large enough for the prefix threshold pass (Q > 128, N >= 8 x 128 x topk)
    N, K, Q, topk = 70_000, 128, 300, 4
    store = _store(wl.gaussian_rows(N, K, seed=90))
    queries = wl.gaussian_rows(Q, K, seed=91).to(DEV)
    want_s, want_i = _single(store, queries, topk)
    got_s, got_i = _chunked(store, queries, topk, [0, 50_000, N], [0, 1])
    np.testing.assert_array_equal(got_i, want_i)
    np.testing.assert_array_equal(got_s.view(np.uint32), want_s.view(np.uint32))


@pytest.mark.parametrize("pinned,least", [(True, False), (False, False), (True, True)])
def test_host_store_streamed_in_chunks(pinned, least):
    N, K, Q, topk, chunk = 60_001, 256, 140, 10, 7_000
    store = _store(_rows_with_duplicates(N, K, 95))
    queries = wl.gaussian_rows(Q, K, seed=96).to(DEV)
    want_s, want_i = _single(store, queries, topk, least=least)
    host = store.cpu()
    if pinned:
        host = host.pin_memory()
    ws = bg.workspace_tensor(bg.bergson_score_topk_host_workspace(chunk, K, Q, topk), DEV)
    s = torch.full((Q, topk), float("nan"), dtype=torch.float32, device=DEV)
    i = torch.full((Q, topk), -7, dtype=torch.int64, device=DEV)
    copy_stream = torch.cuda.Stream() if pinned else None
    bg.bergson_score_topk_host(host, N, K, queries, topk, chunk, s, i, ws,
                               copy_stream=copy_stream, least=least)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    torch.cuda.synchronize()
    np.testing.assert_array_equal(i.cpu().numpy(), want_i)
    np.testing.assert_array_equal(np32(s).view(np.uint32), want_s.view(np.uint32))


@pytest.mark.parametrize("Q", [3, 200])
def test_fewer_usable_scores_than_topk(Q):
    # NaN rows never enter the result; with only 9 usable rows the result is
    # those 9 in order, then (-inf, -1).  Before the merge kept only real keys,
    # the empty-slot keys tying with the k-th could push real rows out.
    N, K, topk = 600, 128, 16
    X = wl.gaussian_rows(N, K, seed=98)
    store = _store(X)
    keep = np.array([3, 77, 128, 255, 256, 300, 411, 512, 599])
    dead = torch.ones(N, dtype=torch.bool)
    dead[torch.from_numpy(keep)] = False
    store[dead.to(DEV)] = float("nan")
    queries = wl.gaussian_rows(Q, K, seed=99).to(DEV)
    got_s, got_i = _single(store, queries, topk)
    S = orc.cosine_scores(store[torch.from_numpy(keep).to(DEV)].cpu().numpy(),
                          queries.cpu().numpy().astype(np.float64))
    for q in range(Q):
        # the 9 usable rows (order among near-ties follows the fp32 scores)
        assert sorted(got_i[q, :9].tolist()) == sorted(keep.tolist())
        want = dict(zip(keep.tolist(), S[q]))
        np.testing.assert_allclose(got_s[q, :9], [want[r] for r in got_i[q, :9]], atol=1e-3)
        assert np.all(np.diff(got_s[q, :9]) <= 0)
        assert np.all(got_i[q, 9:] == -1) and np.all(np.isneginf(got_s[q, 9:]))
    # the same through the chunked path, chunks smaller than topk included
    got_s2, got_i2 = _chunked(store, queries, topk, [0, 5, 130, 257, N], [2, 0, 3, 1])
    np.testing.assert_array_equal(got_i2, got_i)
    np.testing.assert_array_equal(got_s2.view(np.uint32), got_s.view(np.uint32))
