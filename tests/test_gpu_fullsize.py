"""Full-size parity: each workload at its real sizes and launch shape, checked
on sampled outputs the fp64 oracle can compute one at a time, and through
properties that hold at any size.

* pythia160m: the exact setup bench.py times (48 modules in one call, B=32,
  T=2048, ~10% padding); sampled (example, module) blocks and one whole
  unit-normalised store row against the oracle.
* pythia1b4 / llama8b: one transformer block per call at full B and T (the
  streamed launch shape), sampled blocks against the oracle, every stored row
  of unit norm.
* score4m: the full 4M x 8192 store with planted neighbours for sampled
  queries (known exact top-100 sets), returned scores re-derived by the
  oracle from the returned rows.
"""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import np32

pytestmark = [pytest.mark.gpu, pytest.mark.slow]
DEV = "cuda"
TIGHT = 1e-4


def _oracle_block(A_b, G_b, m_b, k_in, k_out, s_in, s_out, r=None, c=None):
    L = orc.Layer(np32(A_b)[None], np32(G_b)[None], k_in, k_out, s_in, s_out,
                  None if r is None else np32(r).astype(np.float64),
                  None if c is None else np32(c).astype(np.float64))
    return orc.project_module(L, None if m_b is None else m_b[None])[0]


def test_pythia160m_bench_setup_sampled_blocks():
    import bench
    cfg, layers, mask, ws, out = bench.collection_setup(torch.device(DEV))
    bg.bergson_project_grads(layers, cfg.B, cfg.T, mask, out, ws)
    store = torch.empty((cfg.B, cfg.k_total), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(out, cfg.B, cfg.k_total, True, store, 0)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    got = np32(out).astype(np.float64)
    mask_np = mask.cpu().numpy()
    blk = cfg.k * cfg.k
    for b, m in [(0, 0), (31, 47), (7, 1), (19, 46), (12, 22)]:
        ly = layers[m]
        want = _oracle_block(ly.A[b], ly.G[b], mask_np[b], cfg.k, cfg.k, ly.seed_in, ly.seed_out)
        g = got[b, m * blk:(m + 1) * blk]
        assert np.linalg.norm(g - want) / np.linalg.norm(want) <= TIGHT, (b, m)
    # one whole row: all 48 blocks, then the unit-normalised fp16 store row
    b = 5
    row = np.concatenate([
        _oracle_block(ly.A[b], ly.G[b], mask_np[b], cfg.k, cfg.k, ly.seed_in, ly.seed_out)
        for ly in layers])
    assert np.linalg.norm(got[b] - row) / np.linalg.norm(row) <= TIGHT
    want_store, _ = orc.build_store(row[None])
    g16 = store[b].float().cpu().numpy()
    w16 = want_store[0].astype(np.float64)
    # fp16 rounding of a row that itself carries ~1e-5 relative error: within
    # one fp16 ulp of the largest entry everywhere, 1e-3 relative overall
    assert np.max(np.abs(g16 - w16)) <= 2.0 ** -10 * np.abs(w16).max()
    assert np.linalg.norm(g16 - w16) / np.linalg.norm(w16) <= 1e-3
    norms = np.linalg.norm(store.float().cpu().numpy().astype(np.float64), axis=1)
    np.testing.assert_allclose(norms, 1.0, atol=1e-3)


@pytest.mark.parametrize("name,blocks,samples", [
    ("pythia1b4", [0, 23], [(0, 0), (15, 3), (9, 2)]),
    ("llama8b", [0, 31], [(0, 2), (7, 4)]),
])
def test_streamed_block_calls_sampled_blocks(name, blocks, samples):
    cfg = wl.COLLECT_WORKLOADS[name]
    k = cfg.k
    blk = k * k
    nmod = cfg.modules_per_block
    ld = cfg.k_total
    out = torch.full((cfg.B, ld), float("nan"), dtype=torch.float32, device=DEV)
    ws = None
    for bi in blocks:
        specs = cfg.block_modules(bi)
        layers = []
        ins = wl.module_inputs(specs, cfg.B, cfg.T, [20_000 + bi * nmod + j for j in range(nmod)],
                               device=DEV, input_scale=True)
        for j, (spec, (A, G)) in enumerate(zip(specs, ins)):
            m = bi * nmod + j
            r = c = None
            if cfg.second_moments:
                r, c = wl.second_moments(spec.d_out, spec.d_in, seed=30_000 + m, device=DEV)
            s_in, s_out = bg.bergson_module_seeds(0, m)
            layers.append(bg.Layer(A, G, k, k, s_in, s_out, r, c, cfg.col_offset(m)))
        need = bg.bergson_project_grads_workspace(layers, cfg.B, cfg.T)
        if ws is None or ws.numel() < need:
            ws = bg.workspace_tensor(need, DEV)
        bg.bergson_project_grads(layers, cfg.B, cfg.T, None, out, ws)
        assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
        got = np32(out).astype(np.float64)
        for b, j in samples:
            ly = layers[j]
            m = bi * nmod + j
            want = _oracle_block(ly.A[b], ly.G[b], None, k, k, ly.seed_in, ly.seed_out, ly.r, ly.c)
            g = got[b, m * blk:(m + 1) * blk]
            assert np.linalg.norm(g - want) / np.linalg.norm(want) <= TIGHT, (name, bi, b, j)
        del layers, ins
        torch.cuda.empty_cache()
    # the written blocks form rows that the store normalises to unit length
    cols = np.concatenate([np.arange(bi * nmod * blk, (bi + 1) * nmod * blk) for bi in blocks])
    sub = out[:, torch.as_tensor(cols, device=DEV)].contiguous()
    store = torch.empty((cfg.B, sub.shape[1]), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(sub, cfg.B, sub.shape[1], True, store, 0)
    torch.cuda.synchronize()
    np.testing.assert_allclose(np.linalg.norm(store.float().cpu().numpy(), axis=1), 1.0, atol=1e-3)


def test_score4m_planted_sampled_queries():
    sw = wl.SCORE4M
    N, K, Q, topk = sw.N, sw.K, sw.Q, sw.topk
    store = torch.empty((N, K), dtype=torch.float16, device=DEV)
    g = wl.generator(7, DEV)
    for n0 in range(0, N, 1 << 17):
        n1 = min(N, n0 + (1 << 17))
        rows = torch.randn((n1 - n0, K), generator=g, device=DEV)
        bg.bergson_build_store(rows, n1 - n0, K, True, store, n0)
    del rows
    queries = wl.gaussian_rows(Q, K, seed=8, device=DEV)
    sampled = [0, 1, 255, 256, 700, 1023]          # across all four query groups
    qs = queries[sampled]
    pos = wl.planted_positions(N, len(sampled), topk, seed=9)
    planted = wl.planted_rows(qs, topk, seed=10)
    pstore = torch.empty((planted.shape[0], K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(planted, planted.shape[0], K, True, pstore, 0)
    store[pos.reshape(-1).to(DEV)] = pstore
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(N, K, Q, topk), DEV)
    s = torch.empty((Q, topk), dtype=torch.float32, device=DEV)
    i = torch.empty((Q, topk), dtype=torch.int64, device=DEV)
    bg.bergson_score_topk(store, N, K, queries, topk, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    s_np, i_np = np32(s), i.cpu().numpy()
    for j, q in enumerate(sampled):
        assert set(i_np[q].tolist()) == set(pos[j].tolist()), q
        rows = store[i[q]].float().cpu().numpy().astype(np.float64)
        qv = np32(queries[q]).astype(np.float64)
        want = rows @ (qv / np.linalg.norm(qv))
        np.testing.assert_allclose(s_np[q], want, atol=1e-3, rtol=0)
        assert np.all(np.diff(s_np[q]) <= 0)
    # every query: indices distinct and valid, scores descending and finite
    assert np.all((i_np >= 0) & (i_np < N))
    assert all(len(set(r.tolist())) == topk for r in i_np)
    assert np.all(np.diff(s_np, axis=1) <= 0) and np.all(np.isfinite(s_np))
    # two unplanted queries: re-derive the returned scores, and check that no row
    # of a random 262,144-row sample outside the result beats the k-th score.
    sample = torch.randperm(N, generator=wl.generator(11, "cpu"))[: 1 << 18].to(DEV)
    srows = store[sample].float().cpu().numpy().astype(np.float64)
    for q in (5, 900):
        qv = np32(queries[q]).astype(np.float64)
        qv /= np.linalg.norm(qv)
        rows = store[i[q]].float().cpu().numpy().astype(np.float64)
        np.testing.assert_allclose(s_np[q], rows @ qv, atol=1e-3, rtol=0)
        outside = ~np.isin(sample.cpu().numpy(), i_np[q])
        assert np.max((srows @ qv)[outside]) <= s_np[q, -1] + 1e-4
