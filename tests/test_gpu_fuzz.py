"""Seeded random calls of the projection, the scorer and the skinny GEMM
against the oracle.

Each case draws module widths (multiples of 8), (k_in, k_out) pairs, B, T,
a right-padding-plus-holes mask, optional Adafactor moments, optional bias
blocks and layers that share an input tensor, so that the planner's
combinations (fused slots, pieces, shared-input units, mixed-k groups) are
exercised together.  Sizes stay small enough for the fp64 oracle.
"""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import check_topk, make_layers, np32, rel_frobenius, run_project

pytestmark = pytest.mark.gpu
DEV = "cuda"
TIGHT = 1e-4
KS = (16, 32, 64)


def _case(seed):
    rng = np.random.default_rng(1000 + seed)
    n_mod = int(rng.integers(1, 5))
    specs, kp = [], []
    for m in range(n_mod):
        share = m > 0 and rng.random() < 0.3
        d_in = specs[-1].d_in if share else int(rng.integers(1, 65)) * 8
        d_out = int(rng.integers(1, 97)) * 8
        specs.append(wl.ModuleSpec(f"m{m}", d_in, d_out, share))
        kp.append((int(rng.choice(KS)), int(rng.choice(KS))))
    B = int(rng.integers(1, 7))
    T = int(rng.integers(1, 600))
    rc = bool(rng.random() < 0.5)
    bias = [bool(rng.random() < 0.3) for _ in range(n_mod)]
    masked = bool(rng.random() < 0.7)
    return specs, kp, B, T, rc, bias, masked, rng


@pytest.mark.parametrize("seed", range(24))
def test_random_projection_calls(seed):
    specs, kp, B, T, rc, bias, masked, rng = _case(seed)
    gl, ol, ld = make_layers(specs, B, T, kp, base_seed=seed, data_seed=seed, rc=rc,
                             input_scale=True)
    off = ld
    for m, on in enumerate(bias):
        if on:
            gl[m].bias_col_offset = ol[m].bias_col_offset = off
            off += kp[m][1]
    mask = None
    if masked:
        keep = rng.integers(0, T + 1, size=B)
        mnp = (np.arange(T)[None, :] < keep[:, None]).astype(np.uint8)
        holes = rng.random((B, T)) < 0.1
        mnp[holes] = 0
        mask = torch.from_numpy(mnp)
    out = run_project(gl, B, T, None if mask is None else mask.to(DEV), off)
    want = orc.project_grads(ol, None if mask is None else mask.numpy(), off)
    got = np32(out).astype(np.float64)
    nz = np.linalg.norm(want, axis=1) > 0
    assert rel_frobenius(got[nz], want[nz]).max() <= TIGHT, (seed, bg.bergson_debug_project_plan(gl, B, T))
    np.testing.assert_array_equal(got[~nz], 0.0)


def _store(rows):
    N, K = rows.shape
    store = torch.empty((N, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(rows.to(DEV), N, K, True, store, 0)
    return store


@pytest.mark.parametrize("seed", range(12))
def test_random_score_calls(seed):
    """Random N, K, Q, topk (exact duplicates give ties across tiles)."""
    rng = np.random.default_rng(2000 + seed)
    N = int(rng.integers(1, 20000))
    K = int(rng.integers(1, 129)) * 8
    Q = int(rng.integers(1, 300))
    topk = int(rng.integers(1, min(N, 200) + 1))
    g = wl.generator(3000 + seed, "cpu")
    rows = torch.randn((N, K), generator=g)
    if N > 10:
        dup = rng.integers(0, N, size=(min(N // 4, 64), 2))
        rows[torch.as_tensor(dup[:, 1])] = rows[torch.as_tensor(dup[:, 0])]
    queries = torch.randn((Q, K), generator=g)
    store = _store(rows)
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(N, K, Q, topk), DEV)
    s = torch.empty((Q, topk), dtype=torch.float32, device=DEV)
    i = torch.empty((Q, topk), dtype=torch.int64, device=DEV)
    bg.bergson_score_topk(store, N, K, queries.to(DEV), topk, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    S = orc.cosine_scores(store.float().cpu().numpy().astype(np.float64),
                          queries.numpy().astype(np.float64))
    check_topk(np32(s), i.cpu().numpy(), S, topk)


@pytest.mark.parametrize("seed", range(8))
def test_random_onthefly_calls(seed):
    rng = np.random.default_rng(4000 + seed)
    B = int(rng.integers(1, 300))
    K = int(rng.integers(1, 800)) * 4
    Q = int(rng.integers(1, 600))
    unit = bool(rng.random() < 0.5)
    g = wl.generator(5000 + seed, "cpu")
    x = torch.randn((B, K), generator=g)
    y = torch.randn((Q, K), generator=g)
    ws = bg.workspace_tensor(bg.bergson_score_grads_workspace(B, K, Q), DEV)
    out = torch.empty((B, Q), dtype=torch.float32, device=DEV)
    bg.bergson_score_grads(x.to(DEV), B, K, y.to(DEV), unit, out, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    want = orc.onthefly_scores(x.numpy(), y.numpy(), unit)
    xa, ya = np.abs(x.numpy().astype(np.float64)), np.abs(y.numpy().astype(np.float64))
    bound = xa @ ya.T
    if unit:
        bound = bound / np.linalg.norm(xa, axis=1)[:, None] / np.linalg.norm(ya, axis=1)[None, :]
    assert np.all(np.abs(np32(out) - want) <= 2e-6 * bound + 1e-12)
