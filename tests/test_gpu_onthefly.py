"""GPU parity of on-the-fly scoring (bergson_score_grads) against the oracle."""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import make_layers, np32, run_project

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _scores(x, y, unit, ld_pad=0):
    B, K = x.shape
    Q = y.shape[0]
    ws = bg.workspace_tensor(bg.bergson_score_grads_workspace(B, K, Q), DEV)
    out = torch.full((B, Q + ld_pad), float("nan"), dtype=torch.float32, device=DEV)
    bg.bergson_score_grads(x, B, K, y, unit, out, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(out)


@pytest.mark.parametrize("B,K,Q", [(37, 12288, 130), (1, 36, 1), (64, 520, 1000), (3, 4096, 7),
                                   (300, 1000, 200), (16, 4, 129),
                                   # K slices of 16 to 26 steps of 32 columns: accumulation
                                   # chains of 8 steps, then 1 or 2, over 150+ tiles of y
                                   (64, 1056, 40000), (20, 4128, 39000), (33, 8224, 515)])
@pytest.mark.parametrize("unit", [True, False])
def test_random_rows(B, K, Q, unit):
    g = wl.generator(B * 31 + K + Q, "cpu")
    x = torch.randn((B, K), generator=g) * 0.05
    y = torch.randn((Q, K), generator=g) * 3.0
    if B > 2:
        x[2] = 0.0
    got = _scores(x.to(DEV), y.to(DEV), unit, ld_pad=5)
    want = orc.onthefly_scores(x.numpy(), y.numpy(), unit)
    assert np.all(np.isnan(got[:, Q:]))
    scale = 1.0 if unit else np.abs(want).max()
    np.testing.assert_allclose(got[:, :Q], want, atol=2e-6 * scale, rtol=0)


def test_padded_leading_dimensions():
    g = wl.generator(5, "cpu")
    xb = torch.randn((10, 260), generator=g)
    yb = torch.randn((9, 300), generator=g)
    x, y = xb[:, :256].to(DEV), yb[:, :256].to(DEV)      # row strides 260 and 300
    got = _scores(x, y, True)
    want = orc.onthefly_scores(xb[:, :256].numpy(), yb[:, :256].numpy(), True)
    np.testing.assert_allclose(got, want, atol=2e-6, rtol=0)


def test_end_to_end_tiny_workload():
    cfg = wl.TINY
    gl, ol, ld = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], rc=True)
    train = run_project(gl, cfg.B, cfg.T, None, ld)
    gq, oq, _ = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], data_seed=1, rc=True)
    for a, b in zip(gq, gl):
        a.seed_in, a.seed_out, a.r, a.c = b.seed_in, b.seed_out, b.r, b.c
    for a, b in zip(oq, ol):
        a.seed_in, a.seed_out, a.r, a.c = b.seed_in, b.seed_out, b.r, b.c
    queries = run_project(gq, cfg.B, cfg.T, None, ld)
    got = _scores(train, queries, True)
    want = orc.onthefly_scores(orc.project_grads(ol, None, ld), orc.project_grads(oq, None, ld))
    np.testing.assert_allclose(got, want, atol=1e-4, rtol=0)


def test_deterministic():
    g = wl.generator(6, "cpu")
    x = torch.randn((32, 12288), generator=g).to(DEV)
    y = torch.randn((1024, 12288), generator=g).to(DEV)
    a = _scores(x, y, True)
    b = _scores(x, y, True)
    assert np.array_equal(a, b)


@pytest.mark.parametrize("B,K", [(40, 1000), (1, 128), (257, 520)])
def test_precondition_rows_random_matrix(B, K):
    """M x_b for a dense random M, against fp64: the same skinny product with y = M."""
    g = wl.generator(B + K, "cpu")
    x = torch.randn((B, K), generator=g)
    M = torch.randn((K, K), generator=g) / np.sqrt(K)
    M = (M + M.T) / 2                       # the entry point's contract: M symmetric
    ws = bg.workspace_tensor(bg.bergson_score_grads_workspace(B, K, K), DEV)
    out = torch.full((B, K), float("nan"), dtype=torch.float32, device=DEV)
    bg.bergson_precondition_rows(x.to(DEV), B, K, M.to(DEV), out, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    want = x.numpy().astype(np.float64) @ M.numpy().astype(np.float64).T
    np.testing.assert_allclose(np32(out), want, atol=2e-6 * np.abs(want).max(), rtol=0)
