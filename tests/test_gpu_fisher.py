"""GPU parity of the empirical-Fisher preconditioner against the fp64 oracle."""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import make_layers, np32, run_project

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _fit(x):
    n, K = x.shape
    R = torch.full((K, K), float("nan"), device=DEV)
    ws = bg.workspace_tensor(bg.bergson_fisher_fit_workspace(n, K), DEV)
    bg.bergson_fisher_fit(x, n, K, R, ws)
    return R


def _power(R1, R2, lam, damping, power, iters=30):
    K = R1.shape[0]
    M = torch.full((K, K), float("nan"), device=DEV)
    ws = bg.workspace_tensor(bg.bergson_fisher_preconditioner_workspace(K), DEV)
    bg.bergson_fisher_preconditioner(R1, R2, K, lam, damping, power, iters, M, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return M


def _rel(a, b):
    return np.linalg.norm(a - b) / np.linalg.norm(b)


@pytest.mark.parametrize("n,K", [(100, 256), (37, 260), (600, 132)])
def test_fisher_fit(n, K):
    g = wl.generator(n + K, "cpu")
    x = torch.randn((n, K), generator=g) * torch.linspace(0.1, 2.0, K)
    R = np32(_fit(x.to(DEV))).astype(np.float64)
    assert bg.bergson_sync_status() == bg.BERGSON_OK
    want = orc.fisher_fit(x.numpy())
    assert _rel(R, want) < 1e-5


@pytest.mark.parametrize("power", [bg.BERGSON_FISHER_INV_SQRT, bg.BERGSON_FISHER_INV])
def test_mixed_preconditioner(power):
    g = wl.generator(21, "cpu")
    K = 256
    x1 = torch.randn((300, K), generator=g) * torch.linspace(0.2, 3.0, K)
    x2 = torch.randn((120, K), generator=g)
    R1, R2 = _fit(x1.to(DEV)), _fit(x2.to(DEV))
    M = np32(_power(R1, R2, 0.3, 0.1, power)).astype(np.float64)
    Rm = orc.fisher_mix(orc.fisher_fit(x1.numpy()), orc.fisher_fit(x2.numpy()), 0.3, 0.1)
    p = -0.5 if power == bg.BERGSON_FISHER_INV_SQRT else -1.0
    want = orc.fisher_power(Rm, p)
    assert _rel(M, want) < 1e-3
    if power == bg.BERGSON_FISHER_INV_SQRT:
        np.testing.assert_allclose(M @ Rm @ M, np.eye(K), atol=2e-3)
    else:
        np.testing.assert_allclose(M @ Rm, np.eye(K), atol=2e-3)


def test_single_fisher_low_rank_with_damping():
    g = wl.generator(22, "cpu")
    K = 384
    x = torch.randn((64, K), generator=g)                 # rank 64 < K: damping is essential
    R = _fit(x.to(DEV))
    M = np32(_power(R, None, 1.0, 0.5, bg.BERGSON_FISHER_INV_SQRT, 40)).astype(np.float64)
    want = orc.fisher_power(orc.fisher_mix(orc.fisher_fit(x.numpy()), None, 1.0, 0.5), -0.5)
    assert _rel(M, want) < 1e-3


def test_precondition_rows_and_whitened_scores():
    cfg = wl.TINY
    gl, ol, ld = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], rc=True)
    out = run_project(gl, cfg.B, cfg.T, None, ld)            # [8, 256] projected gradients
    g = wl.generator(23, "cpu")
    fit_rows = torch.randn((500, ld), generator=g) * 0.01
    R = _fit(fit_rows.to(DEV))
    M = _power(R, None, 1.0, 0.05, bg.BERGSON_FISHER_INV_SQRT)
    ws = bg.workspace_tensor(bg.bergson_score_grads_workspace(cfg.B, ld, ld), DEV)
    pre = torch.full((cfg.B, ld), float("nan"), device=DEV)
    bg.bergson_precondition_rows(out, cfg.B, ld, M, pre, ws)
    store = torch.empty((cfg.B, ld), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(pre, cfg.B, ld, True, store, 0)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    M_o = orc.fisher_power(orc.fisher_mix(orc.fisher_fit(fit_rows.numpy()), None, 1.0, 0.05), -0.5)
    want = orc.precondition_rows(orc.project_grads(ol, None, ld), M_o)
    got = np32(pre).astype(np.float64)
    assert _rel(got, want) < 2e-3
    want_store, _ = orc.build_store(want)
    np.testing.assert_allclose(store.float().cpu().numpy(), want_store.astype(np.float32), atol=2e-3)


def test_newton_schulz_stays_converged_on_ill_conditioned_R():
    # rank 64 of K = 1024 with damping 0.01: condition number ~2,500 (far above
    # the ~34 at which taking Y T^T for Y T made the converged iterates
    # diverge).  Every residual after convergence stays at the fp32 floor.
    g = wl.generator(25, "cpu")
    K = 1024
    x = torch.randn((64, K), generator=g)
    R = _fit(x.to(DEV))
    M = torch.full((K, K), float("nan"), device=DEV)
    ws = bg.workspace_tensor(bg.bergson_fisher_preconditioner_workspace(K), DEV)
    done, res = bg.bergson_fisher_preconditioner_tol(R, None, K, 1.0, 0.01,
                                                     bg.BERGSON_FISHER_INV_SQRT, 60, 0.0, M, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    assert done == 60 and len(res) == 61
    first = next(i for i, r in enumerate(res) if r <= 1e-4)
    assert first <= 40 and max(res[first:]) <= 1e-4, res
    want = orc.fisher_power(orc.fisher_mix(orc.fisher_fit(x.numpy()), None, 1.0, 0.01), -0.5)
    assert _rel(np32(M).astype(np.float64), want) < 1e-3
    # the stopping rule ends at the first iterate within tol, with the same M
    M2 = torch.full((K, K), float("nan"), device=DEV)
    done2, res2 = bg.bergson_fisher_preconditioner_tol(R, None, K, 1.0, 0.01,
                                                       bg.BERGSON_FISHER_INV_SQRT, 60, 1e-4, M2,
                                                       ws)
    assert done2 == first and len(res2) == first + 1 and res2[-1] <= 1e-4
    assert _rel(np32(M2).astype(np.float64), want) < 1e-3
