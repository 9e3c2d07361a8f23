"""The empirical-Fisher preconditioner at the size the benchmark times.

TrackStar's mixed empirical Fisher (Sec. 3.1; Fig. 2, Fisher fitting and
mixing), exactly as the benchmark's Fisher leg runs it: R fitted on 1,024
rows of N(0, I_12288) drawn on the device (seed 14), damping 0.1 (a rank-1,024
matrix that only the damping keeps invertible: its spectrum runs from 0.1 to
about 20), M = R^-1/2 by 20 coupled Newton-Schulz updates, applied to a
32-row batch that then goes into the fp16 store.  Every step is held to the
fp64 oracle on host copies of the same inputs; the oracle's R^-1/2 is an
eigendecomposition of the 12,288 x 12,288 matrix (a few minutes on the host
cores), computed once for the whole module.
"""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import np32, rel_frobenius

pytestmark = [pytest.mark.gpu, pytest.mark.slow]
DEV = "cuda"
K, N_FIT, B, ITERS, DAMPING = 12288, 1024, 32, 20, 0.1


@pytest.fixture(scope="module")
def fisher_case():
    fit = wl.gaussian_rows(N_FIT, K, seed=14, device=DEV)
    batch = wl.gaussian_rows(B, K, seed=24, device=DEV) * 0.01
    R = torch.full((K, K), float("nan"), device=DEV)
    M = torch.full((K, K), float("nan"), device=DEV)
    fws = bg.workspace_tensor(bg.bergson_fisher_fit_workspace(N_FIT, K), DEV)
    bg.bergson_fisher_fit(fit, N_FIT, K, R, fws)
    del fws
    pws = bg.workspace_tensor(bg.bergson_fisher_preconditioner_workspace(K), DEV)
    done, residuals = bg.bergson_fisher_preconditioner_tol(
        R, None, K, 1.0, DAMPING, bg.BERGSON_FISHER_INV_SQRT, ITERS, 0.0, M, pws)
    del pws
    aws = bg.workspace_tensor(bg.bergson_score_grads_workspace(B, K, K), DEV)
    pre = torch.full((B, K), float("nan"), device=DEV)
    bg.bergson_precondition_rows(batch, B, K, M, pre, aws)
    store = torch.full((B, K), float("nan"), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(pre, B, K, True, store, 0)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    got = {"R": np32(R).astype(np.float64), "M": np32(M).astype(np.float64),
           "pre": np32(pre).astype(np.float64), "store": np32(store).astype(np.float64),
           "done": done, "residuals": residuals}
    del R, M, aws, pre, store
    torch.cuda.empty_cache()
    x = np32(fit).astype(np.float64)
    R_o = orc.fisher_fit(x)
    M_o = orc.fisher_power(orc.fisher_mix(R_o, None, 1.0, DAMPING), -0.5)
    pre_o = orc.precondition_rows(np32(batch).astype(np.float64), M_o)
    store_o, _ = orc.build_store(pre_o)
    want = {"R": R_o, "M": M_o, "pre": pre_o, "store": store_o.astype(np.float64)}
    return got, want


def test_fit_matches_oracle(fisher_case):
    got, want = fisher_case
    R, R_o = got["R"], want["R"]
    # entry-wise, relative to the Cauchy-Schwarz scale sqrt(R_ii R_jj) of each entry
    d = np.sqrt(np.diag(R_o))
    err = np.abs(R - R_o) / np.outer(d, d)
    assert err.max() <= 1e-5, f"max entry error {err.max():.3e}"
    assert np.linalg.norm(R - R_o) / np.linalg.norm(R_o) <= 1e-5


def test_newton_schulz_converges_in_the_benchmarked_iterations(fisher_case):
    got, _ = fisher_case
    res = got["residuals"]
    assert got["done"] == ITERS and len(res) == ITERS + 1
    print("Newton-Schulz residuals ||I - Z Y||_F / sqrt(K):", ", ".join(f"{r:.2e}" for r in res))
    assert res[-1] <= 1e-3 * res[0]
    assert res[-1] <= 1e-4


def test_inverse_sqrt_matches_oracle(fisher_case):
    got, want = fisher_case
    rel = np.linalg.norm(got["M"] - want["M"]) / np.linalg.norm(want["M"])
    print(f"relative Frobenius error of M: {rel:.3e}")
    assert rel <= 1e-3


def test_preconditioned_rows_and_store_match_oracle(fisher_case):
    got, want = fisher_case
    err = rel_frobenius(got["pre"], want["pre"])
    assert err.max() <= 2e-3, f"max row error {err.max():.3e}"
    np.testing.assert_allclose(got["store"], want["store"], atol=2e-3, rtol=0)
