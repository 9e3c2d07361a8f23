"""Shared helpers for the parity tests (test code only)."""
from __future__ import annotations

import importlib.util
import os

import numpy as np
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl


def np32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


def make_layers(specs, B, T, k_pairs, base_seed=0, data_seed=0, rc=False, input_scale=False,
                device="cuda", kind=bg.BERGSON_PROJ_GAUSSIAN):
    """Seeded inputs for several modules; returns (gpu Layers, oracle Layers, ld_out)."""
    gl, ol = [], []
    off = 0
    ins = wl.module_inputs(specs, B, T, [data_seed * 1000 + m for m in range(len(specs))],
                           input_scale=input_scale)
    for m, (spec, (ki, ko), (A, G)) in enumerate(zip(specs, k_pairs, ins)):
        r = c = None
        if rc:
            r, c = wl.second_moments(spec.d_out, spec.d_in, seed=data_seed * 1000 + 500 + m)
        s_in, s_out = orc.module_seeds(base_seed, m)
        A_dev = gl[-1].A if spec.shares_input else A.to(device)   # one device tensor when shared
        gl.append(bg.Layer(A_dev, G.to(device), ki, ko, s_in, s_out,
                           None if r is None else r.to(device), None if c is None else c.to(device),
                           off, kind))
        ol.append(orc.Layer(np32(A), np32(G), ki, ko, s_in, s_out,
                            None if r is None else r.numpy().astype(np.float64),
                            None if c is None else c.numpy().astype(np.float64), off, kind))
        off += ki * ko
    return gl, ol, off


def run_project(layers, B, T, mask, ld_out, device="cuda"):
    ws = bg.workspace_tensor(bg.bergson_project_grads_workspace(layers, B, T), device)
    out = torch.full((B, ld_out), float("nan"), dtype=torch.float32, device=device)
    bg.bergson_project_grads(layers, B, T, mask, out, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return out


def rel_frobenius(got: np.ndarray, want: np.ndarray) -> np.ndarray:
    """Per-row ||got - want|| / ||want|| (rows with ||want|| = 0 use the absolute error)."""
    d = np.linalg.norm(got - want, axis=1)
    n = np.linalg.norm(want, axis=1)
    return np.where(n > 0, d / np.where(n > 0, n, 1.0), d)


def check_topk(got_s, got_i, S, k, score_atol=1e-3, tie=1e-4):
    """GPU top-k against oracle scores S [Q, N]: exact sets except near-ties, scores close."""
    Q = S.shape[0]
    for q in range(Q):
        row = S[q]
        gi = got_i[q].astype(np.int64)
        gs = got_s[q].astype(np.float64)
        assert len(set(gi.tolist())) == k, "duplicate indices"
        assert np.all(gi >= 0) and np.all(gi < row.shape[0])
        assert np.all(np.diff(gs) <= 0), "scores not descending"
        np.testing.assert_allclose(gs, row[gi], atol=score_atol, rtol=0)
        order = np.lexsort((np.arange(row.shape[0]), -row))
        kth = row[order[k - 1]]
        must = set(order[:k][row[order[:k]] > kth + tie].tolist())
        assert must <= set(gi.tolist()), f"query {q}: missing clear top-k members"
        assert np.all(row[gi] >= kth - tie), f"query {q}: returned a row clearly below the k-th"


GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def golden_lines(name: str):
    """Non-comment lines of a fixture in tests/golden."""
    with open(os.path.join(GOLDEN, name)) as f:
        return [line.strip() for line in f if line.strip() and not line.startswith("#")]


def load_make_golden():
    """tests/golden/make_golden.py as a module (it calls only the oracle)."""
    spec = importlib.util.spec_from_file_location("make_golden", os.path.join(GOLDEN, "make_golden.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod
