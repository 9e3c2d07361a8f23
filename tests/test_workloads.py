"""The synthetic inputs that stand in for the paper's data have the stated
shapes and statistics (host only).  Nothing here runs the method."""
import math

import numpy as np
import pytest
import torch

from paper_2606_11660_gb300 import workloads as wl


def _cos(a, b):
    a = a / a.norm(dim=-1, keepdim=True)
    b = b / b.norm(dim=-1, keepdim=True)
    return a @ b.T


def test_collection_workload_shapes():
    p = wl.PYTHIA160M
    assert (p.B, p.T, p.k, len(p.modules), p.k_total) == (32, 2048, 16, 48, 12288)
    assert sum(2 * (s.d_in + s.d_out) for s in p.modules) == 294_912          # bytes per token
    l = wl.LLAMA8B
    assert (l.B, l.T, l.k, len(l.modules)) == (8, 4096, 16, 160)
    shared = [s for s in l.modules if s.shares_input]
    assert len(shared) == 32 and all(s.d_in == 4096 and s.d_out == 14336 for s in shared)
    q = wl.PYTHIA1B4
    assert (q.B, q.T, q.k, len(q.modules)) == (16, 2048, 32, 96)
    s4 = wl.SCORE4M
    assert (s4.N, s4.K, s4.Q, s4.topk) == (4_000_000, 8192, 1024, 100)
    assert s4.N * s4.K * 2 == 65_536_000_000


def test_padding_mask_is_right_padding_of_about_ten_percent():
    p = wl.PYTHIA160M
    m = wl.right_padding_mask(4096, p.T, p.max_pad, seed=3).numpy().astype(bool)
    lengths = m.sum(axis=1)
    assert np.all(m[np.arange(4096), lengths - 1]) and not np.any(m & ~(np.arange(p.T)[None] < lengths[:, None]))
    pad = p.T - lengths
    assert pad.min() >= 0 and pad.max() <= p.max_pad
    # pad ~ U{0..409}: mean 204.5 (about 10% of 2048), variance 410^2/12 - ...
    assert abs(pad.mean() - p.max_pad / 2) < 5 * math.sqrt((p.max_pad + 1) ** 2 / 12 / 4096)
    assert 0.09 < 1 - lengths.mean() / p.T < 0.11


def test_inputs_are_seeded_and_scaled():
    spec = wl.ModuleSpec("m", 768, 3072)
    A1, G1 = wl.layer_inputs(spec, 2, 64, seed=5, input_scale=True)
    A2, G2 = wl.layer_inputs(spec, 2, 64, seed=5, input_scale=True)
    assert torch.equal(A1, A2) and torch.equal(G1, G2)
    assert A1.dtype == torch.bfloat16 and A1.shape == (2, 64, 768) and G1.shape == (2, 64, 3072)
    # N(0, 1/d): per-row squared norms near 1
    assert abs(A1.float().pow(2).sum(-1).mean().item() - 1.0) < 0.05
    assert abs(G1.float().pow(2).sum(-1).mean().item() - 1.0) < 0.05
    r, c = wl.second_moments(3072, 768, seed=1)
    assert r.min() >= 0.5 and r.max() <= 2.0 and c.min() >= 0.5 and c.max() <= 2.0


def test_planted_neighbours_stand_far_above_the_background():
    K, Q, per = 8192, 4, 100
    queries = wl.gaussian_rows(Q, K, seed=8)
    planted = wl.planted_rows(queries, per, seed=9).reshape(Q, per, K)
    cos = torch.stack([_cos(queries[q:q + 1], planted[q])[0] for q in range(Q)])
    assert cos.min() > 0.30 and cos.max() < 0.92          # t / sqrt(1 + t^2), t in [0.35, 2]
    background = wl.gaussian_rows(100_000, K, seed=10)
    bmax = _cos(queries, background).abs().max().item()
    assert bmax < 0.07                                     # ~sqrt(2 ln 2e5 / K) = 0.055
    pos = wl.planted_positions(4_000_000, 1024, 100, seed=11)
    assert pos.shape == (1024, 100) and len(torch.unique(pos)) == 1024 * 100
    assert pos.min() >= 0 and pos.max() < 4_000_000
