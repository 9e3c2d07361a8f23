"""GPU parity of per-token scores (bergson_token_scores) against the oracle."""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import make_layers, np32, run_project

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _tokens(layers, B, T, mask, queries):
    Q = queries.shape[0]
    ws = bg.workspace_tensor(bg.bergson_token_scores_workspace(layers, B, T, Q), DEV)
    out = torch.full((Q, B, T), float("nan"), dtype=torch.float32, device=DEV)
    bg.bergson_token_scores(layers, B, T, mask, queries, out, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(out).astype(np.float64)


def _close(got, want, rel=1e-4):
    scale = np.abs(want).max(axis=(1, 2), keepdims=True)
    assert np.all(np.abs(got - want) <= rel * scale + 1e-12)


def test_tiny_workload_token_scores():
    cfg = wl.TINY
    gl, ol, ld = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], rc=True)
    g = wl.generator(3, "cpu")
    queries = torch.randn((3, ld), generator=g)
    got = _tokens(gl, cfg.B, cfg.T, None, queries.to(DEV))
    want = orc.token_scores(ol, None, queries.numpy())
    _close(got, want)


def test_multi_module_mask_ragged_mixed_k():
    specs = [wl.ModuleSpec("a", 64, 200), wl.ModuleSpec("b", 136, 64), wl.ModuleSpec("c", 96, 72)]
    kp = [(16, 16), (32, 16), (16, 32)]
    B, T = 3, 300
    gl, ol, ld = make_layers(specs, B, T, kp, base_seed=4, data_seed=2, rc=True)
    g = wl.generator(7, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.25).to(torch.uint8)
    mask[1, 128:256] = 0
    mask[2] = 0
    queries = torch.randn((8, ld + 16), generator=g)       # padded query rows
    got = _tokens(gl, B, T, mask.to(DEV), queries.to(DEV))
    want = orc.token_scores(ol, mask.numpy(), queries.numpy())
    _close(got, want)
    assert np.all(got[:, mask.numpy() == 0] == 0.0)
    # summed over tokens: the per-sequence inner product
    seq = np32(run_project(gl, B, T, mask.to(DEV), ld)).astype(np.float64)
    np.testing.assert_allclose(got.sum(axis=2), queries[:, :ld].numpy() @ seq.T,
                               rtol=1e-4, atol=1e-4 * np.abs(got.sum(axis=2)).max())


def test_shared_input_layers_token_scores():
    """Token mode with layers that read one A tensor: their items run from a
    work table (side by side); per-token scores still match the oracle."""
    specs = [wl.ModuleSpec("gate", 256, 512), wl.ModuleSpec("up", 256, 512, True),
             wl.ModuleSpec("down", 512, 256)]
    B, T = 3, 300
    gl, ol, ld = make_layers(specs, B, T, [(16, 16)] * 3, base_seed=6, data_seed=5, rc=True,
                             input_scale=True)
    assert gl[1].A.data_ptr() == gl[0].A.data_ptr()
    assert bg.bergson_debug_project_plan(gl, B, T)[3] == 2
    g = wl.generator(8, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.2).to(torch.uint8)
    queries = torch.randn((4, ld), generator=g)
    got = _tokens(gl, B, T, mask.to(DEV), queries.to(DEV))
    want = orc.token_scores(ol, mask.numpy(), queries.numpy())
    _close(got, want)


def test_query_limit_is_enforced():
    spec = wl.ModuleSpec("lin", 64, 64)
    gl, _, ld = make_layers([spec], 1, 8, [(64, 64)])
    queries = torch.zeros((257, ld), device=DEV)
    ws = bg.workspace_tensor(1 << 24, DEV)
    out = torch.empty((257, 1, 8), device=DEV)
    with pytest.raises(bg.BergsonError) as e:
        bg.bergson_token_scores(gl, 1, 8, None, queries, out, ws)
    assert e.value.status == bg.BERGSON_EUNSUPPORTED


@pytest.mark.parametrize("Q", [17, 70, 256])
def test_many_queries_stream_through_shared_memory_in_blocks(Q):
    # more queries than one shared-memory block for every (k_in, k_out): the
    # blocks (16 queries of 16x16, 9 of 32x32, 4 of 64x64) are streamed per
    # tile group, the last one ragged; one pass over A and G serves them all
    specs = [wl.ModuleSpec("a", 64, 200), wl.ModuleSpec("b", 136, 64), wl.ModuleSpec("c", 96, 72)]
    kp = [(16, 16), (32, 32), (64, 64)]
    B, T = 2, 300
    gl, ol, ld = make_layers(specs, B, T, kp, base_seed=9, data_seed=7, rc=True)
    g = wl.generator(10 + Q, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.2).to(torch.uint8)
    queries = torch.randn((Q, ld), generator=g)
    got = _tokens(gl, B, T, mask.to(DEV), queries.to(DEV))
    want = orc.token_scores(ol, mask.numpy(), queries.numpy())
    _close(got, want)
    assert np.all(got[:, mask.numpy() == 0] == 0.0)


@pytest.mark.slow
def test_pythia160m_full_size_token_scores():
    import bench
    cfg, layers, mask, _, _ = bench.collection_setup(torch.device(DEV))
    K = cfg.k_total
    Q = 64
    queries = wl.gaussian_rows(Q, K, seed=13, device=DEV)
    got = _tokens(layers, cfg.B, cfg.T, mask, queries)
    mask_np = mask.cpu().numpy()
    assert np.all(got[:, mask_np == 0] == 0.0)
    # sampled tokens of two examples against the explicit per-token oracle
    for b in (0, 31):
        valid = np.flatnonzero(mask_np[b])
        pick = np.zeros((1, cfg.T), np.uint8)
        pick[0, valid[[0, 1, len(valid) // 2, len(valid) - 1]]] = 1
        ol = [orc.Layer(np32(ly.A[b])[None], np32(ly.G[b])[None], cfg.k, cfg.k, ly.seed_in,
                        ly.seed_out, col_offset=ly.out_col_offset) for ly in layers]
        want = orc.token_scores(ol, pick, np32(queries).astype(np.float64))[:, 0, :]
        sel = pick[0] == 1
        scale = np.abs(got[:, b, :]).max(axis=1, keepdims=True)
        assert np.all(np.abs(got[:, b, sel] - want[:, sel]) <= 1e-4 * scale)
