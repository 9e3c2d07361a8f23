"""Edge cases of the launch logic: multi-pass scoring, the largest top-k,
extreme projection shapes and many layers."""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import check_topk, make_layers, np32, rel_frobenius, run_project

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _score(store, queries, topk):
    N, K = store.shape
    Q = queries.shape[0]
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(N, K, Q, topk), DEV)
    s = torch.empty((Q, topk), dtype=torch.float32, device=DEV)
    i = torch.empty((Q, topk), dtype=torch.int64, device=DEV)
    bg.bergson_score_topk(store, N, K, queries, topk, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(s), i.cpu().numpy()


def _store(rows):
    N, K = rows.shape
    st = torch.empty((N, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(rows.to(DEV), N, K, True, st, 0)
    return st


def test_more_query_groups_than_sms():
    # 39,012 queries = 153 groups of 256 (> 152 SMs): the scorer runs in passes
    g = wl.generator(41, "cpu")
    N, K, Q, topk = 1000, 64, 39_012, 5
    store = _store(torch.randn((N, K), generator=g))
    queries = torch.randn((Q, K), generator=g)
    s, i = _score(store, queries.to(DEV), topk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    sample = np.r_[0:50, 38_900:Q]
    check_topk(s[sample], i[sample], S[sample], topk)


def test_largest_topk_multi_round_merge():
    g = wl.generator(42, "cpu")
    N, K, Q, topk = 60_000, 128, 300, 1024
    store = _store(torch.randn((N, K), generator=g))
    queries = torch.randn((Q, K), generator=g)
    s, i = _score(store, queries.to(DEV), topk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(s[:40], i[:40], S[:40], topk)


def test_single_token_single_example_and_wide_module():
    spec = wl.ModuleSpec("wide", 14336, 4096)
    gl, ol, ld = make_layers([spec], 1, 1, [(64, 64)], input_scale=True)
    out = run_project(gl, 1, 1, None, ld)
    want = orc.project_grads(ol, None, ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= 1e-4


def test_many_small_layers():
    specs = [wl.ModuleSpec(f"l{i}", 8 * (1 + i % 5), 8 * (1 + (i * 3) % 7)) for i in range(200)]
    gl, ol, ld = make_layers(specs, 2, 40, [(16, 16)] * 200, base_seed=3)
    out = run_project(gl, 2, 40, None, ld)
    want = orc.project_grads(ol, None, ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= 1e-4


@pytest.mark.parametrize("bad", [0.0, -1.0, float("nan")])
def test_nonpositive_second_moment_is_reported_by_the_device(bad):
    # r, c live on the device, so only the kernel that reads them can check
    # r, c > 0: it records BERGSON_EMOMENT in the status word, nothing faults,
    # and the context stays usable (the word is cleared once reported).
    spec = wl.ModuleSpec("lin", 64, 128)
    gl, ol, ld = make_layers([spec], 4, 50, [(16, 16)], rc=True)
    assert bg.bergson_sync_status() == bg.BERGSON_OK
    r_bad = gl[0].r.clone()
    r_bad[17] = bad
    bad_layer = bg.Layer(gl[0].A, gl[0].G, 16, 16, gl[0].seed_in, gl[0].seed_out, r_bad, gl[0].c,
                         0)
    ws = bg.workspace_tensor(bg.bergson_project_grads_workspace([bad_layer], 4, 50), DEV)
    out = torch.empty((4, ld), device=DEV)
    bg.bergson_project_grads([bad_layer], 4, 50, None, out, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_EMOMENT
    assert "second-moment" in bg.bergson_last_error()
    assert bg.bergson_sync_status() == bg.BERGSON_OK          # cleared once reported
    c_bad = gl[0].c.clone()
    c_bad[3] = bad
    P = torch.empty((spec.d_in, 16), device=DEV)
    bg.bergson_projection_matrix(gl[0].seed_in, spec.d_in, 16, bg.BERGSON_PROJ_GAUSSIAN, c_bad, P)
    assert bg.bergson_sync_status() == bg.BERGSON_EMOMENT
    # the same call with valid moments still matches the oracle afterwards
    out = run_project(gl, 4, 50, None, ld)
    want = orc.project_grads(ol, None, ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= 1e-4
