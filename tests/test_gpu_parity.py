"""GPU parity: the CUDA path (through the C ABI) against the fp64 CPU oracle.

Tolerances follow the stated bar: projected gradients within 2e-3 max
per-example relative Frobenius error, scores within 1e-3 absolute, top-k index
sets exact except among scores within 1e-4 of the k-th.  The hi/lo bf16 split
of the projection predicts errors near 1e-5, so a second, tighter bound
(1e-4) guards against a silently dropped low-order term.
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
BAR = 2e-3
TIGHT = 1e-4


@pytest.mark.parametrize("seed,d,k,moment", [(0, 64, 16, False), (12345, 768, 16, True),
                                              (2**63 + 7, 200, 32, True), (99, 64, 64, False)])
def test_projection_matrix_matches_generator(seed, d, k, moment):
    mom = torch.rand(d, generator=wl.generator(seed % 1000, "cpu")) * 1.5 + 0.5 if moment else None
    out = torch.empty((d, k), dtype=torch.float32, device=DEV)
    bg.bergson_projection_matrix(seed, d, k, bg.BERGSON_PROJ_GAUSSIAN,
                                 None if mom is None else mom.to(DEV), out)
    torch.cuda.synchronize()
    want = orc.projection_matrix(seed, d, k)
    if mom is not None:
        want = want / np.sqrt(mom.numpy().astype(np.float64))[:, None]
    got = np32(out)
    # fp32 Box-Muller against the fp64 definition: a few fp32 ulps per entry
    assert np.max(np.abs(got - want)) < 5e-6
    err = np.abs(got - want) / np.sqrt(np.mean(want * want))   # relative to the entry scale
    assert np.median(err) < 2e-7 and np.quantile(err, 0.999) < 2e-6


@pytest.mark.parametrize("kind", [bg.BERGSON_PROJ_RADEMACHER, bg.BERGSON_PROJ_UNIFORM])
@pytest.mark.parametrize("seed,d,k,moment", [(2**63 + 11, 200, 32, False), (3, 768, 16, True),
                                              (41, 64, 64, True)])
def test_rademacher_uniform_matrices_match_generator(kind, seed, d, k, moment):
    mom = torch.rand(d, generator=wl.generator(seed % 1000, "cpu")) * 1.5 + 0.5 if moment else None
    out = torch.empty((d, k), dtype=torch.float32, device=DEV)
    bg.bergson_projection_matrix(seed, d, k, kind, None if mom is None else mom.to(DEV), out)
    torch.cuda.synchronize()
    want = orc.projection_matrix(seed, d, k, kind)
    if mom is not None:
        want = want / np.sqrt(mom.numpy().astype(np.float64))[:, None]
    got = np32(out)
    if kind == bg.BERGSON_PROJ_RADEMACHER and mom is None:
        np.testing.assert_array_equal(got, want)          # +-fl32(1/sqrt(k)): exact
    else:
        # the draw is exact in fp32; only the scalings round (a few ulps)
        assert np.max(np.abs(got - want) / np.abs(want)) < 1e-6
    assert np.array_equal(np.sign(got), np.sign(want))


@pytest.mark.parametrize("kind", [bg.BERGSON_PROJ_RADEMACHER, bg.BERGSON_PROJ_UNIFORM])
def test_rademacher_uniform_projection_parity(kind):
    specs = [wl.ModuleSpec("a", 64, 200), wl.ModuleSpec("b", 136, 64), wl.ModuleSpec("c", 768, 2304)]
    kp = [(16, 16), (32, 16), (16, 32)]
    B, T = 3, 300
    gl, ol, ld = make_layers(specs, B, T, kp, base_seed=11, data_seed=4, rc=True,
                             input_scale=True, kind=kind)
    g = wl.generator(8, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.1).to(torch.uint8)
    out = run_project(gl, B, T, mask.to(DEV), ld)
    want = orc.project_grads(ol, mask.numpy(), ld)
    err = rel_frobenius(np32(out).astype(np.float64), want)
    assert err.max() <= TIGHT
    # a different distribution really is used: the Gaussian call differs
    gl_g = [bg.Layer(x.A, x.G, x.k_in, x.k_out, x.seed_in, x.seed_out, x.r, x.c, x.out_col_offset)
            for x in gl]
    out_g = run_project(gl_g, B, T, mask.to(DEV), ld)
    assert rel_frobenius(np32(out_g).astype(np.float64), want).min() > 0.1


def test_tiny_workload_parity():
    cfg = wl.TINY
    gl, ol, ld = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], rc=True)
    out = run_project(gl, cfg.B, cfg.T, None, ld)
    want = orc.project_grads(ol, None, ld)
    err = rel_frobenius(np32(out).astype(np.float64), want)
    assert err.max() <= BAR
    assert err.max() <= TIGHT, f"max rel err {err.max():.2e}"


def test_tiny_workload_matches_golden_fixtures():
    """CUDA path against the stored oracle fixtures of tests/golden (projected
    rows, then the store and an exact top-4 for 8 queries)."""
    from tests._util import golden_lines
    cfg = wl.TINY
    gl, _, ld = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], rc=True)
    out = run_project(gl, cfg.B, cfg.T, None, ld)
    want = np.array([[float(v) for v in line.split()] for line in golden_lines("tiny_projected.txt")])
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= TIGHT
    store = torch.empty((cfg.B, ld), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(out, cfg.B, ld, True, store, 0)
    queries = wl.gaussian_rows(cfg.B, ld, seed=3).to(DEV)
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(cfg.B, ld, cfg.B, 4), DEV)
    s = torch.empty((cfg.B, 4), dtype=torch.float32, device=DEV)
    i = torch.empty((cfg.B, 4), dtype=torch.int64, device=DEV)
    bg.bergson_score_topk(store, cfg.B, ld, queries, 4, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    rows = [[tok.split(":") for tok in line.split()] for line in golden_lines("tiny_topk.txt")]
    np.testing.assert_array_equal(i.cpu().numpy(), [[int(a) for a, _ in r] for r in rows])
    np.testing.assert_allclose(np32(s), [[float(b) for _, b in r] for r in rows], atol=1e-3, rtol=0)


def test_identity_projection_gives_normalised_gradient():
    spec = wl.ModuleSpec("lin", 64, 64)
    gl, ol, ld = make_layers([spec], 3, 100, [(64, 64)], rc=True, kind=bg.BERGSON_PROJ_IDENTITY)
    out = run_project(gl, 3, 100, None, ld)
    want = orc.project_grads(ol, None, ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= TIGHT


def test_multi_module_mask_ragged_mixed_k():
    specs = [wl.ModuleSpec("a", 64, 200), wl.ModuleSpec("b", 136, 64), wl.ModuleSpec("c", 96, 512),
             wl.ModuleSpec("d", 520, 72)]
    kp = [(16, 16), (32, 16), (16, 32), (32, 32)]
    B, T = 4, 300                      # 3 tiles, the last one ragged
    gl, ol, ld = make_layers(specs, B, T, kp, base_seed=7, data_seed=3, rc=True)
    g = wl.generator(5, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.2).to(torch.uint8)
    mask[2] = 0                        # an all-masked example
    mask[1, 128:256] = 0               # a fully masked middle tile
    ld_pad = ld + 40                   # columns nothing writes keep their value
    out = run_project(gl, B, T, mask.to(DEV), ld_pad)
    got = np32(out).astype(np.float64)
    want = orc.project_grads(ol, mask.numpy(), ld)
    assert np.all(np.isnan(got[:, ld:]))
    err = rel_frobenius(got[:, :ld], want)
    assert err[[0, 1, 3]].max() <= TIGHT
    np.testing.assert_array_equal(got[2, :ld], 0.0)


def test_masked_tokens_ignore_nonfinite_values():
    spec = wl.ModuleSpec("lin", 64, 128)
    gl, ol, ld = make_layers([spec], 2, 160, [(16, 16)])
    mask = torch.ones((2, 160), dtype=torch.uint8)
    mask[0, 5] = 0
    mask[1, 150] = 0
    A, G = gl[0].A.clone(), gl[0].G.clone()
    A[0, 5, 3] = float("nan")
    G[1, 150, 7] = float("inf")
    gl[0].A, gl[0].G = A, G
    out = run_project(gl, 2, 160, mask.to(DEV), ld)
    want = orc.project_grads(ol, mask.numpy(), ld)
    got = np32(out).astype(np.float64)
    assert np.all(np.isfinite(got))
    assert rel_frobenius(got, want).max() <= TIGHT


def test_unmasked_nan_propagates():
    spec = wl.ModuleSpec("lin", 64, 64)
    gl, _, ld = make_layers([spec], 2, 64, [(16, 16)])
    A = gl[0].A.clone()
    A[1, 3, 0] = float("nan")
    gl[0].A = A
    got = np32(run_project(gl, 2, 64, None, ld))
    assert np.all(np.isfinite(got[0])) and np.any(np.isnan(got[1]))


def test_empty_token_axis_writes_zero_blocks():
    spec = wl.ModuleSpec("lin", 64, 64)
    A = torch.zeros((3, 0, 64), dtype=torch.bfloat16, device=DEV)
    G = torch.zeros((3, 0, 64), dtype=torch.bfloat16, device=DEV)
    ly = bg.Layer(A, G, 16, 16, 1, 2)
    out = run_project([ly], 3, 0, None, 256)
    np.testing.assert_array_equal(np32(out), 0.0)


def test_deterministic_bitwise():
    specs = [wl.ModuleSpec("a", 256, 768), wl.ModuleSpec("b", 768, 256)]
    gl, _, ld = make_layers(specs, 6, 1024, [(16, 16), (16, 16)], input_scale=True)
    assert bg.bergson_debug_project_plan(gl, 6, 1024)[2] > 0     # pieces: last finisher varies
    a = run_project(gl, 6, 1024, None, ld)
    b = run_project(gl, 6, 1024, None, ld)
    assert torch.equal(a, b)


def test_piece_path_wide_modules_mask_bias_moments():
    """Few examples, wide modules: slots are cut into per-side pieces whose
    token projections the last piece sums; ragged tail, masked tiles, bias."""
    specs = [wl.ModuleSpec("up", 1024, 4096), wl.ModuleSpec("down", 3072, 1024),
             wl.ModuleSpec("small", 256, 264)]
    B, T = 3, 700                       # 6 tiles, the last one ragged
    gl, ol, ld = make_layers(specs, B, T, [(16, 16)] * 3, base_seed=21, data_seed=8, rc=True,
                             input_scale=True)
    gl[1].bias_col_offset = ol[1].bias_col_offset = ld
    ld_b = ld + 16
    slots, items, pieces, _ = bg.bergson_debug_project_plan(gl, B, T)
    assert pieces > 0 and items > slots
    g = wl.generator(12, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.25).to(torch.uint8)
    mask[1, 128:384] = 0                # two fully masked tiles
    mask[2, 650:] = 0
    out = run_project(gl, B, T, mask.to(DEV), ld_b)
    want = orc.project_grads(ol, mask.numpy(), ld_b)
    got = np32(out).astype(np.float64)
    assert rel_frobenius(got, want).max() <= TIGHT
    assert rel_frobenius(got[:, ld:ld_b], want[:, ld:ld_b]).max() <= TIGHT


@pytest.mark.parametrize("kp", [[(16, 32), (32, 16)], [(32, 32), (64, 64)]])
def test_piece_path_mixed_k_groups(kp):
    specs = [wl.ModuleSpec("a", 2048, 512), wl.ModuleSpec("b", 512, 1536)]
    B, T = 2, 520
    gl, ol, ld = make_layers(specs, B, T, kp, base_seed=5, data_seed=9, rc=True, input_scale=True)
    assert bg.bergson_debug_project_plan(gl, B, T)[2] > 0
    out = run_project(gl, B, T, None, ld)
    want = orc.project_grads(ol, None, ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= TIGHT


def test_fused_path_many_slots():
    """Enough (module, example) slots that the planner keeps every item fused."""
    specs = [wl.ModuleSpec("a", 64, 128), wl.ModuleSpec("b", 128, 64)]
    B, T = 200, 500
    gl, ol, ld = make_layers(specs, B, T, [(16, 16), (16, 16)], base_seed=3, data_seed=6, rc=True)
    assert bg.bergson_debug_project_plan(gl, B, T)[2] == 0
    g = wl.generator(14, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.1).to(torch.uint8)
    out = run_project(gl, B, T, mask.to(DEV), ld)
    want = orc.project_grads(ol, mask.numpy(), ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= TIGHT


@pytest.mark.parametrize("blk", [0, 11])
def test_pythia1b4_block_slice(blk):
    cfg = wl.PYTHIA1B4
    specs = cfg.block_modules(blk)
    B, T = 2, 256
    gl, ol, ld = make_layers(specs, B, T, [(32, 32)] * len(specs), base_seed=blk, data_seed=blk,
                             rc=True, input_scale=True)
    out = run_project(gl, B, T, None, ld)
    want = orc.project_grads(ol, None, ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= TIGHT


def test_llama8b_block_slice():
    cfg = wl.LLAMA8B
    specs = cfg.block_modules(0)
    B, T = 1, 160
    gl, ol, ld = make_layers(specs, B, T, [(16, 16)] * len(specs), input_scale=True)
    out = run_project(gl, B, T, None, ld)
    want = orc.project_grads(ol, None, ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= TIGHT


def test_build_store_matches_oracle():
    g = wl.generator(11, "cpu")
    X = torch.randn((9, 264), generator=g) * 3.0
    X[4] = 0.0
    proj = X.to(DEV)
    store = torch.full((20, 272), float("nan"), dtype=torch.float16, device=DEV)
    norms = torch.empty(9, dtype=torch.float32, device=DEV)
    bg.bergson_build_store(proj, 9, 264, True, store, 5, norms)
    torch.cuda.synchronize()
    want, want_norms = orc.build_store(X.numpy().astype(np.float64))
    got = store.cpu()
    assert torch.isnan(got[:5]).all() and torch.isnan(got[14:]).all() and torch.isnan(got[5:14, 264:]).all()
    g16 = got[5:14, :264].float().numpy()
    ulp = np.spacing(np.abs(want)).astype(np.float32)           # one fp16 ulp per element
    assert np.all(np.abs(g16 - want.astype(np.float32)) <= ulp)
    np.testing.assert_array_equal(g16[4], 0.0)
    np.testing.assert_allclose(np32(norms), want_norms, rtol=1e-6)
    rn = np.linalg.norm(g16.astype(np.float64), axis=1)
    np.testing.assert_allclose(rn[[0, 1, 2, 3, 5, 6, 7, 8]], 1.0, atol=1e-3)
    # unit_normalize = 0 stores the values as they are
    bg.bergson_build_store(proj, 9, 264, False, store, 0)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(store[:9, :264].cpu().numpy(), X.numpy().astype(np.float16))


def test_build_store_blocks_matches_oracle():
    # per-module unit norm: blocks of 256, 512, 1024 and 256 columns (module
    # blocks k_out x k_in), scaled very differently, one zero block, rows
    # appended at an offset into a store with padded rows
    g = wl.generator(12, "cpu")
    offs = [0, 256, 768, 1792, 2048]
    scale = torch.cat([torch.full((256,), 30.0), torch.full((512,), 1e-3), torch.ones(1024),
                       torch.full((256,), 5.0)])
    X = torch.randn((7, 2048), generator=g) * scale
    X[3, 256:768] = 0.0
    proj = torch.full((7, 2052), float("nan"))
    proj[:, :2048] = X
    proj = proj.to(DEV)
    store = torch.full((12, 2056), float("nan"), dtype=torch.float16, device=DEV)
    norms = torch.empty((7, 4), dtype=torch.float32, device=DEV)
    bg.bergson_build_store_blocks(proj, 7, 2048, offs, store, 4, norms)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    want, want_norms = orc.build_store_blocks(X.numpy().astype(np.float64), offs)
    got = store.cpu()
    assert torch.isnan(got[:4]).all() and torch.isnan(got[11:]).all()
    assert torch.isnan(got[4:11, 2048:]).all()
    g16 = got[4:11, :2048].float().numpy()
    ulp = np.spacing(np.abs(want)).astype(np.float32)           # one fp16 ulp per element
    assert np.all(np.abs(g16 - want.astype(np.float32)) <= ulp)
    np.testing.assert_array_equal(g16[3, 256:768], 0.0)
    np.testing.assert_allclose(np32(norms), want_norms, rtol=1e-6)
    # one block equals the whole-row store, bit for bit
    a = torch.empty((7, 2048), dtype=torch.float16, device=DEV)
    b = torch.empty((7, 2048), dtype=torch.float16, device=DEV)
    bg.bergson_build_store_blocks(proj, 7, 2048, [0, 2048], a, 0)
    bg.bergson_build_store(proj, 7, 2048, True, b, 0)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


def test_build_store_blocks_one_per_module_of_a_llama_block_set():
    # 160 modules of 256 columns (the Llama-8B-shaped layer set at k = 16)
    g = wl.generator(13, "cpu")
    K = 160 * 256
    X = torch.randn((8, K), generator=g) * torch.rand((1, K), generator=g).mul(10).add(0.1)
    offs = list(range(0, K + 1, 256))
    store = torch.empty((8, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store_blocks(X.to(DEV), 8, K, offs, store, 0)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    want, _ = orc.build_store_blocks(X.numpy().astype(np.float64), offs)
    g16 = store.cpu().float().numpy()
    assert np.all(np.abs(g16 - want.astype(np.float32)) <= np.spacing(np.abs(want)))


def _store_from_rows(rows: torch.Tensor) -> torch.Tensor:
    N, K = rows.shape
    store = torch.empty((N, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(rows.to(DEV), N, K, True, store, 0)
    return store


def _score(store, queries, topk):
    N, K = store.shape
    Q = queries.shape[0]
    ws = bg.workspace_tensor(bg.bergson_score_topk_workspace(N, K, Q, topk), DEV)
    s = torch.empty((Q, topk), dtype=torch.float32, device=DEV)
    i = torch.empty((Q, topk), dtype=torch.int64, device=DEV)
    bg.bergson_score_topk(store, N, K, queries, topk, s, i, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    return np32(s), i.cpu().numpy()


def test_tiny_end_to_end_scores():
    cfg = wl.TINY
    gl, ol, ld = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], rc=True)
    out = run_project(gl, cfg.B, cfg.T, None, ld)
    store = torch.empty((cfg.B, ld), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(out, cfg.B, ld, True, store, 0)
    want_store, _ = orc.build_store(orc.project_grads(ol, None, ld))
    # (i) queries = the store's own examples: symmetric, self is top-1
    s, i = _score(store, out, 4)
    np.testing.assert_array_equal(i[:, 0], np.arange(cfg.B))
    np.testing.assert_allclose(s[:, 0], 1.0, atol=1e-3)
    S = orc.cosine_scores(want_store, orc.project_grads(ol, None, ld))
    check_topk(s, i, S, 4)
    # (ii) eight fresh examples (data seed 1) as queries
    gq, oq, _ = make_layers(cfg.modules, cfg.B, cfg.T, [(16, 16)], data_seed=1, rc=True)
    for a, b in zip(gq, gl):        # same projection and moments, new data
        a.seed_in, a.seed_out, a.r, a.c = b.seed_in, b.seed_out, b.r, b.c
    for a, b in zip(oq, ol):
        a.seed_in, a.seed_out, a.r, a.c = b.seed_in, b.seed_out, b.r, b.c
    qout = run_project(gq, cfg.B, cfg.T, None, ld)
    s, i = _score(store, qout, 4)
    S = orc.cosine_scores(store.cpu().numpy(), orc.project_grads(oq, None, ld))
    check_topk(s, i, S, 4)


@pytest.mark.parametrize("N,K,Q,topk", [(5000, 520, 200, 17), (40, 64, 1, 40), (777, 128, 129, 5),
                                         (3000, 1024, 64, 100)])
def test_score_topk_random(N, K, Q, topk):
    g = wl.generator(N + K, "cpu")
    rows = torch.randn((N, K), generator=g)
    store = _store_from_rows(rows)
    queries = torch.randn((Q, K), generator=g)
    s, i = _score(store, queries.to(DEV), topk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(s, i, S, topk)


@pytest.mark.parametrize("Q,topk", [(130, 5), (200, 3), (40, 3)])
def test_score_prefix_threshold_pass(Q, topk):
    # N >= 8 * 128 * topk and Q > 128: the scorer first takes the exact top-k of
    # a prefix of the store and starts the full pass from its k-th score (Q = 40
    # takes the single-pass path on the same data).
    N, K = 30_000, 256
    g = wl.generator(Q * 7 + topk, "cpu")
    rows = torch.randn((N, K), generator=g)
    queries = torch.randn((Q, K), generator=g)
    rows[N - 5:] = rows[:5]                  # exact ties across the prefix boundary
    queries[:5] = rows[:5]
    rows[100:100 + Q] = queries + 0.3 * torch.randn((Q, K), generator=g)   # strong prefix hits
    rows[N - 200:N - 200 + 20] = queries[:20] * 2.0 + torch.randn((20, K), generator=g)
    store = _store_from_rows(rows)
    s, i = _score(store, queries.to(DEV), topk)
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(s, i, S, topk)
    for r in range(5):
        assert set(i[r, :2].tolist()) == {r, N - 5 + r}


def test_score_ties_prefer_lower_index():
    g = wl.generator(3, "cpu")
    base = torch.randn((50, 256), generator=g)
    rows = torch.cat([base, base[:10]], 0)         # rows 50..59 duplicate rows 0..9
    store = _store_from_rows(rows)
    q = base[:10].clone().to(DEV)
    s, i = _score(store, q, 2)
    for r in range(10):
        assert set(i[r].tolist()) == {r, 50 + r}
        if s[r, 0] == s[r, 1]:
            assert i[r, 0] == r
    S = orc.cosine_scores(store.cpu().numpy(), base[:10].numpy().astype(np.float64))
    check_topk(s, i, S, 2)


def test_zero_query_scores_zero():
    g = wl.generator(4, "cpu")
    store = _store_from_rows(torch.randn((300, 64), generator=g))
    q = torch.zeros((2, 64), device=DEV)
    q[1, 0] = 1.0
    s, i = _score(store, q, 3)
    np.testing.assert_array_equal(s[0], 0.0)
    np.testing.assert_array_equal(i[0], [0, 1, 2])


def test_planted_neighbours_exact_set():
    N, K, Q, per = 60_000, 1024, 48, 100
    g = wl.generator(21, "cpu")
    rows = torch.randn((N, K), generator=g)
    queries = torch.randn((Q, K), generator=g)
    pos = wl.planted_positions(N, Q, per, seed=22)
    rows[pos.reshape(-1)] = wl.planted_rows(queries, per, seed=23)
    store = _store_from_rows(rows)
    s, i = _score(store, queries.to(DEV), per)
    for q in range(Q):
        assert set(i[q].tolist()) == set(pos[q].tolist())
    S = orc.cosine_scores(store.cpu().numpy(), queries.numpy().astype(np.float64))
    check_topk(s, i, S, per)


def test_bounded_wait_reports_timeout_and_context_survives():
    assert bg.bergson_sync_status() == bg.BERGSON_OK
    bg.bergson_debug_wait_probe(2_000_000)          # 2 ms wait that nothing completes
    assert bg.bergson_sync_status() == bg.BERGSON_EDEVICE_TIMEOUT
    assert bg.bergson_sync_status() == bg.BERGSON_OK  # cleared
    test_tiny_workload_parity()                      # the context still works


def test_bias_blocks_with_mask_and_moments():
    specs = [wl.ModuleSpec("a", 64, 200), wl.ModuleSpec("b", 136, 64), wl.ModuleSpec("c", 96, 72)]
    kp = [(16, 16), (32, 32), (16, 32)]
    B, T = 3, 300
    gl, ol, ld = make_layers(specs, B, T, kp, base_seed=9, data_seed=4, rc=True)
    # bias blocks after the weight blocks, for layers 0 and 2 only
    gl[0].bias_col_offset = ol[0].bias_col_offset = ld
    gl[2].bias_col_offset = ol[2].bias_col_offset = ld + 16
    ld_b = ld + 16 + 32
    g = wl.generator(10, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.3).to(torch.uint8)
    mask[1, 128:256] = 0
    out = run_project(gl, B, T, mask.to(DEV), ld_b)
    want = orc.project_grads(ol, mask.numpy(), ld_b)
    got = np32(out).astype(np.float64)
    assert rel_frobenius(got, want).max() <= TIGHT
    for off, k in ((ld, 16), (ld + 16, 32)):
        blk_g, blk_w = got[:, off:off + k], want[:, off:off + k]
        assert rel_frobenius(blk_g, blk_w).max() <= TIGHT
    # overlapping a bias block with a weight block is rejected
    gl[2].bias_col_offset = 8
    ws = bg.workspace_tensor(1 << 24, DEV)
    with pytest.raises(bg.BergsonError) as e:
        bg.bergson_project_grads(gl, B, T, None, out, ws)
    assert e.value.status == bg.BERGSON_EINVAL


@pytest.mark.parametrize("B,T,d,f", [(2, 700, 1024, 2048), (200, 256, 128, 256)])
def test_shared_input_layers(B, T, d, f):
    """Layers reading one A tensor (a gate and an up projection) are scheduled
    side by side; results match the oracle on the piece path (few examples)
    and on the fused path (many)."""
    specs = [wl.ModuleSpec("gate", d, f), wl.ModuleSpec("up", d, f, True),
             wl.ModuleSpec("down", f, d)]
    gl, ol, ld = make_layers(specs, B, T, [(16, 16)] * 3, base_seed=4, data_seed=2, rc=True,
                             input_scale=True)
    assert gl[1].A.data_ptr() == gl[0].A.data_ptr()
    slots, items, pieces, shared = bg.bergson_debug_project_plan(gl, B, T)
    assert shared == 2 and (pieces > 0) == (B == 2)
    g = wl.generator(15, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.2).to(torch.uint8)
    out = run_project(gl, B, T, mask.to(DEV), ld)
    want = orc.project_grads(ol, mask.numpy(), ld)
    assert rel_frobenius(np32(out).astype(np.float64), want).max() <= TIGHT
