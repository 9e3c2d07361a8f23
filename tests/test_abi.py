"""Host-side checks of the C ABI that need no GPU: load, exports, validation."""
import ctypes
import os
import re

import pytest

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built_library():
    from paper_2606_11660_gb300 import _build
    _build.build()
    yield


def _declared_symbols():
    src = open(os.path.join(ROOT, "include", "bergson.h")).read()
    return sorted(set(re.findall(r"BERGSON_API\s+[\w\s\*]*?\b(bergson_\w+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    declared = _declared_symbols()
    assert len(declared) >= 12
    assert sorted(bg.EXPORTED) == declared
    L = ctypes.CDLL(bg.LIB_PATH)
    for name in declared:
        assert hasattr(L, name), name
    assert bg.bergson_version() == 100


def test_module_seeds_match_oracle_derivation():
    for base, m in [(0, 0), (0, 47), (123456789, 3), (2**64 - 1, 159)]:
        assert bg.bergson_module_seeds(base, m) == orc.module_seeds(base, m)


FAKE = 0x7F0000000000  # aligned, never dereferenced: validation fails first or no device


def _layer(**kw):
    d = dict(A=FAKE, G=FAKE + 4096, d_in=64, d_out=64, k_in=16, k_out=16, seed_in=1, seed_out=2,
             proj_kind=0, flags=0, r=None, c=None, out_col_offset=0)
    d.update(kw)
    return bg.bergson_layer(**d)


def _ws(layers, B=2, T=32):
    arr = (bg.bergson_layer * len(layers))(*layers)
    n = ctypes.c_size_t()
    st = bg.lib().bergson_project_grads_workspace(arr, len(layers), B, T, ctypes.byref(n))
    return st, n.value


def _proj(layers, B=2, T=32, out=FAKE, ld_out=256, ws=FAKE, ws_bytes=1 << 30, mask=None):
    arr = (bg.bergson_layer * len(layers))(*layers)
    return bg.lib().bergson_project_grads(arr, len(layers), B, T, mask, out, ld_out, ws, ws_bytes,
                                          None)


@pytest.mark.parametrize("kw,code", [
    (dict(d_in=60), bg.BERGSON_EALIGN),
    (dict(d_out=4), bg.BERGSON_EINVAL),
    (dict(k_in=24), bg.BERGSON_EUNSUPPORTED),
    (dict(k_out=128), bg.BERGSON_EUNSUPPORTED),
    (dict(proj_kind=7), bg.BERGSON_EINVAL),
    (dict(proj_kind=1), bg.BERGSON_EINVAL),            # identity needs k == d
    (dict(r=FAKE), bg.BERGSON_EINVAL),                 # r without c
    (dict(A=FAKE + 8), bg.BERGSON_EALIGN),
    (dict(G=None), bg.BERGSON_EINVAL),
    (dict(flags=2), bg.BERGSON_EINVAL),
    (dict(flags=1, bias_col_offset=-3), bg.BERGSON_EINVAL),
    (dict(out_col_offset=-1), bg.BERGSON_EINVAL),
])
def test_layer_validation(kw, code):
    st, _ = _ws([_layer(**kw)])
    assert st == code
    assert bg.bergson_last_error() != ""
    assert _proj([_layer(**kw)]) == code


def test_every_projection_kind_validates():
    for kind in (bg.BERGSON_PROJ_GAUSSIAN, bg.BERGSON_PROJ_RADEMACHER, bg.BERGSON_PROJ_UNIFORM):
        st, n = _ws([_layer(proj_kind=kind)])
        assert st == bg.BERGSON_OK and n > 0
    assert _ws([_layer(proj_kind=4)])[0] == bg.BERGSON_EINVAL
    assert bg.lib().bergson_projection_matrix(1, 64, 16, 4, None, FAKE, None) == bg.BERGSON_EINVAL


def test_workspace_query_and_block_checks():
    st, n = _ws([_layer(), _layer(out_col_offset=256, k_in=32)])
    assert st == bg.BERGSON_OK and n > 0 and n % 256 == 0
    st2, n2 = _ws([_layer(), _layer(out_col_offset=256, k_in=32)], B=64, T=4096)
    assert st2 == bg.BERGSON_OK and n2 > n
    # overlapping output blocks
    assert _proj([_layer(), _layer(out_col_offset=128)], ld_out=512) == bg.BERGSON_EINVAL
    assert "overlap" in bg.bergson_last_error()
    # block past ld_out
    assert _proj([_layer(out_col_offset=100)], ld_out=256) == bg.BERGSON_EINVAL
    # workspace too small / misaligned / missing
    assert _proj([_layer()], ws_bytes=16) == bg.BERGSON_EWORKSPACE
    assert _proj([_layer()], ws=FAKE + 16) == bg.BERGSON_EALIGN
    assert _proj([_layer()], ws=None) == bg.BERGSON_EINVAL
    assert _proj([_layer()], B=-1) == bg.BERGSON_EINVAL
    assert bg.lib().bergson_project_grads(None, 1, 2, 3, None, FAKE, 256, FAKE, 1 << 20, None) == bg.BERGSON_EINVAL


def test_empty_batch_is_a_no_op_and_injection_hook():
    assert _proj([_layer()], B=0) == bg.BERGSON_OK
    bg.bergson_debug_inject_status(bg.BERGSON_ECUDA, 1)
    assert _proj([_layer()], B=0) == bg.BERGSON_ECUDA
    assert "injected" in bg.bergson_last_error()
    assert _proj([_layer()], B=0) == bg.BERGSON_OK     # one-shot
    bg.bergson_debug_inject_status(bg.BERGSON_ECUDA, 0)


def test_store_validation():
    f = bg.lib().bergson_build_store
    ok_args = dict(proj=FAKE, B=4, K=64, ld_proj=64, unit=1, store=FAKE, ld_store=64, row_offset=0,
                   N_cap=4, norms=None, stream=None)

    def call(**kw):
        a = dict(ok_args)
        a.update(kw)
        return f(*a.values())
    assert call(K=60) == bg.BERGSON_EALIGN
    assert call(ld_proj=32) == bg.BERGSON_EINVAL
    assert call(ld_proj=66) == bg.BERGSON_EALIGN
    assert call(ld_store=72 + 4) == bg.BERGSON_EALIGN
    assert call(row_offset=1) == bg.BERGSON_EINVAL      # does not fit N_cap
    assert call(store=FAKE + 8) == bg.BERGSON_EALIGN
    assert call(B=0) == bg.BERGSON_OK


@pytest.mark.parametrize("entry", ["bergson_score_topk", "bergson_score_bottomk"])
def test_score_validation(entry):
    f = getattr(bg.lib(), entry)
    n = ctypes.c_size_t()
    assert bg.lib().bergson_score_topk_workspace(100, 64, 10, 5, ctypes.byref(n)) == bg.BERGSON_OK
    ws = n.value

    def call(N=100, K=64, ld=64, q=FAKE, Q=10, ldq=64, topk=5, ws_bytes=ws, store=FAKE):
        return f(store, N, K, ld, q, Q, ldq, topk, FAKE, FAKE, FAKE, ws_bytes, None)
    assert call(topk=101) == bg.BERGSON_EINVAL           # k > N
    assert call(topk=0) == bg.BERGSON_EUNSUPPORTED
    assert call(topk=2000, N=5000) == bg.BERGSON_EUNSUPPORTED
    assert call(K=60, ld=64) == bg.BERGSON_EALIGN
    assert call(ld=68) == bg.BERGSON_EALIGN
    assert call(ldq=32) == bg.BERGSON_EINVAL
    assert call(ws_bytes=ws - 1) == bg.BERGSON_EWORKSPACE
    assert call(store=FAKE + 8) == bg.BERGSON_EALIGN
    assert call(N=0) == bg.BERGSON_EINVAL
    assert call(Q=0) == bg.BERGSON_OK


def test_projection_matrix_validation():
    f = bg.lib().bergson_projection_matrix
    assert f(1, 64, 24, 0, None, FAKE, None) == bg.BERGSON_EUNSUPPORTED
    assert f(1, 64, 16, 1, None, FAKE, None) == bg.BERGSON_EINVAL
    assert f(1, 64, 16, 0, None, None, None) == bg.BERGSON_EINVAL
    assert bg.lib().bergson_debug_wait_probe(0, None) == bg.BERGSON_EINVAL


def test_calls_without_device_fail_cleanly():
    import torch
    if torch.cuda.is_available():
        pytest.skip("host without a GPU only")
    st = _proj([_layer()])
    assert st == bg.BERGSON_ECUDA
    assert bg.bergson_last_error() != ""


def test_onthefly_validation():
    f = bg.lib().bergson_score_grads
    n = ctypes.c_size_t()
    assert bg.lib().bergson_score_grads_workspace(32, 12288, 1024, ctypes.byref(n)) == bg.BERGSON_OK
    ws = n.value
    assert ws >= 4 * 32 * 1024

    def call(B=32, K=12288, ldp=12288, Q=1024, ldq=12288, lds=1024, ws_bytes=ws, proj=FAKE,
             queries=FAKE, scores=FAKE, wsp=FAKE):
        return f(proj, B, K, ldp, queries, Q, ldq, 1, scores, lds, wsp, ws_bytes, None)
    assert call(K=10) == bg.BERGSON_EALIGN
    assert call(ldp=100) == bg.BERGSON_EINVAL
    assert call(ldq=12290) == bg.BERGSON_EALIGN
    assert call(lds=10) == bg.BERGSON_EINVAL
    assert call(proj=FAKE + 4) == bg.BERGSON_EALIGN
    assert call(ws_bytes=ws - 1) == bg.BERGSON_EWORKSPACE
    assert call(queries=None) == bg.BERGSON_EINVAL
    assert call(B=0) == bg.BERGSON_OK
    assert call(Q=0) == bg.BERGSON_OK


def test_aggregate_validation():
    f = bg.lib().bergson_aggregate_rows

    def call(rows=FAKE, n=10, K=64, ld=64, offsets=FAKE, G=3, mode=1, norm=1, out=FAKE,
             ld_out=64, ws=FAKE, ws_bytes=1 << 20):
        return f(rows, n, K, ld, offsets, G, mode, norm, out, ld_out, ws, ws_bytes, None)
    assert call(K=62) == bg.BERGSON_EALIGN
    assert call(mode=5) == bg.BERGSON_EINVAL
    assert call(ld=60) == bg.BERGSON_EINVAL
    assert call(offsets=None) == bg.BERGSON_EINVAL
    assert call(offsets=FAKE + 4) == bg.BERGSON_EALIGN
    assert call(ws_bytes=8) == bg.BERGSON_EWORKSPACE
    assert call(G=0) == bg.BERGSON_OK


def test_fisher_validation():
    L = bg.lib()
    n = ctypes.c_size_t()
    assert L.bergson_fisher_preconditioner_workspace(256, ctypes.byref(n)) == bg.BERGSON_OK
    assert n.value >= 4 * 256 * 256 * 4
    f = L.bergson_fisher_preconditioner
    ok = dict(R1=FAKE, R2=None, K=256, ldr=256, lam=0.5, damping=0.1, power=0, iters=20, M=FAKE,
              ldm=256, ws=FAKE, wsb=n.value)

    def call(**kw):
        a = dict(ok)
        a.update(kw)
        return f(*a.values(), None)
    assert call(K=254) == bg.BERGSON_EALIGN
    assert call(lam=1.5) == bg.BERGSON_EINVAL
    assert call(damping=-1.0) == bg.BERGSON_EINVAL
    assert call(power=7) == bg.BERGSON_EINVAL
    assert call(iters=0) == bg.BERGSON_EINVAL
    assert call(R1=None) == bg.BERGSON_EINVAL
    assert call(M=FAKE + 4) == bg.BERGSON_EALIGN
    assert call(wsb=16) == bg.BERGSON_EWORKSPACE
    fit = L.bergson_fisher_fit
    assert fit(FAKE, 0, 256, 256, FAKE, 256, FAKE, 1 << 30, None) == bg.BERGSON_EINVAL
    assert fit(FAKE, 10, 256, 200, FAKE, 256, FAKE, 1 << 30, None) == bg.BERGSON_EINVAL


def test_store_io_validation(tmp_path):
    L = bg.lib()
    assert L.bergson_store_save(FAKE, 10, 64, 32, b"/tmp/x", 0, None) == bg.BERGSON_EINVAL
    assert L.bergson_store_save(FAKE, 10, 64, 64, b"", 0, None) == bg.BERGSON_EINVAL
    assert L.bergson_store_load(str(tmp_path / "missing").encode(), 0, 1, 64, FAKE, 64, None) == bg.BERGSON_EINVAL


def _plan(layers, B, T):
    return bg.bergson_debug_project_plan(layers, B, T)


def _block_layers(specs, k):
    out, off = [], 0
    for i, s in enumerate(specs):
        a = out[-1].A if s.shares_input else FAKE + 8192 * i       # a shared input: one pointer
        out.append(_layer(A=a, d_in=s.d_in, d_out=s.d_out, k_in=k, k_out=k, out_col_offset=off))
        off += k * k
    return out


def test_planner_keeps_fine_launches_fused():
    """48 modules x 32 examples x 4 slots: enough work items, no pieces."""
    cfg = wl.PYTHIA160M
    assert _plan(_block_layers(cfg.modules, 16), cfg.B, cfg.T) == (48 * 32 * 4, 48 * 32 * 4, 0, 0)
    cfg = wl.PYTHIA1B4                  # one block per call: 512 slots, still balanced enough
    assert _plan(_block_layers(cfg.block_modules(0), 32), cfg.B, cfg.T) == (512, 512, 0, 0)


@pytest.mark.parametrize("name,B,T,k", [("llama8b", 8, 4096, 16), ("tiny", 8, 32, 16),
                                        ("llama8b", 1, 160, 16), ("pythia1b4", 2, 256, 32)])
def test_planner_cuts_coarse_launches_into_pieces(name, B, T, k):
    cfg = wl.COLLECT_WORKLOADS[name]
    specs = cfg.block_modules(0)
    slots, items, pieces, _ = _plan(_block_layers(specs, k), B, T)
    fused = items - pieces
    split = slots - fused
    assert pieces > 0 and split > 0
    assert pieces >= 2 * split          # every cut slot has pieces on both sides
    st, n = _ws(_block_layers(specs, k), B, T)
    assert st == bg.BERGSON_OK and n % 256 == 0


def test_planner_validates_like_the_workspace_query():
    with pytest.raises(bg.BergsonError) as e:
        _plan([_layer(k_in=24)], 2, 32)
    assert e.value.status == bg.BERGSON_EUNSUPPORTED


def test_planner_groups_layers_that_share_an_input():
    """Llama-shaped block: gate and up read one A tensor."""
    cfg = wl.LLAMA8B
    layers = _block_layers(cfg.block_modules(0), 16)
    slots, items, pieces, shared = _plan(layers, cfg.B, cfg.T)
    assert shared == 2 and pieces > 0
    # many examples: no pieces, but a work table lists the shared layers' items together
    slots, items, pieces, shared = _plan(layers, 256, cfg.T)
    assert shared == 2 and pieces == 0 and items == slots
    # different d_in, or different k, is not sharing
    a = _layer(d_in=64, d_out=128)
    b = _layer(A=a.A, d_in=128, d_out=64, out_col_offset=256)
    c = _layer(A=a.A, d_in=64, d_out=64, k_in=32, out_col_offset=512)
    assert _plan([a, b, c], 2, 32)[3] == 0
    assert _plan([a, _layer(A=a.A, d_in=64, d_out=64, out_col_offset=256)], 2, 32)[3] == 2


# --- scorer launch planning (host only) ---------------------------------------

@pytest.mark.parametrize("N,Q,topk,ctas", [
    (4_000_000, 1024, 100, 152),     # the score4m workload: pairs, two tiles, prefix cut
    (4_000_000, 1024, 100, 148),     # fewer co-resident clusters
    (4_000_000, 256, 100, 152),      # pairs with one tile per CTA
    (4_000_000, 16, 100, 152),       # single-CTA kernel, no prefix
    (110_000, 1024, 100, 152),       # prefix cut to one round of tiles
    (10_000, 129, 17, 152),
    (30_000, 300, 3, 151),           # odd resident count: pairs use 150 CTAs
    (1000, 39_012, 5, 152),          # more query groups than CTAs: several passes
    (1000, 39_012, 5, 150),
    (60_000, 300, 1024, 152),        # the largest topk
    (300, 511, 300, 152),            # topk = N
    (5000, 256, 5, 7),               # few resident CTAs
    (1, 1, 1, 1),
])
def test_score_planner_invariants(N, Q, topk, ctas):
    check_score_plan(N, Q, topk, ctas)


def check_score_plan(N, Q, topk, ctas):
    K = 64
    plan = bg.bergson_debug_score_plan(N, K, Q, topk, ctas)
    assert plan
    pair, qt = Q >= 129, (2 if Q > 256 else 1)
    gsize = qt * 128
    limit = min(ctas, 160) & (~1 if pair else ~0)
    n_qg_total = -(-Q // gsize)
    if pair:
        n_qg_total += n_qg_total % 2
    covered = []
    passes = sorted({l["pass"] for l in plan})
    assert passes == list(range(0, n_qg_total, limit))
    for l in plan:
        assert (l["pair"], l["qt"]) == (int(pair), qt)
        assert l["grid"] == l["n_qg"] * l["cpg"] <= limit
        assert l["n_tiles"] == -(-l["rows"] // 256) and 1 <= l["cpg"] <= l["n_tiles"]
        assert l["qg_base"] == l["pass"] and l["q_begin"] == l["pass"] * gsize
        assert 0 < l["q_end"] - l["q_begin"] <= l["n_qg"] * gsize
        if pair:                             # whole clusters, pairs of query groups
            assert l["grid"] % 2 == 0 and l["n_qg"] % 2 == 0 and l["qg_base"] % 2 == 0
        if l["stage"] == 1:
            assert l["rows"] == N
            covered += range(l["q_begin"], l["q_end"])
        else:                                # prefix: enough rows for a real k-th best
            round_rows = (limit // l["n_qg"]) * 256
            want = -(-128 * topk // 256) * 256
            assert topk <= l["rows"] <= want and l["rows"] % 256 == 0
            assert l["rows"] == want or l["rows"] % round_rows == 0
            assert 8 * want <= N and Q >= 129
    assert covered == list(range(Q))         # every query merged exactly once
    stages = [(l["pass"], l["stage"]) for l in plan]
    assert stages == sorted(stages)          # prefix (if any) before its full pass
    n = ctypes.c_size_t()
    assert bg.lib().bergson_score_topk_workspace(N, K, Q, topk, ctypes.byref(n)) == bg.BERGSON_OK
    heaps = max(l["grid"] for l in plan) * topk * gsize * 8
    pace_words = max(l["grid"] for l in plan) * 8          # the pair kernel's pacing words
    assert n.value >= heaps + Q * K * 2 + pace_words


@pytest.mark.parametrize("N,Q", [(20_000, 600), (4_000_000, 1024), (20_000, 1300), (500_000, 4096),
                                 (3_000, 2000), (10_000_000, 40_000)])
def test_pair_pacing_peers_stay_in_the_grid(N, Q):
    # The pair scorer paces each CTA against the same-rank CTA of the next pair
    # group on the same store tiles: blockIdx = nt0 * n_qg + g_local, g_local =
    # 2 * pair group + rank.  For every planned launch that peer must be another
    # CTA of the grid with the same tile sequence and rank, and the workspace
    # must hold a pacing word per CTA.
    K, topk = 256, 10
    plan = bg.bergson_debug_score_plan(N, K, Q, topk, 152)
    n = ctypes.c_size_t()
    assert bg.lib().bergson_score_topk_workspace(N, K, Q, topk, ctypes.byref(n)) == bg.BERGSON_OK
    for l in plan:
        assert l["pair"] == 1 and l["n_qg"] % 2 == 0 and l["grid"] == l["n_qg"] * l["cpg"]
        assert l["grid"] <= 160                       # pacing words in the workspace
        if l["n_qg"] < 4:
            continue                                  # one pair group: no pacing
        n_pg = l["n_qg"] // 2
        peers = set()
        for b in range(l["grid"]):
            g_local, nt0 = b % l["n_qg"], b // l["n_qg"]
            peer = nt0 * l["n_qg"] + ((g_local // 2 + 1) % n_pg) * 2 + (g_local & 1)
            assert 0 <= peer < l["grid"] and peer != b
            assert peer // l["n_qg"] == nt0 and (peer % l["n_qg"]) % 2 == g_local % 2
            peers.add(peer)
        assert len(peers) == l["grid"]               # a ring: every CTA is someone's peer


def test_score_planner_edges():
    # a single resident CTA cannot host a two-CTA cluster: no launches (the
    # scoring call reports it as an error)
    assert bg.bergson_debug_score_plan(10_000, 64, 200, 5, 1) == []
    assert len(bg.bergson_debug_score_plan(10_000, 64, 100, 5, 1)) == 1
    assert bg.bergson_debug_score_plan(10_000, 64, 0, 5, 152) == []
    with pytest.raises(bg.BergsonError):
        bg.bergson_debug_score_plan(10, 64, 4, 11, 152)      # topk > N
    with pytest.raises(bg.BergsonError):
        bg.bergson_debug_score_plan(10_000, 64, 4, 5, 0)


# --- skinny-product planning (host only) --------------------------------------

@pytest.mark.parametrize("B,Q,K", [
    (32, 1024, 12288),      # on-the-fly scores of the bench batch
    (32, 12288, 12288),     # Fisher preconditioner applied to a batch
    (1024, 12288, 12288),   # Fisher fit (rows as x)
    (12288, 12288, 12288),  # Newton-Schulz products
    (1, 1, 8), (16, 1, 4), (64, 100, 400), (65, 100, 400), (129, 300, 4096),
    (1000, 7, 520), ((1 << 20), 3, 64),
])
def test_xgemm_planner_invariants(B, Q, K):
    check_xgemm_plan(B, Q, K)


def check_xgemm_plan(B, Q, K):
    p = bg.bergson_debug_xgemm_plan(B, Q, K)
    # batches of up to 64 rows run on CTA pairs (256 rows of y per item, 128
    # per CTA); larger batches on single CTAs with tiles of up to 128 rows
    pair = p["pair"] == 1
    assert pair == (B <= 64)
    assert p["n_pad"] % 16 == 0 and 16 <= p["n_pad"] <= (64 if pair else 128)
    assert p["y_rows"] == (256 if pair else 128)
    # tiles cover the operands
    assert p["n_ntiles"] * p["n_pad"] >= B > (p["n_ntiles"] - 1) * p["n_pad"]
    rows = p["y_rows"]
    assert p["n_mtiles"] * rows >= Q > (p["n_mtiles"] - 1) * rows
    assert p["steps"] * 32 >= K > (p["steps"] - 1) * 32
    S, steps = p["S"], p["steps"]
    if pair:
        # the (y tile, step) space split evenly over min(76, W) clusters:
        # contiguous nonempty ranges that cover it once; S = the most clusters
        # (partial planes) that meet one tile
        W = p["n_mtiles"] * steps
        n = min(76, W)
        starts = [c * W // n for c in range(n + 1)]
        assert starts[0] == 0 and starts[-1] == W and all(a < b for a, b in zip(starts, starts[1:]))
        owner = lambda g: next(c for c in range(n) if starts[c] <= g < starts[c + 1])
        planes = max(owner(mt * steps + steps - 1) - owner(mt * steps) + 1
                     for mt in range(min(p["n_mtiles"], 64)))
        assert planes <= S <= n
    else:
        # every K slice is a nonempty, contiguous range of steps
        assert 1 <= S <= min(steps, 64)
        bounds = [z * steps // S for z in range(S + 1)]
        assert bounds[0] == 0 and bounds[-1] == steps and all(a < b for a, b in zip(bounds, bounds[1:]))
    # TMEM: two accumulator sets of 2 n_pad columns (4 n_pad on pairs with two
    # MMA issuers, batch tiles up to 32 rows), and on pairs the y_hi / y_lo
    # ring after them (64 columns a stage), within 512 columns
    assert p["n_buf"] == 2
    assert p["tmem_cols"] <= 512 and p["tmem_cols"] & (p["tmem_cols"] - 1) == 0
    acc = 2 * (3 if pair and p["n_pad"] <= 32 else 2) * p["n_pad"]
    if pair:
        # a TMEM slot (y_hi, y_lo: 64 columns) per stage
        assert p["a_base"] == acc and p["tmem_cols"] == 512
        assert p["a_slots"] == p["stages"] and p["a_base"] + p["a_slots"] * 64 <= 512
    else:
        assert p["a_base"] == 0 and p["a_slots"] == 0 and acc <= p["tmem_cols"]
    # shared memory: stages of one y tile (128 rows) and, on pairs, this CTA's
    # half of [x_hi; x_lo] (and, with two issuers, its half of x_hi); on single
    # CTAs y_lo and both x parts
    xb = p["n_pad"] * 128
    stage = (128 * 128 + xb + (xb // 2 if p["n_pad"] <= 32 else 0) if pair
             else 2 * 128 * 128 + 2 * xb)
    assert 2 <= p["stages"] <= 8 and 1024 + 512 + p["stages"] * stage <= 232448
    # workspace: ordered, 256-byte aligned regions of the stated sizes
    offs = [p[k] for k in ("xnorm_off", "ynorm_off", "partial_off", "xh_off", "xl_off", "total")]
    assert all(o % 256 == 0 for o in offs) and offs == sorted(offs)
    assert p["ynorm_off"] - p["xnorm_off"] >= 4 * B * p["n_chunks"]
    assert p["n_chunks"] == -(-K // 2048)
    assert p["partial_off"] - p["ynorm_off"] >= 4 * S * Q
    assert p["xh_off"] - p["partial_off"] >= 4 * S * B * Q
    assert p["xl_off"] - p["xh_off"] >= 4 * B * K and p["total"] - p["xl_off"] >= 4 * B * K
    n = ctypes.c_size_t()
    st = bg.lib().bergson_score_grads_workspace(B, K, Q, ctypes.byref(n))
    if B * Q > (1 << 34):                    # beyond what the calls accept
        assert st == bg.BERGSON_EUNSUPPORTED
    else:
        assert st == bg.BERGSON_OK and n.value == p["total"]


def test_xgemm_planner_validation():
    for args in [(0, 4, 8), (4, 0, 8), (4, 4, 6), (4, 4, 2), ((1 << 20) + 1, 4, 8)]:
        with pytest.raises(bg.BergsonError):
            bg.bergson_debug_xgemm_plan(*args)


def test_planners_on_random_shapes():
    """The same invariants over a few hundred random shapes (host only)."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @hyp.settings(max_examples=300, deadline=None, derandomize=True)
    @hyp.given(N=st.integers(1, 5_000_000), Q=st.integers(1, 50_000), topk=st.integers(1, 1024),
               ctas=st.integers(1, 200))
    def score(N, Q, topk, ctas):
        hyp.assume(topk <= N)
        pair_ok = Q < 129 or min(ctas, 160) >= 2
        if pair_ok:
            check_score_plan(N, Q, topk, ctas)

    @hyp.settings(max_examples=300, deadline=None, derandomize=True)
    @hyp.given(B=st.integers(1, 1 << 20), Q=st.integers(1, 1 << 16), K4=st.integers(1, 1 << 16))
    def xgemm(B, Q, K4):
        check_xgemm_plan(B, Q, 4 * K4)

    score()
    xgemm()


# --- documented size limits of the workspace queries --------------------------

def _ws_query(fn, *args):
    n = ctypes.c_size_t()
    st = getattr(bg.lib(), fn)(*args, ctypes.byref(n))
    return st, n.value


def test_workspace_queries_at_their_size_limits():
    L = bg.lib()
    # projection: B * T up to 2^37 tokens
    arr = (bg.bergson_layer * 1)(_layer(d_in=8, d_out=8))
    n = ctypes.c_size_t()
    assert L.bergson_project_grads_workspace(arr, 1, 1 << 20, 1 << 17, ctypes.byref(n)) == bg.BERGSON_OK
    assert 0 < n.value < (1 << 40)
    assert L.bergson_project_grads_workspace(arr, 1, (1 << 20) + 1, 1 << 17, ctypes.byref(n)) == \
        bg.BERGSON_EUNSUPPORTED
    # scoring: N < 2^31, Q <= 2^24, topk <= 1024
    st, n_big = _ws_query("bergson_score_topk_workspace", (1 << 31) - 1, 8192, 1 << 24, 1024)
    assert st == bg.BERGSON_OK and n_big >= (1 << 24) * 8192 * 2
    assert _ws_query("bergson_score_topk_workspace", 1 << 31, 8192, 16, 8)[0] == bg.BERGSON_EINVAL
    assert _ws_query("bergson_score_topk_workspace", 1 << 20, 8192, 16, 1025)[0] == \
        bg.BERGSON_EUNSUPPORTED
    assert _ws_query("bergson_score_topk_workspace", 1 << 20, 8192, (1 << 24) + 1, 8)[0] == \
        bg.BERGSON_EINVAL
    assert _ws_query("bergson_score_topk_workspace", 1 << 20, 8196, 16, 8)[0] == bg.BERGSON_EALIGN
    # on-the-fly scores / preconditioner application: B <= 2^20, Q <= 2^24, K <= 2^26
    st, n_otf = _ws_query("bergson_score_grads_workspace", 1 << 20, 1 << 12, 1 << 10)
    assert st == bg.BERGSON_OK and n_otf >= 2 * 4 * (1 << 20) * (1 << 12)   # x_hi and x_lo
    assert _ws_query("bergson_score_grads_workspace", (1 << 20) + 1, 64, 64)[0] == bg.BERGSON_EINVAL
    # Fisher: n <= 2^24 rows, K <= 65536; the preconditioner holds 4 K^2 floats
    assert _ws_query("bergson_fisher_fit_workspace", 1 << 24, 1 << 16)[0] == bg.BERGSON_OK
    assert _ws_query("bergson_fisher_fit_workspace", 1 << 24, (1 << 16) + 4)[0] == bg.BERGSON_EINVAL
    st, n_pre = _ws_query("bergson_fisher_preconditioner_workspace", 1 << 16)
    assert st == bg.BERGSON_OK and n_pre >= 4 * 4 * (1 << 32)
    # the queries apply their calls' alignment rules too
    assert _ws_query("bergson_score_grads_workspace", 32, 4098, 16)[0] == bg.BERGSON_EALIGN
    assert _ws_query("bergson_score_grads_workspace", 1 << 20, 64, 1 << 24)[0] == \
        bg.BERGSON_EUNSUPPORTED
    assert _ws_query("bergson_fisher_fit_workspace", 64, 258)[0] == bg.BERGSON_EALIGN
    assert _ws_query("bergson_fisher_preconditioner_workspace", 258)[0] == bg.BERGSON_EALIGN
    # aggregation: n < 2^31 rows
    assert _ws_query("bergson_aggregate_rows_workspace", (1 << 31) - 1)[0] == bg.BERGSON_OK
    assert _ws_query("bergson_aggregate_rows_workspace", 1 << 31)[0] == bg.BERGSON_EINVAL


@pytest.mark.parametrize("n_threads,n_devices", [(2, 1), (16, 4), (32, 64)])
def test_attribute_record_is_per_device_and_thread_safe(n_threads, n_devices):
    # Concurrent first calls from several host threads, on several (simulated)
    # devices: the kernel attribute is set exactly once per device.
    calls, failures = bg.bergson_debug_attr_once(n_threads, n_devices)
    assert calls == [1] * n_devices and failures == 0


def test_attribute_record_retries_a_failed_setting():
    calls, failures = bg.bergson_debug_attr_once(8, 3, fail_device=1)
    assert calls == [1, 2, 1] and failures == 1
    with pytest.raises(bg.BergsonError):
        bg.bergson_debug_attr_once(0, 3)


def test_moment_status_is_part_of_the_abi():
    # r_i, c_j > 0 is checked on the device (the values are device memory);
    # the status it records is a public code with a name and a host message.
    import re
    hdr = open(os.path.join(ROOT, "include", "bergson.h")).read()
    m = re.search(r"BERGSON_EMOMENT\s*=\s*(-?\d+)", hdr)
    assert m and int(m.group(1)) == bg.BERGSON_EMOMENT == -7
    assert bg.binding.STATUS_NAMES[bg.BERGSON_EMOMENT] == "BERGSON_EMOMENT"
    bg.bergson_debug_inject_status(bg.BERGSON_EMOMENT, 1)
    assert _proj([_layer()], B=0) == bg.BERGSON_EMOMENT
    assert "injected" in bg.bergson_last_error()
    assert _proj([_layer()], B=0) == bg.BERGSON_OK


def test_store_blocks_validation():
    f = bg.lib().bergson_build_store_blocks

    def call(offs, B=4, K=64, ld_proj=64, ld_store=64, row_offset=0, N_cap=4, n=None):
        arr = (ctypes.c_int64 * len(offs))(*offs)
        return f(FAKE, B, K, ld_proj, arr, len(offs) - 1 if n is None else n, FAKE, ld_store,
                 row_offset, N_cap, None, None)

    assert call([0, 32, 64], B=0) == bg.BERGSON_OK
    assert call([0, 64], B=0) == bg.BERGSON_OK
    assert call([8, 64]) == bg.BERGSON_EINVAL            # must start at 0
    assert call([0, 32]) == bg.BERGSON_EINVAL            # must end at K
    assert call([0, 32, 32, 64]) == bg.BERGSON_EINVAL    # empty block
    assert call([0, 40, 32, 64]) == bg.BERGSON_EINVAL    # decreasing
    assert call([0, 36, 64]) == bg.BERGSON_EALIGN        # not a multiple of 8
    assert call([0, 64], n=0) == bg.BERGSON_EINVAL
    assert call([0, 64], n=2049) == bg.BERGSON_EINVAL
    assert call([0, 64], ld_store=60) == bg.BERGSON_EINVAL
    assert call([0, 64], row_offset=1) == bg.BERGSON_EINVAL
    assert f(FAKE, 4, 64, 64, None, 1, FAKE, 64, 0, 4, None, None) == bg.BERGSON_EINVAL


def test_chunked_and_host_scoring_validation():
    L = bg.lib()
    ws = ctypes.c_size_t()
    assert L.bergson_score_topk_update_workspace(256, 8, 5, ctypes.byref(ws)) == 0
    full = ctypes.c_size_t()
    assert L.bergson_score_topk_workspace(100_000, 256, 8, 5, ctypes.byref(full)) == 0
    assert ws.value == full.value                       # independent of the chunk's rows
    assert L.bergson_score_topk_update_workspace(256, 8, 0, ctypes.byref(ws)) == bg.BERGSON_EINVAL
    assert L.bergson_score_topk_update_workspace(256, 8, 2000, ctypes.byref(ws)) == bg.BERGSON_EUNSUPPORTED

    def upd(N=10, row_base=0, topk=5, K=256, ld=256, init=1, wsb=1 << 30, fn=L.bergson_score_topk_update):
        return fn(FAKE, N, K, ld, row_base, FAKE, 8, K, topk, init, FAKE, FAKE, FAKE, wsb, None)

    # a chunk may hold fewer rows than topk; nothing runs without a device
    assert upd(N=3, topk=5) in (bg.BERGSON_ECUDA, bg.BERGSON_OK)
    assert upd(N=0) == bg.BERGSON_EINVAL
    assert upd(row_base=-1) == bg.BERGSON_EINVAL
    assert upd(row_base=(1 << 31) - 10) == bg.BERGSON_EINVAL
    assert upd(K=100, ld=104) == bg.BERGSON_EALIGN
    assert upd(wsb=16) == bg.BERGSON_EWORKSPACE
    assert upd(fn=L.bergson_score_bottomk_update, topk=2000) == bg.BERGSON_EUNSUPPORTED

    assert L.bergson_score_topk_host_workspace(1000, 256, 8, 5, ctypes.byref(ws)) == 0
    assert ws.value >= 2 * 1000 * 256 * 2 + full.value
    assert L.bergson_score_topk_host_workspace(0, 256, 8, 5, ctypes.byref(ws)) == bg.BERGSON_EINVAL

    def host(ptr=FAKE, N=1000, ld=256, chunk=100, topk=5, wsb=1 << 30):
        return L.bergson_score_topk_host(ptr, N, 256, ld, FAKE, 8, 256, topk, 0, chunk, FAKE, FAKE,
                                         FAKE, wsb, None, None)

    assert host(ptr=None) == bg.BERGSON_EINVAL
    assert host(chunk=0) == bg.BERGSON_EINVAL
    assert host(ld=260) == bg.BERGSON_EALIGN
    assert host(ptr=FAKE + 8) == bg.BERGSON_EALIGN
    assert host(topk=2000) == bg.BERGSON_EUNSUPPORTED
    assert host(N=3) == bg.BERGSON_EINVAL               # the whole store still needs topk rows
    assert host(wsb=1 << 16) == bg.BERGSON_EWORKSPACE
