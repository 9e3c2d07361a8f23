"""GPU parity of query aggregation (bergson_aggregate_rows) against the oracle."""
import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from oracle import bergson_oracle as orc
from paper_2606_11660_gb300 import workloads as wl
from tests._util import np32

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.mark.parametrize("mode", [bg.BERGSON_AGG_SUM, bg.BERGSON_AGG_MEAN])
@pytest.mark.parametrize("normalize", [True, False])
def test_aggregate_groups(mode, normalize):
    g = wl.generator(8, "cpu")
    n, K = 23, 12288
    rows = torch.randn((n, K + 4), generator=g) * 0.1
    rows[5] = 0.0
    offs = [0, 4, 4, 11, 12, 23]                       # includes an empty group
    offsets = torch.tensor(offs, dtype=torch.int64, device=DEV)
    x = rows.to(DEV)[:, :K]                             # padded leading dimension
    out = torch.full((len(offs) - 1, K), float("nan"), device=DEV)
    ws = bg.workspace_tensor(bg.bergson_aggregate_rows_workspace(n), DEV)
    bg.bergson_aggregate_rows(x, n, K, offsets, mode, normalize, out, ws)
    assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
    want = orc.aggregate_rows(rows[:, :K].numpy(), offs, mode, normalize)
    got = np32(out).astype(np.float64)
    np.testing.assert_allclose(got, want, atol=2e-6 * max(1.0, np.abs(want).max()), rtol=1e-5)
    np.testing.assert_array_equal(got[1], 0.0)


def test_aggregated_query_scores_are_member_means():
    g = wl.generator(9, "cpu")
    K = 512
    store_rows = torch.randn((300, K), generator=g)
    store = torch.empty((300, K), dtype=torch.float16, device=DEV)
    bg.bergson_build_store(store_rows.to(DEV), 300, K, True, store, 0)
    members = torch.randn((6, K), generator=g).to(DEV)
    offsets = torch.tensor([0, 6], dtype=torch.int64, device=DEV)
    q = torch.empty((1, K), device=DEV)
    ws = bg.workspace_tensor(bg.bergson_aggregate_rows_workspace(6), DEV)
    bg.bergson_aggregate_rows(members, 6, K, offsets, bg.BERGSON_AGG_MEAN, True, q, ws)
    torch.cuda.synchronize()
    s16 = store.float().cpu().numpy().astype(np.float64)
    mem = np32(members).astype(np.float64)
    mem /= np.linalg.norm(mem, axis=1, keepdims=True)
    np.testing.assert_allclose(s16 @ np32(q)[0].astype(np.float64), (s16 @ mem.T).mean(axis=1),
                               atol=1e-6)
