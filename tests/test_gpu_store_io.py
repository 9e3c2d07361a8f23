"""On-disk store round trip (bergson_store_save / bergson_store_load)."""
import os

import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from paper_2606_11660_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = "cuda"


def test_save_append_memmap_load(tmp_path):
    g = wl.generator(31, "cpu")
    K = 264
    rows = torch.randn((50, K), generator=g)
    store = torch.zeros((50, K + 8), dtype=torch.float16, device=DEV)   # padded leading dim
    bg.bergson_build_store(rows.to(DEV), 50, K, True, store, 0)
    path = str(tmp_path / "store.f16")
    bg.bergson_store_save(store[:30], 30, K, path, 0)                   # first batch
    bg.bergson_store_save(store[30:], 20, K, path, 30)                  # appended batch
    assert os.path.getsize(path) == 50 * K * 2
    mm = np.memmap(path, dtype=np.float16, mode="r", shape=(50, K))
    np.testing.assert_array_equal(np.asarray(mm), store[:, :K].cpu().numpy())
    back = torch.full((20, K), float("nan"), dtype=torch.float16, device=DEV)
    bg.bergson_store_load(path, 25, 20, K, back)
    assert torch.equal(back, store[25:45, :K])
    with pytest.raises(bg.BergsonError):
        bg.bergson_store_load(path, 40, 20, K, back)                    # past the end
