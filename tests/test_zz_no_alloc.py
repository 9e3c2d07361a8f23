"""bergson_project_grads_noalloc: projected gradients without a workspace.

Some callers cannot give the library device memory for its scratch: plugin
or callback interfaces that hand over only input and output buffers, runtimes
that own every byte of device memory through their own pool, and loops that
must not call cudaMalloc because it can synchronise the device or fail when
memory is short.  For them the library runs the regular path on a fixed
static scratch array (BERGSON_NOALLOC_SCRATCH_BYTES) and allocates nothing.

These tests call that entry point through the C ABI and hold its results to
the regular entry point's (which gets a torch-allocated workspace), on two
calls in a row, since every call reuses the same scratch array.  The file is
named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2606_11660_gb300 as bg
from paper_2606_11660_gb300 import binding
from paper_2606_11660_gb300 import workloads as wl
from tests._util import make_layers, np32, rel_frobenius, run_project

pytestmark = pytest.mark.gpu
DEV = "cuda"
TIGHT = 1e-4      # same bound the parity tests use for projected gradients


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    specs = [wl.ModuleSpec("qkv", 768, 2304), wl.ModuleSpec("attn_out", 768, 768),
             wl.ModuleSpec("mlp_down", 3072, 768)]
    B, T = 4, 700
    gl, _, ld = make_layers(specs, B, T, [(16, 16), (16, 16), (32, 16)], input_scale=True)
    g = wl.generator(9, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.1).to(torch.uint8).to(DEV)
    want = np32(run_project(gl, B, T, mask, ld)).astype(np.float64)

    arr = binding._layer_array(gl)
    stream = torch.cuda.current_stream().cuda_stream
    free_after_first = None
    for call in range(2):
        out = torch.full((B, ld), float("nan"), dtype=torch.float32, device=DEV)
        st = bg.lib().bergson_project_grads_noalloc(arr, len(gl), B, T, mask.data_ptr(),
                                                   out.data_ptr(), ld, stream)
        assert st == bg.BERGSON_OK, bg.bergson_last_error()
        assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
        got = np32(out).astype(np.float64)
        assert np.all(np.isfinite(got)), f"call {call}: unwritten outputs"
        assert rel_frobenius(got, want).max() <= TIGHT, f"call {call} differs"
        free = torch.cuda.mem_get_info()[0]
        if free_after_first is None:
            free_after_first = free
        else:
            assert free == free_after_first, "device memory changed between calls"


def test_noalloc_rejects_requests_larger_than_its_scratch():
    # 8 modules of 8192 -> 8192 with k = 64 need 8 * 16384 * 128 * 2 B = 32 MiB of
    # projection slices alone, more than the fixed scratch; nothing is enqueued.
    fake = 0x7F0000000000
    L = bg.bergson_layer(A=fake, G=fake, d_in=8192, d_out=8192, k_in=64, k_out=64, seed_in=1,
                         seed_out=2, proj_kind=0, flags=0, r=None, c=None, out_col_offset=0)
    arr = (bg.bergson_layer * 8)()
    for m in range(8):
        arr[m] = L
        arr[m].out_col_offset = m * 4096
    need = ctypes.c_size_t()
    assert bg.lib().bergson_project_grads_workspace(arr, 8, 2, 256, ctypes.byref(need)) == 0
    assert need.value > (32 << 20)
    st = bg.lib().bergson_project_grads_noalloc(arr, 8, 2, 256, None, fake, 8 * 4096, None)
    assert st == bg.BERGSON_EWORKSPACE
    assert "fixed" in bg.bergson_last_error()
