"""bergson_project_grads_noalloc: projected gradients without a workspace.

Some callers cannot give the library device memory for its scratch: plugin
or callback interfaces that hand over only input and output buffers, runtimes
that own every byte of device memory through their own pool, and loops that
must not call cudaMalloc because it can synchronise the device or fail when
memory is short.  For them the library runs the regular path on a fixed
static scratch array (BERGSON_NOALLOC_SCRATCH_BYTES) and allocates nothing.

These tests call that entry point through the C ABI and hold its results to
the regular entry point's (which gets a torch-allocated workspace).  Every call
reuses the same scratch array, so a request is checked on consecutive calls
with a different request (other modules and k, a bias block, no mask, more
tokens) run on the same scratch in between: a stale descriptor, counter or
partial sum left by the other request would show.  The device's free memory
is read before the warm-up call that makes the driver reserve the array and
must not move after it.  The file is named so that pytest collects it last.
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
SCRATCH = 32 << 20


def _request_a():
    specs = [wl.ModuleSpec("qkv", 768, 2304), wl.ModuleSpec("attn_out", 768, 768),
             wl.ModuleSpec("mlp_down", 3072, 768)]
    B, T = 4, 700
    gl, _, ld = make_layers(specs, B, T, [(16, 16), (16, 16), (32, 16)], input_scale=True)
    g = wl.generator(9, "cpu")
    mask = (torch.rand((B, T), generator=g) > 0.1).to(torch.uint8).to(DEV)
    return gl, B, T, mask, ld


def _request_b():
    # other modules and (k_in, k_out), bias blocks after the weight blocks, no mask, more tokens
    specs = [wl.ModuleSpec("up", 2048, 6144), wl.ModuleSpec("small", 1024, 512)]
    B, T = 3, 2500
    gl, _, ld = make_layers(specs, B, T, [(32, 32), (64, 16)], data_seed=5, input_scale=True)
    for ly in gl:
        ly.bias_col_offset = ld
        ld += ly.k_out
    return gl, B, T, None, ld


def _noalloc(arr, n, B, T, mask, out, ld, stream):
    return bg.lib().bergson_project_grads_noalloc(
        arr, n, B, T, None if mask is None else mask.data_ptr(),
        None if out is None else out.data_ptr(), ld, stream)


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    reqs = [_request_a(), _request_b()]
    want = [np32(run_project(gl, B, T, mask, ld)).astype(np.float64)
            for gl, B, T, mask, ld in reqs]
    arrs = [binding._layer_array(r[0]) for r in reqs]
    for gl, B, T, _, _ in reqs:
        assert bg.bergson_project_grads_workspace(gl, B, T) <= SCRATCH
    # every output buffer exists before the first free-memory reading
    outs = {i: torch.empty((r[1], r[4]), dtype=torch.float32, device=DEV)
            for i, r in enumerate(reqs)}
    stream = torch.cuda.current_stream().cuda_stream
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]

    # warm-up: B = 0 and out = NULL looks up (and, on first use, reserves) the
    # scratch array on the current device and enqueues nothing
    gl, _, T, _, ld = reqs[0]
    st = _noalloc(arrs[0], len(gl), 0, T, None, None, ld, stream)
    assert st == bg.BERGSON_OK, bg.bergson_last_error()
    torch.cuda.synchronize()
    free_warm = torch.cuda.mem_get_info()[0]
    reserved = free_before - free_warm
    print(f"warm-up reserved {reserved / 2**20:.1f} MiB on the device")
    assert 0 <= reserved <= 2 * SCRATCH

    for call, i in enumerate([0, 1, 0, 1]):
        gl, B, T, mask, ld = reqs[i]
        out = outs[i]
        out.fill_(float("nan"))
        st = _noalloc(arrs[i], len(gl), B, T, mask, out, ld, stream)
        assert st == bg.BERGSON_OK, bg.bergson_last_error()
        assert bg.bergson_sync_status() == bg.BERGSON_OK, bg.bergson_last_error()
        got = np32(out).astype(np.float64)
        assert np.all(np.isfinite(got)), f"call {call} (request {i}): unwritten outputs"
        err = rel_frobenius(got, want[i]).max()
        assert err <= TIGHT, f"call {call} (request {i}) differs: {err:.3e}"
        assert torch.cuda.mem_get_info()[0] == free_warm, \
            f"device memory changed at call {call}"


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
    assert need.value > SCRATCH
    st = bg.lib().bergson_project_grads_noalloc(arr, 8, 2, 256, None, fake, 8 * 4096, None)
    assert st == bg.BERGSON_EWORKSPACE
    assert "fixed" in bg.bergson_last_error()
