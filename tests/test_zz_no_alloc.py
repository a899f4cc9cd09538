"""The allocation-free entry point, nld_block_attn_static_scratch.

It serves callers that cannot hand the library a workspace (for example a
plugin inside another runtime's enqueue step, or code held to a fixed memory
budget): the split partials live in a fixed 16 MiB array compiled into the
library. Its results must match nld_block_attn with a caller workspace, call
after call, since every call reuses the same array.

This file is collected last on purpose, so a failure here comes after every
other test has run; it also passes when run alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from gpu_helpers import MAX_ABS, REL_L2, DeviceCase
from paper_2607_05722_gb300 import nld
from paper_2607_05722_gb300 import workloads as W

pytestmark = pytest.mark.gpu

STATIC_SCRATCH_BYTES = 16 << 20


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05722_gb300 import build
    build.build()
    nld.lib()


def _static_call(dc, params, mode, out, lse):
    c = dc.case
    L = nld.lib()
    return L.nld_block_attn_static_scratch(ctypes.byref(params), ctypes.c_void_p(dc.q[mode].data_ptr()),
                                           ctypes.c_void_p(dc.k.data_ptr()), ctypes.c_void_p(dc.v.data_ptr()),
                                           ctypes.c_void_p(dc.table.data_ptr()), ctypes.c_void_p(dc.prefix.data_ptr()),
                                           c.block_len, mode, ctypes.c_void_p(out.data_ptr()),
                                           ctypes.c_void_p(lse.data_ptr()),
                                           ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _close(a, b):
    a64, b64 = a.float().cpu().double().numpy(), b.float().cpu().double().numpy()
    max_abs = float(np.abs(a64 - b64).max())
    rel = float(np.linalg.norm(a64 - b64) / max(np.linalg.norm(b64), 1e-30))
    return max_abs <= MAX_ABS and rel <= REL_L2


@pytest.mark.parametrize("name", ["8b_b1_h32x8_d128_L4096_bl16", "tiny_b1_h4x1_d64_L256_bl8"])
def test_static_scratch_matches_workspace_entry_twice(name):
    wl = W.make_workload(name, seed=3)
    dc = DeviceCase(wl.attn)
    c = wl.attn
    params = dc.params(0)
    need = nld.nld_block_attn_workspace_size(params, c.block_len)
    assert need <= STATIC_SCRATCH_BYTES
    if name.startswith("8b"):
        assert need > 0, "this case must exercise the split partials"
    for mode in (W.MODE_DIFFUSION, W.MODE_VERIFY):
        ref_out, ref_lse = dc.run(mode)
        for _ in range(2):  # the array keeps the previous call's contents
            out = torch.full_like(ref_out, float("nan"))
            lse = torch.full_like(ref_lse, float("nan"))
            assert _static_call(dc, params, mode, out, lse) == 0
            torch.cuda.synchronize()
            assert _close(out, ref_out)
            assert torch.allclose(lse, ref_lse, atol=2e-3, rtol=0)


def test_static_scratch_rejects_oversized_plan():
    # An explicit 127 pieces of the 32800-token range (no cluster size divides
    # 127) round to 272-token splits, i.e. 121 partials of 32 rows x 32 heads
    # x 128 dims in bf16: about 32 MB, more than the 16 MiB array.
    wl = W.make_workload("long_b1_h32x8_d128_L32768_bl32", seed=0, prefix_override=[32768])
    dc = DeviceCase(wl.attn)
    params = dc.params(127)
    plan = nld.nld_block_attn_plan(params, 32, 148)
    assert (plan["splits"], plan["chunk"], plan["cluster"], plan["partials"]) == (121, 272, 1, 121)
    assert nld.nld_block_attn_workspace_size(params, 32) >= 121 * 32 * 32 * 128 * 2 > STATIC_SCRATCH_BYTES
    out = torch.zeros((1, 32, 32, 128), dtype=torch.bfloat16, device="cuda")
    lse = torch.zeros((1, 32, 32), dtype=torch.float32, device="cuda")
    assert _static_call(dc, params, W.MODE_VERIFY, out, lse) == 3  # NLD_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.count_nonzero(out) == 0
