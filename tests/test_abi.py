"""The C ABI library without a GPU: it loads, exports every function that
include/nld.h declares, and rejects bad arguments on the host before any
CUDA call (the checks below return before the library touches a device)."""
import ctypes
import os

import numpy as np
import pytest

from paper_2607_05722_gb300 import build, nld

FAKE = ctypes.c_void_p(0x10000)  # aligned, never dereferenced: every call below fails a host check first


@pytest.fixture(scope="module")
def L():
    build.build()
    return nld.lib()


def test_header_declares_the_abi():
    names = nld.header_functions()
    for f in ("nld_block_attn", "nld_block_attn_partials", "nld_block_attn_workspace_size", "nld_block_attn_num_splits",
              "nld_split_kv_combine", "nld_accept", "nld_unmask", "nld_status_string", "nld_device_error",
              "nld_check_wait_timeout"):
        assert f in names, f


def test_library_exports_every_declared_symbol(L):
    for f in nld.header_functions():
        assert hasattr(L, f), f"libnld.so does not export {f}"


def test_status_strings(L):
    for code, name in ((0, "NLD_OK"), (1, "NLD_ERR_INVALID_ARG"), (2, "NLD_ERR_UNSUPPORTED"),
                       (3, "NLD_ERR_WORKSPACE"), (4, "NLD_ERR_CUDA")):
        assert nld.nld_status_string(code) == name


def params(**kw):
    base = dict(batch=1, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16, num_pages=300,
                max_pages_per_seq=257, num_splits=3, softmax_scale=0.0)
    base.update(kw)
    return nld.make_params(**base)


def test_split_plan_and_workspace_size(L):
    p = params(num_splits=19)
    assert nld.nld_block_attn_num_splits(p, 16) == 19
    # 4112 tokens / 19 -> 217 -> 224 per split -> 19 splits
    S, B, Hq, bl, D = 19, 1, 32, 16, 128
    o = S * B * Hq * bl * D * 2  # bf16 partial rows, then fp32 log-sum-exps
    assert nld.nld_block_attn_workspace_size(p, 16) == ((o + 255) // 256) * 256 + S * B * Hq * bl * 4
    assert nld.nld_block_attn_workspace_size(params(num_splits=1), 16) == 0
    # 16 pieces run as two clusters of 8 (tcgen05 kernel, 64 packed rows): 2 partials
    assert nld.nld_block_attn_num_splits(params(num_splits=16), 16) == 2
    assert nld.nld_block_attn_workspace_size(params(num_splits=16), 16) == \
        ((2 * Hq * bl * D * 2 + 255) // 256) * 256 + 2 * Hq * bl * 4
    # without clusters every piece is a partial
    assert nld.nld_block_attn_num_splits(params(num_splits=16, flags=nld.NLD_ATTN_NO_CLUSTER), 16) == 16
    # 4 pieces (chunk >= 16 tokens of 64) merge in one cluster: final output, no workspace
    assert nld.nld_block_attn_num_splits(params(num_splits=64, max_pages_per_seq=4), 8) == 1
    assert nld.nld_block_attn_workspace_size(params(num_splits=8), 16) == 0
    # 160 packed rows with an even block length: two CTAs per split (16 block
    # slots each), no clusters, so 8 pieces leave 8 partials; with an odd
    # block length (5 x 31 = 155 rows) one CTA with two M tiles, and 8 pieces
    # merge in one cluster
    assert nld.nld_block_attn_num_splits(params(num_q_heads=40, num_splits=8), 32) == 8
    assert nld.nld_block_attn_num_splits(params(num_q_heads=40, num_splits=8), 31) == 1


@pytest.mark.parametrize("kw,bl,code", [
    (dict(num_q_heads=30), 16, 1),          # Hq % Hkv != 0
    (dict(head_dim=96), 16, 2),             # head_dim not built
    (dict(page_size=24), 16, 1),            # not a power of two
    (dict(page_size=8), 16, 1),             # below 16
    (dict(page_size=512), 16, 1),           # above 256
    (dict(num_splits=129), 16, 1),          # too many splits
    (dict(), 0, 1),                         # block_len 0
    (dict(), 33, 1),                        # block_len > 32
    (dict(num_q_heads=72, num_kv_heads=8), 32, 2),  # 9 * 32 = 288 packed rows > 256
    (dict(batch=0), 16, 1),
    (dict(flags=2), 16, 1),                 # unknown flag bit
    (dict(flags=8), 16, 1),                 # unknown flag bit
])
def test_block_attn_rejects_bad_shapes(L, kw, bl, code):
    p = params(**kw)
    st = L.nld_block_attn(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, FAKE, bl, 0, FAKE, None, None, 0, None)
    assert st == code


def test_block_attn_rejects_bad_pointers_and_workspace(L):
    p = params()
    st = L.nld_block_attn(ctypes.byref(p), None, FAKE, FAKE, FAKE, FAKE, 16, 0, FAKE, None, None, 0, None)
    assert st == 1
    mis = ctypes.c_void_p(0x10008)  # 8-byte aligned, not 16
    st = L.nld_block_attn(ctypes.byref(p), FAKE, mis, FAKE, FAKE, FAKE, 16, 0, FAKE, None, None, 0, None)
    assert st == 1
    st = L.nld_block_attn(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, FAKE, 16, 2, FAKE, None, None, 0, None)
    assert st == 1  # mode
    need = nld.nld_block_attn_workspace_size(p, 16)
    st = L.nld_block_attn(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, FAKE, 16, 0, FAKE, None, FAKE, need - 1, None)
    assert st == 3
    st = L.nld_block_attn(ctypes.byref(p), FAKE, FAKE, FAKE, FAKE, FAKE, 16, 0, FAKE, None, None, 0, None)
    assert st == 3


def test_decisions_reject_bad_sizes(L):
    assert L.nld_accept(FAKE, FAKE, 1, 33, FAKE, None) == 1
    assert L.nld_accept(FAKE, FAKE, 0, 8, FAKE, None) == 1
    assert L.nld_accept(None, FAKE, 1, 8, FAKE, None) == 1
    assert L.nld_unmask(FAKE, 1, 8, 9, FAKE, None, None) == 1
    assert L.nld_unmask(FAKE, 1, 8, 0, FAKE, None, None) == 1
    assert L.nld_unmask(FAKE, 1, 40, 4, FAKE, None, None) == 1
    assert L.nld_unmask_threshold(FAKE, 1, 33, 0.5, FAKE, None, None) == 1
    assert L.nld_unmask_threshold(FAKE, 0, 8, 0.5, FAKE, None, None) == 1
    assert L.nld_unmask_threshold(FAKE, 1, 0, 0.5, FAKE, None, None) == 1
    assert L.nld_unmask_threshold(None, 1, 8, 0.5, FAKE, None, None) == 1
    assert L.nld_greedy_accept(FAKE, FAKE, FAKE, 1, 33, FAKE, None, None) == 1
    assert L.nld_greedy_accept(FAKE, FAKE, FAKE, 0, 8, FAKE, None, None) == 1
    assert L.nld_greedy_accept(FAKE, None, FAKE, 1, 8, FAKE, None, None) == 1
    assert L.nld_greedy_accept(FAKE, FAKE, FAKE, 1, 8, FAKE, ctypes.c_void_p(0x10002), None) == 1
    assert L.nld_logits_ensemble_argmax(FAKE, FAKE, 1, 8, 8, 1.5, FAKE, FAKE, None) == 1
    assert L.nld_logits_ensemble_argmax(FAKE, FAKE, 1, 8, 8, float("nan"), FAKE, FAKE, None) == 1
    assert L.nld_logits_ensemble_argmax(FAKE, FAKE, 1, 9, 12, 0.5, FAKE, FAKE, None) == 1
    assert L.nld_logits_argmax(FAKE, 0, 8, 8, FAKE, FAKE, None) == 1
    assert L.nld_split_kv_combine(FAKE, FAKE, 0, 1, 4, 8, 128, FAKE, None, None) == 1
    assert L.nld_split_kv_combine(FAKE, FAKE, 2, 1, 4, 8, 80, FAKE, None, None) == 2


def test_quadss_table_matches_oracle(L, orc):
    """The library's host-side table of quadratic self-speculation (written on
    its own) equals the oracle's; k beyond 5 (more than 32 slots) is refused."""
    for k in range(1, 6):
        assert np.array_equal(nld.nld_quadss_block_mask(k), orc.quadss_mask(k)), f"k={k}"
    for k in (0, 6):
        with pytest.raises(ValueError):
            nld.nld_quadss_block_mask(k)


def test_no_cpu_fallback_without_library(tmp_path):
    with pytest.raises(RuntimeError):
        nld.lib(str(tmp_path / "missing.so"))


def test_wait_timeout_check_rejects_bad_limits(L):
    # argument checks come before any device use
    assert L.nld_check_wait_timeout(0, None) == 1
    assert L.nld_check_wait_timeout(2_000_000_000, None) == 1


# ---------------------------------------------------------------------------
# the split plan (host logic, no device): 152 SMs as on GB300
# ---------------------------------------------------------------------------

def _plan(B, Hq, Hkv, D, P, prefix_max, bl, splits=0, sms=152):
    pages = (prefix_max + bl + P - 1) // P
    p = nld.make_params(B, Hq, Hkv, D, P, B * pages, pages, splits, 0.0, 0)
    return nld.nld_block_attn_plan(p, bl, sms), pages * P


def test_plan_8b_shape_takes_whole_paired_products(L):
    plan, tokens = _plan(1, 32, 8, 128, 16, 4096, 16)
    assert plan == {"splits": 17, "chunk": 256, "cluster": 1, "partials": 17}
    assert plan["splits"] * 8 <= 152


def test_plan_long_prefix_streams_whole_tiles(L):
    plan, tokens = _plan(1, 32, 8, 128, 16, 32768, 32)
    assert plan["splits"] == 19 and plan["chunk"] % 64 == 0
    assert (plan["splits"] - 1) * plan["chunk"] < tokens <= plan["splits"] * plan["chunk"]


def test_plan_many_units_one_split(L):
    plan, _ = _plan(32, 32, 8, 128, 16, 8192, 8)  # 256 units > 152 SMs
    assert plan["splits"] == 1 and plan["partials"] == 1


def test_plan_ragged_batch_caps_pieces_at_2048_tokens(L):
    # 64 units fit one wave: floor(152/64) = 2 splits, raised so that no piece
    # of the 8208-token range exceeds 2048 tokens; pieces end on whole tiles
    plan, tokens = _plan(8, 32, 8, 128, 16, 8192, 8)
    assert tokens == 8208
    assert plan["splits"] == -(-tokens // 2048) == 5
    assert plan["chunk"] % 64 == 0 and plan["chunk"] <= 2048


@pytest.mark.parametrize("B,Hq,Hkv,D,P,L_,bl", [(1, 4, 1, 64, 256, 256, 8), (2, 8, 2, 128, 16, 300, 16),
                                               (3, 4, 2, 64, 32, 200, 5), (16, 40, 8, 128, 16, 16384, 32),
                                               (1, 16, 2, 64, 16, 100, 32), (5, 12, 4, 128, 64, 1000, 20)])
def test_plan_invariants(L, B, Hq, Hkv, D, P, L_, bl):
    for sms in (1, 8, 148, 152, 160):
        for S in (0, 1, 3, 7, 19):
            plan, tokens = _plan(B, Hq, Hkv, D, P, L_, bl, splits=S, sms=sms)
            assert plan["chunk"] % 16 == 0 and plan["chunk"] > 0
            assert plan["splits"] * plan["chunk"] >= tokens
            assert (plan["splits"] - 1) * plan["chunk"] < tokens
            assert 1 <= plan["splits"] <= 128 and plan["partials"] == plan["splits"] // plan["cluster"]
            if S:
                assert plan["splits"] <= S


def test_plan_without_clusters(L):
    """NLD_ATTN_NO_CLUSTER: every piece of an explicit split count is a
    partial (pieces are whole 16-token groups, so 64 pieces of 32800 tokens
    are 63 of 528)."""
    for S in (2, 4, 8, 16, 32, 64):
        plan, tokens = _plan(1, 32, 8, 128, 16, 32768, 32, splits=S)
        assert plan["cluster"] == (8 if S % 8 == 0 else S)
        p = nld.make_params(1, 32, 8, 128, 16, 2050, 2050, S, 0.0, nld.NLD_ATTN_NO_CLUSTER)
        nc = nld.nld_block_attn_plan(p, 32, 152)
        assert nc["cluster"] == 1 and nc["partials"] == nc["splits"]
        assert S - 1 <= nc["splits"] <= S


def test_flags_accepted(L):
    for f in (nld.NLD_ATTN_PREFIX_READY, nld.NLD_ATTN_NO_CLUSTER, 5):
        assert nld.nld_block_attn_workspace_size(params(flags=f), 16) > 0


def test_plan_rejects_bad_arguments(L):
    p = nld.make_params(1, 32, 8, 128, 16, 300, 300, 0, 0.0, 0)
    with pytest.raises(nld.NldError):
        nld.nld_block_attn_plan(p, 16, 0)
    with pytest.raises(nld.NldError):
        nld.nld_block_attn_plan(p, 33, 152)
