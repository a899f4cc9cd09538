"""The in-grid split merge of the attention kernel (NLD_ATTN_MERGE_IN_GRID).

When a plan splits the KV range of each (sequence, KV head) into S partials
and the grid fits in one wave, this flag makes nld_block_attn merge the
partials inside the attention grid (split-combine rule: partials weighted by
their log-sum-exps) instead of launching the combine kernel. Checked here:
  - the in-grid merge, the combine kernel (the default) and the give-up path
    where no CTA waits and the last CTA of each unit to arrive merges every
    row (NLD_ATTN_MERGE_NO_WAIT) give the same bits, and match the fp64
    oracle on every row, in both passes;
  - every call leaves the workspace's merge counters consistent (per unit:
    arrival count equal to its base word, give-up bits clear), call after
    call;
  - a workspace whose counters are inconsistent is reported as
    NLD_DEVERR_MERGE_STATE (and the next call on a zeroed workspace is right);
  - plans that do not fit in one wave keep the combine kernel.
"""
import numpy as np
import pytest
import torch

from gpu_helpers import DeviceCase, compare_attn, oracle_full
from paper_2607_05722_gb300 import nld
from paper_2607_05722_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DIFF, VER = W.MODE_DIFFUSION, W.MODE_VERIFY


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05722_gb300 import build
    build.build()
    nld.lib()
    nld.nld_device_error(clear=True)
    yield
    assert nld.nld_device_error(clear=True) == 0, "a kernel flagged a device error"


# name, B, Hq, Hkv, D, P, bl, prefix lengths
SHAPES = [
    ("8b_like_L2000", 1, 32, 8, 128, 16, 16, [2000]),
    ("rep4_d64", 1, 4, 1, 64, 16, 8, [900]),
    ("ragged_b3_d64", 3, 8, 2, 64, 32, 5, [0, 130, 1500]),
    ("rows96_d128", 2, 6, 2, 128, 16, 32, [700, 1400]),
    ("rows160_mt2", 1, 10, 2, 128, 16, 32, [1800]),
    ("rows256_mt2_d64", 1, 16, 2, 64, 16, 32, [600]),
]


def counters_consistent(ws):
    w = ws[:nld.MERGE_CTR_BYTES].view(torch.int32).view(-1, 8).cpu().numpy()
    return bool(np.array_equal(w[:, 0], w[:, 1]) and not w[:, 2:].any())


def _case(spec, seed):
    name, B, Hq, Hkv, D, P, bl, prefix = spec
    return W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix, seed=seed)


def _run(dc, mode, params, ws):
    c = dc.case
    out = torch.full((c.batch, c.block_len, c.num_q_heads, c.head_dim), float("nan"), dtype=torch.bfloat16,
                     device="cuda")
    lse = torch.full((c.batch, c.num_q_heads, c.block_len), float("nan"), dtype=torch.float32, device="cuda")
    nld.nld_block_attn(params, dc.q[mode], dc.k, dc.v, dc.table, dc.prefix, c.block_len, mode, out, lse, ws)
    return out, lse


@pytest.mark.parametrize("spec", SHAPES, ids=[s[0] for s in SHAPES])
@pytest.mark.parametrize("splits", [0, 3, 7])
def test_in_grid_merge_matches_combine_and_oracle(orc, spec, splits):
    case = _case(spec, seed=sum(spec[7]) + 7 * splits + 1)
    dc = DeviceCase(case)
    bl = case.block_len
    IG = nld.NLD_ATTN_MERGE_IN_GRID
    base = dc.params(splits, flags=nld.NLD_ATTN_NO_CLUSTER | IG)
    sep = dc.params(splits, flags=nld.NLD_ATTN_NO_CLUSTER)
    nowait = dc.params(splits, flags=nld.NLD_ATTN_NO_CLUSTER | IG | nld.NLD_ATTN_MERGE_NO_WAIT)
    parts = nld.nld_block_attn_num_splits(base, bl)
    if parts < 2:
        pytest.skip("the plan has one split: nothing to merge")
    assert nld.nld_block_attn_kernels(base, bl) == 1, "one wave: the merge runs inside the attention grid"
    assert nld.nld_block_attn_kernels(sep, bl) == 2
    ws = nld.alloc_workspace(base, bl)
    for mode in (DIFF, VER):
        ro, rl = oracle_full(orc, case, mode)
        o1, l1 = _run(dc, mode, base, ws)
        o2, l2 = _run(dc, mode, sep, ws)
        o3, l3 = _run(dc, mode, nowait, ws)
        torch.cuda.synchronize()
        assert torch.equal(o1, o2) and torch.equal(l1, l2), "in-grid merge vs combine kernel"
        assert torch.equal(o1, o3) and torch.equal(l1, l3), "waiting vs last-one-out merge"
        compare_attn(o1, l1, ro, rl, f"{case.name} mode={mode} S={splits} partials={parts}")
        assert counters_consistent(ws), "merge counters consistent after the calls"


def test_repeated_calls_reuse_the_workspace(orc):
    case = _case(SHAPES[0], seed=5)
    dc = DeviceCase(case)
    p = dc.params(0, flags=nld.NLD_ATTN_MERGE_IN_GRID)
    assert nld.nld_block_attn_kernels(p, case.block_len) == 1
    ws = nld.alloc_workspace(p, case.block_len)
    assert ws is not None
    ro, rl = oracle_full(orc, case, VER)
    first = None
    for it in range(12):
        mode = VER if it % 2 == 0 else DIFF
        o, l = _run(dc, mode, p, ws)
        if mode == VER:
            if first is None:
                first = (o, l)
                compare_attn(o, l, ro, rl, "repeated")
            else:
                assert torch.equal(o, first[0]) and torch.equal(l, first[1]), f"call {it}"
    torch.cuda.synchronize()
    assert counters_consistent(ws)


def test_graph_replays_keep_counters_consistent(orc):
    """A CUDA graph of several calls replayed: every replay leaves the
    counters consistent and gives the same output."""
    case = _case(SHAPES[0], seed=6)
    dc = DeviceCase(case)
    p = dc.params(0, flags=nld.NLD_ATTN_PREFIX_READY | nld.NLD_ATTN_MERGE_IN_GRID)
    bl = case.block_len
    ws = nld.alloc_workspace(p, bl)
    out = torch.empty((1, bl, 32, 128), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((1, 32, bl), dtype=torch.float32, device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        nld.nld_block_attn(p, dc.q[DIFF], dc.k, dc.v, dc.table, dc.prefix, bl, DIFF, out, lse, ws, stream=s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            for _ in range(4):
                nld.nld_block_attn(p, dc.q[VER], dc.k, dc.v, dc.table, dc.prefix, bl, VER, out, lse, ws, stream=s)
        for _ in range(5):
            g.replay()
    torch.cuda.synchronize()
    assert counters_consistent(ws)
    ro, rl = oracle_full(orc, case, VER)
    compare_attn(out, lse, ro, rl, "graph replays")


def test_nonzero_counters_are_reported(orc):
    """A workspace handed over with inconsistent merge counters (arrival
    counts far past their base words): the kernel flags NLD_DEVERR_MERGE_STATE
    (its reads stay inside the workspace); a zeroed workspace then gives the
    right result again."""
    case = _case(SHAPES[0], seed=8)
    dc = DeviceCase(case)
    p = dc.params(0, flags=nld.NLD_ATTN_MERGE_IN_GRID)
    ws = nld.alloc_workspace(p, case.block_len)
    ws[:nld.MERGE_CTR_BYTES].view(torch.int32).view(-1, 8)[:, 0] = 1000
    nld.nld_device_error(clear=True)
    _run(dc, VER, p, ws)
    torch.cuda.synchronize()
    assert nld.nld_device_error(clear=True) & nld.NLD_DEVERR_MERGE_STATE
    ws.zero_()
    o, l = _run(dc, VER, p, ws)
    torch.cuda.synchronize()
    assert nld.nld_device_error(clear=True) == 0
    ro, rl = oracle_full(orc, case, VER)
    compare_attn(o, l, ro, rl, "after re-zeroing")


def test_plan_beyond_one_wave_keeps_the_combine(orc):
    """More CTAs than SMs: the partials go through the combine kernel."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    B, Hq, Hkv, bl = 24, 8, 4, 8
    case = W.make_block_attn_case("multiwave_split", B, Hq, Hkv, 128, block_len=bl, page_size=16,
                                  prefix_lens=list(range(100, 100 + 37 * B, 37)), seed=12)
    dc = DeviceCase(case)
    p = dc.params(3, flags=nld.NLD_ATTN_NO_CLUSTER | nld.NLD_ATTN_MERGE_IN_GRID)
    assert 3 * B * Hkv > sms
    assert nld.nld_block_attn_kernels(p, bl) == 2
    ws = nld.alloc_workspace(p, bl)
    for mode in (DIFF, VER):
        o, l = _run(dc, mode, p, ws)
        ro, rl = oracle_full(orc, case, mode)
        compare_attn(o, l, ro, rl, f"multiwave split mode={mode}")


def test_masked_pass_merges_in_grid(orc):
    """The table-mask instantiation (quadratic self-speculation) shares the
    epilogue: in-grid merge and combine give the same bits."""
    k = 3
    bl = 1 + k + k * k
    case = W.make_block_attn_case("quadss_merge", 1, 16, 4, 128, block_len=bl, page_size=16, prefix_lens=[1500],
                                  seed=31)
    dc = DeviceCase(case)
    table = nld.nld_quadss_block_mask(k)
    bm = torch.from_numpy(np.asarray(table, dtype=np.uint32).view(np.int32)).cuda()
    ro, rl, _ = orc.block_attn_masked(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                      case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, bl, table, case.scale)
    res = []
    for flags in (nld.NLD_ATTN_NO_CLUSTER | nld.NLD_ATTN_MERGE_IN_GRID, nld.NLD_ATTN_NO_CLUSTER):
        p = dc.params(5, flags=flags)
        ws = nld.alloc_workspace(p, bl)
        out = torch.empty((1, bl, 16, 128), dtype=torch.bfloat16, device="cuda")
        lse = torch.empty((1, 16, bl), dtype=torch.float32, device="cuda")
        nld.nld_block_attn_masked(p, dc.q[DIFF], dc.k, dc.v, dc.table, dc.prefix, bl, bm, out, lse, ws)
        res.append((out, lse))
        compare_attn(out, lse, ro, rl, f"quadss flags={flags}")
    assert torch.equal(res[0][0], res[1][0]) and torch.equal(res[0][1], res[1][1])
