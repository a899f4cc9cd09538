"""CUDA path vs the fp64 oracle, through the C ABI, on seeded inputs.

Bars: accept/unmask bit-exact; attention max-abs <= 1e-2 and rel-L2 <= 5e-3
against the fp64 oracle (bf16 inputs, fp32 accumulation), lse within 2e-3.
Small cases run the oracle on every row; the full-size workloads run in the
launch configuration the bench times (automatic split count) and compare a
sample of rows the oracle computes one by one.
"""
import math

import numpy as np
import pytest
import torch

import oracle_pins
from gpu_helpers import DeviceCase, compare_attn, oracle_full, rows_per_unit, sample_rows
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


# ---------------------------------------------------------------------------
# token decisions: bit-exact
# ---------------------------------------------------------------------------

def gpu_accept(d, v):
    dt, vt = torch.from_numpy(d).cuda(), torch.from_numpy(v).cuda()
    acc = torch.full((d.shape[0],), -7, dtype=torch.int32, device="cuda")
    nld.nld_accept(dt, vt, acc)
    return acc.cpu().numpy()


def gpu_unmask(conf, k):
    ct = torch.from_numpy(np.ascontiguousarray(conf)).cuda()
    pos = torch.full((conf.shape[0], k), -7, dtype=torch.int32, device="cuda")
    nsel = torch.full((conf.shape[0],), -7, dtype=torch.int32, device="cuda")
    nld.nld_unmask(ct, k, pos, nsel)
    return pos.cpu().numpy(), nsel.cpu().numpy()


def gpu_unmask_threshold(conf, thr):
    ct = torch.from_numpy(np.ascontiguousarray(conf, dtype=np.float32)).cuda()
    pos = torch.full(conf.shape, -7, dtype=torch.int32, device="cuda")
    nsel = torch.full((conf.shape[0],), -7, dtype=torch.int32, device="cuda")
    nld.nld_unmask_threshold(ct, float(np.float32(thr)), pos, nsel)
    return pos.cpu().numpy(), nsel.cpu().numpy()


def gpu_greedy(pred, target, conf):
    pt = torch.from_numpy(np.ascontiguousarray(pred, dtype=np.int32)).cuda()
    tt = torch.from_numpy(np.ascontiguousarray(target, dtype=np.int32)).cuda()
    ct = torch.from_numpy(np.ascontiguousarray(conf, dtype=np.float32)).cuda()
    pos = torch.full(conf.shape, -7, dtype=torch.int32, device="cuda")
    nsel = torch.full((conf.shape[0],), -7, dtype=torch.int32, device="cuda")
    nld.nld_greedy_accept(pt, tt, ct, pos, nsel)
    return pos.cpu().numpy(), nsel.cpu().numpy()


def tied_confidences(rng, B, n):
    conf = rng.integers(0, 5, size=(B, n)).astype(np.float32) / 4
    conf[rng.random((B, n)) < 0.2] = -np.inf
    conf[rng.random((B, n)) < 0.05] = np.nan
    z = rng.random((B, n)) < 0.05
    conf[z] = np.where(rng.random(z.sum()) < 0.5, 0.0, -0.0)
    return conf


def test_unmask_threshold_golden_cases():
    for c, thr, pos, nsel in oracle_pins.read_golden("unmask_threshold_cases.txt"):
        conf = np.array([[float(x) for x in c.split()]], dtype=np.float32)
        p, s = gpu_unmask_threshold(conf, float(thr))
        assert p[0].tolist() == [int(x) for x in pos.split()] and int(s[0]) == int(nsel), f"{c} | {thr}"


@pytest.mark.parametrize("n", [1, 5, 8, 16, 31, 32])
def test_unmask_threshold_matches_oracle(orc, n):
    rng = np.random.default_rng(300 + n)
    conf = tied_confidences(rng, 257, n)
    for thr in (-np.inf, -1.0, 0.0, 0.25, 0.5, 0.75, 1.0, np.inf, np.nan):
        p, s = gpu_unmask_threshold(conf, thr)
        po, so = orc.unmask_threshold(conf, thr)
        assert np.array_equal(p, po) and np.array_equal(s, so), f"n={n} thr={thr}"
    conf = rng.random((5000, n), dtype=np.float32)  # many CTAs, no ties
    p, s = gpu_unmask_threshold(conf, 0.9)
    po, so = orc.unmask_threshold(conf, 0.9)
    assert np.array_equal(p, po) and np.array_equal(s, so)


def test_greedy_accept_golden_cases():
    for pr, tg, c, pos, nsel in oracle_pins.read_golden("greedy_accept_cases.txt"):
        row = lambda t, dt: np.array([[float(x) for x in t.split()]], dtype=dt)
        p, s = gpu_greedy(row(pr, np.int32), row(tg, np.int32), row(c, np.float32))
        assert p[0].tolist() == [int(x) for x in pos.split()] and int(s[0]) == int(nsel), f"{pr} | {tg} | {c}"


@pytest.mark.parametrize("n", [1, 7, 8, 16, 32])
def test_greedy_accept_matches_oracle(orc, n):
    rng = np.random.default_rng(400 + n)
    for p_match in (0.0, 0.1, 0.5, 1.0):
        conf = tied_confidences(rng, 257, n)
        target = rng.integers(0, 131072, size=(257, n)).astype(np.int32)
        pred = np.where(rng.random((257, n)) < p_match, target, rng.integers(0, 131072, size=(257, n))).astype(np.int32)
        p, s = gpu_greedy(pred, target, conf)
        po, so = orc.greedy_accept(pred, target, conf)
        assert np.array_equal(p, po) and np.array_equal(s, so), f"n={n} p={p_match}"


def test_greedy_accept_chain(orc):
    """Iterated greedy acceptance until a 32-position block is unmasked (Sec. 5):
    each side chains its own commits; they agree at every iteration."""
    rng = np.random.default_rng(41)
    B, n = 64, 32
    target = rng.integers(0, 131072, size=(B, n)).astype(np.int32)
    conf_g = rng.random((B, n), dtype=np.float32)
    conf_o = conf_g.copy()
    for it in range(n):
        fresh = rng.random((B, n), dtype=np.float32)
        pred = np.where(rng.random((B, n)) < 0.4, target, target + 1).astype(np.int32)
        cg = np.where(conf_g == -np.inf, -np.inf, fresh).astype(np.float32)
        co = np.where(conf_o == -np.inf, -np.inf, fresh).astype(np.float32)
        pg, sg = gpu_greedy(pred, target, cg)
        po, so = orc.greedy_accept(pred, target, co)
        assert np.array_equal(pg, po) and np.array_equal(sg, so), f"iteration {it}"
        for b in range(B):
            conf_g[b, pg[b, :sg[b]]] = -np.inf
            conf_o[b, po[b, :so[b]]] = -np.inf
    assert np.all(conf_g == -np.inf), "the block is fully unmasked within n iterations"


# ---------------------------------------------------------------------------
# block KV commit
# ---------------------------------------------------------------------------

def bits_dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def dev_bits(t):
    return t.cpu().view(torch.int16).numpy().view(np.uint16)


def commit_case(seed, B=3, Hq=8, Hkv=2, D=128, P=16, bl=12, prefix=(40, 3, 100)):
    rng = np.random.default_rng(seed)
    case = W.make_block_attn_case("commit", B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=list(prefix),
                                  seed=seed)
    shape = (B, bl, Hkv, D)
    k_new = W.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
    v_new = W.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
    return rng, case, k_new, v_new


def gpu_commit(case, k_new, v_new, counts, advance, k_bits=None, v_bits=None, prefix=None, table=None):
    kv = case.kv
    p = nld.make_params(case.batch, case.num_q_heads, case.num_kv_heads, case.head_dim, case.page_size,
                        kv.num_pages, kv.max_pages, 0, 0.0, 0)
    kp = bits_dev(kv.k_bits if k_bits is None else k_bits)
    vp = bits_dev(kv.v_bits if v_bits is None else v_bits)
    pl = torch.from_numpy(np.array(kv.prefix_lens if prefix is None else prefix, np.int32)).cuda()
    cnt = None if counts is None else torch.from_numpy(np.asarray(counts, np.int32)).cuda()
    tab = torch.from_numpy(np.ascontiguousarray(kv.page_table if table is None else table, np.int32)).cuda()
    nld.nld_kv_commit(p, bits_dev(k_new), bits_dev(v_new), cnt, tab, pl,
                      case.block_len, advance, kp, vp)
    return dev_bits(kp), dev_bits(vp), pl.cpu().numpy()


@pytest.mark.parametrize("D,P", [(128, 16), (64, 32), (128, 256)])
def test_kv_commit_matches_oracle(orc, D, P):
    rng, case, k_new, v_new = commit_case(D + P, D=D, P=P)
    kv = case.kv
    for counts, advance in ((None, False), (None, True), (rng.integers(0, case.block_len + 1, case.batch), True),
                            (np.array([0, case.block_len, 5]), False)):
        g = gpu_commit(case, k_new, v_new, counts, advance)
        o = orc.kv_commit(k_new, v_new, counts, kv.page_table, kv.prefix_lens, kv.k_bits, kv.v_bits, advance)
        for x, y, what in zip(g, o, ("k_pages", "v_pages", "prefix_lens")):
            assert np.array_equal(x, y), f"{what} counts={counts} advance={advance}"


def test_kv_commit_staged_block_attention(orc):
    """The block's K/V staged by nld_kv_commit is what nld_block_attn reads:
    bit-identical to attention over pools staged on the host by the oracle,
    and within tolerance of the oracle's attention."""
    _, case, k_new, v_new = commit_case(5)
    kv = case.kv
    kp, vp, _ = gpu_commit(case, k_new, v_new, None, False)
    okp, ovp, _ = orc.kv_commit(k_new, v_new, None, kv.page_table, kv.prefix_lens, kv.k_bits, kv.v_bits, False)
    assert np.array_equal(kp, okp) and np.array_equal(vp, ovp)
    p = nld.make_params(case.batch, case.num_q_heads, case.num_kv_heads, case.head_dim, case.page_size,
                        kv.num_pages, kv.max_pages, 0, 0.0, 0)
    for mode, qb in ((DIFF, case.q_draft_bits), (VER, case.q_verify_bits)):
        out = torch.empty((case.batch, case.block_len, case.num_q_heads, case.head_dim), dtype=torch.bfloat16,
                          device="cuda")
        lse = torch.empty((case.batch, case.num_q_heads, case.block_len), dtype=torch.float32, device="cuda")
        ws = torch.zeros(max(16, nld.nld_block_attn_workspace_size(p, case.block_len)), dtype=torch.uint8,
                         device="cuda")
        nld.nld_block_attn(p, bits_dev(qb), bits_dev(kp), bits_dev(vp), torch.from_numpy(kv.page_table).cuda(),
                           torch.from_numpy(kv.prefix_lens).cuda(), case.block_len, mode, out, lse, ws)
        ro, rl = orc.block_attn(qb, okp, ovp, kv.page_table, kv.prefix_lens, case.num_q_heads, case.num_kv_heads,
                                case.block_len, mode, case.scale)
        compare_attn(out, lse, ro, rl, f"staged block mode={mode}")


def test_kv_commit_verify_chain(orc):
    """Three verify steps: accept on the GPU, commit the accepted rows and
    advance; pools and prefix lengths equal the oracle's chain."""
    rng, case, _, _ = commit_case(6, prefix=(0, 17, 33))
    kv = case.kv
    gk, gv, gl = kv.k_bits.copy(), kv.v_bits.copy(), kv.prefix_lens.copy()
    ok, ov, ol = kv.k_bits.copy(), kv.v_bits.copy(), kv.prefix_lens.copy()
    cap = kv.max_pages * case.page_size
    for _ in range(3):
        shape = (case.batch, case.block_len, case.num_kv_heads, case.head_dim)
        k_new = W.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
        v_new = W.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
        d, v = W.make_accept_ids(rng, case.batch, case.block_len, 131072, 0.7)
        acc = np.minimum(gpu_accept(d, v), cap - gl).astype(np.int32)
        assert np.array_equal(acc, np.minimum(orc.accept(d, v), cap - ol))
        gk, gv, gl = gpu_commit(case, k_new, v_new, acc, True, gk, gv, gl)
        ok, ov, ol = orc.kv_commit(k_new, v_new, acc, kv.page_table, ol, ok, ov, True)
        assert np.array_equal(gk, ok) and np.array_equal(gv, ov) and np.array_equal(gl, ol)


def test_kv_commit_range_flags(orc):
    """Counts past the block, a slot past the page table and a page id outside
    the pool are flagged on the device; those rows are not written."""
    _, case, k_new, v_new = commit_case(7)
    kv = case.kv
    err = nld.nld_device_error(clear=True)
    kp, vp, pl = gpu_commit(case, k_new, v_new, np.array([case.block_len + 3, 0, 0]), False)
    err = nld.nld_device_error(clear=True)
    assert err & nld.NLD_DEVERR_PREFIX_RANGE
    okp, _, _ = orc.kv_commit(k_new, v_new, np.array([case.block_len, 0, 0]), kv.page_table, kv.prefix_lens,
                              kv.k_bits, kv.v_bits, False)
    assert np.array_equal(kp, okp), "an oversized count is clamped to the block"
    far = kv.prefix_lens.copy()
    far[1] = kv.max_pages * case.page_size  # every row of sequence 1 past the table
    kp, _, _ = gpu_commit(case, k_new, v_new, np.array([0, 4, 0]), False, prefix=far)
    assert nld.nld_device_error(clear=True) & nld.NLD_DEVERR_PREFIX_RANGE
    assert np.array_equal(kp, kv.k_bits), "nothing written"
    bad = kv.page_table.copy()
    L2 = int(kv.prefix_lens[2])
    bad[2, L2 // case.page_size] = kv.num_pages + 5  # the page of sequence 2's first block slot
    kp, _, _ = gpu_commit(case, k_new, v_new, np.array([0, 0, 1]), False, table=bad)
    assert nld.nld_device_error(clear=True) & nld.NLD_DEVERR_PAGE_RANGE
    assert np.array_equal(kp, kv.k_bits), "nothing written"


# ---------------------------------------------------------------------------
# logits -> (argmax id, confidence)
# ---------------------------------------------------------------------------

# conf relative tolerance: one ex2.approx per logit (relative error ~2^-21)
# plus fp32 sums of at most 512 positive terms per thread before an fp32
# tree merge (<= 512 * 2^-24 = 3.1e-5 relative).
LOGITS_RTOL = 4e-5


def gpu_logits(bits, vocab=None):
    rows, ld = bits.shape
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()
    ids = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
    conf = torch.full((rows,), -7.0, dtype=torch.float32, device="cuda")
    nld.nld_logits_argmax(t, ids, conf, vocab=vocab)
    return ids.cpu().numpy(), conf.cpu().numpy().astype(np.float64)


def check_logits(got, ref, what):
    (gi, gc), (ri, rc) = got, ref
    assert np.array_equal(gi, ri), f"{what}: argmax differs at {np.flatnonzero(gi != ri)[:5]}"
    nan = np.isnan(rc)
    assert np.array_equal(np.isnan(gc), nan), f"{what}: NaN pattern"
    err = np.abs(gc[~nan] - rc[~nan])
    assert np.all(err <= LOGITS_RTOL * np.abs(rc[~nan])), f"{what}: conf rel err {np.max(err / np.maximum(rc[~nan], 1e-30)):.2e}"


def test_logits_golden_cases():
    for lg, idx, cf in oracle_pins.read_golden("logits_argmax_cases.txt"):
        x = np.array([[float(v) for v in lg.split()]], dtype=np.float32)
        V = x.shape[1]
        bits = np.zeros((1, (V + 7) // 8 * 8), dtype=np.uint16)
        bits[0, :V] = W.f32_to_bf16_bits(x)[0]
        gi, gc = gpu_logits(bits, vocab=V)
        assert int(gi[0]) == int(idx), lg
        want = float(cf)
        assert (math.isnan(gc[0]) and math.isnan(want)) or abs(gc[0] - want) <= LOGITS_RTOL * max(want, 1e-30), lg


@pytest.mark.parametrize("rows,vocab,ld", [(1, 1, 8), (3, 7, 8), (5, 8, 8), (7, 9, 16), (16, 131072, 131072),
                                           (16, 131077, 131080), (2, 50000, 50008), (300, 32000, 32000),
                                           (1024, 4096, 4096), (152, 131072, 131072)])
def test_logits_matches_oracle(orc, rows, vocab, ld):
    rng = np.random.default_rng(rows * 7 + vocab)
    x = (rng.standard_normal((rows, ld)) * 3.0).astype(np.float32)
    x[:, vocab:] = 1e4  # padding past vocab must never be read
    if rows >= 3:
        x[0, :vocab] = -np.inf                                   # nothing above -inf
        x[1, rng.integers(0, vocab)] = np.nan                    # a NaN logit
        x[2, :vocab] = np.round(x[2, :vocab])                    # many ties
    x[rng.random(x.shape) < 0.01] = -np.inf
    bits = W.f32_to_bf16_bits(x)
    check_logits(gpu_logits(bits, vocab), orc.logits_argmax(bits, vocab), f"rows={rows} V={vocab} ld={ld}")


def gpu_ensemble(a_bits, d_bits, lam, vocab=None):
    rows = a_bits.shape[0]
    ta = torch.from_numpy(np.ascontiguousarray(a_bits).view(np.int16)).view(torch.bfloat16).cuda()
    td = torch.from_numpy(np.ascontiguousarray(d_bits).view(np.int16)).view(torch.bfloat16).cuda()
    ids = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
    conf = torch.full((rows,), -7.0, dtype=torch.float32, device="cuda")
    nld.nld_logits_ensemble_argmax(ta, td, lam, ids, conf, vocab=vocab)
    return ids.cpu().numpy(), conf.cpu().numpy().astype(np.float64)


def mixture_f64(a_bits, d_bits, lam, vocab):
    def sm(bits):
        x = W.bf16_bits_to_f32(bits[:, :vocab]).astype(np.float64)
        m = x.max(axis=1, keepdims=True)
        w = np.where(np.isfinite(m), np.exp(x - np.where(np.isfinite(m), m, 0)), 0.0)
        s = w.sum(axis=1, keepdims=True)
        return np.where(s > 0, w / np.where(s > 0, s, 1), 0.0)
    return lam * sm(a_bits) + (1 - lam) * sm(d_bits)


def test_ensemble_golden_cases():
    for ar, df, lam, idx, cf in oracle_pins.read_golden("ensemble_cases.txt"):
        a = W.f32_to_bf16_bits(np.array([[float(v) for v in ar.split()]], np.float32))
        d = W.f32_to_bf16_bits(np.array([[float(v) for v in df.split()]], np.float32))
        V = a.shape[1]
        pa = np.zeros((1, 8), np.uint16); pa[0, :V] = a[0]
        pd = np.zeros((1, 8), np.uint16); pd[0, :V] = d[0]
        gi, gc = gpu_ensemble(pa, pd, float(lam), vocab=V)
        assert int(gi[0]) == int(idx) and abs(gc[0] - float(cf)) <= LOGITS_RTOL * float(cf), f"{ar} | {df} | {lam}"


@pytest.mark.parametrize("rows,vocab,ld,lam", [(16, 131072, 131072, 0.5), (5, 1001, 1008, 0.3), (300, 32000, 32000, 0.7),
                                               (2, 131077, 131080, 1.0), (3, 9, 16, 0.0), (1, 7, 8, 0.25)])
def test_ensemble_matches_oracle(orc, rows, vocab, ld, lam):
    """ids: the oracle's where its two best mixture values are apart by more
    than the fp32 error, else any position whose mixture value is within that
    error of the max; conf within the logits bound."""
    rng = np.random.default_rng(rows + vocab)
    a = W.f32_to_bf16_bits((rng.standard_normal((rows, ld)) * 3).astype(np.float32))
    d = W.f32_to_bf16_bits((rng.standard_normal((rows, ld)) * 3).astype(np.float32))
    if rows >= 3:
        a[1, :vocab] = W.f32_to_bf16_bits(np.full(vocab, -np.inf, np.float32))  # one side empty
    gi, gc = gpu_ensemble(a, d, lam, vocab)
    oi, oc = orc.ensemble_argmax(a, d, lam, vocab)
    p = mixture_f64(a, d, lam, vocab)
    assert np.all(np.abs(gc - oc) <= LOGITS_RTOL * oc)
    tol = 2 * LOGITS_RTOL * oc
    top2 = np.sort(p, axis=1)[:, -2:]
    clear = top2[:, 1] - top2[:, 0] > tol
    assert np.array_equal(gi[clear], oi[clear])
    assert np.all(p[np.arange(rows), gi] >= oc - tol), "the GPU's id is a maximiser within the error"


def test_logits_peaked_rows(orc):
    """Peaked rows (a confident prediction): the confidence near 1 is kept to
    the same relative bound."""
    rng = np.random.default_rng(77)
    x = (rng.standard_normal((64, 131072)) * 1.0).astype(np.float32)
    hot = rng.integers(0, 131072, size=64)
    x[np.arange(64), hot] = np.linspace(2, 30, 64)
    bits = W.f32_to_bf16_bits(x)
    check_logits(gpu_logits(bits), orc.logits_argmax(bits), "peaked")


def test_accept_golden_cases():
    for d, v, acc in oracle_pins.read_golden("accept_cases.txt"):
        d = np.array([[int(x) for x in d.split()]], dtype=np.int32)
        v = np.array([[int(x) for x in v.split()]], dtype=np.int32)
        assert int(gpu_accept(d, v)[0]) == int(acc)


@pytest.mark.parametrize("name", sorted(W.WORKLOADS))
def test_accept_workload_ids(orc, name):
    cfg = W.WORKLOADS[name]
    for seed in range(5):
        rng = np.random.default_rng(seed)
        d, v = W.make_accept_ids(rng, max(cfg["batch"], 1000), cfg["bl"], cfg["vocab"], cfg["p"])
        assert np.array_equal(gpu_accept(d, v), orc.accept(d, v))


def test_accept_all_widths(orc):
    rng = np.random.default_rng(1)
    for n in range(1, 33):
        for p in (0.0, 0.6, 1.0):
            d, v = W.make_accept_ids(rng, 77, n, 1000, p)
            assert np.array_equal(gpu_accept(d, v), orc.accept(d, v)), (n, p)


def test_unmask_golden_cases():
    for c, k, pos, nsel in oracle_pins.read_golden("unmask_cases.txt"):
        conf = np.array([[float(x) for x in c.split()]], dtype=np.float32)
        p, s = gpu_unmask(conf, int(k))
        assert p[0].tolist() == [int(x) for x in pos.split()]
        assert int(s[0]) == int(nsel)


def test_unmask_ties_and_ineligible(orc):
    rng = np.random.default_rng(2)
    for n in (1, 2, 3, 8, 16, 31, 32):
        for k in sorted({k for k in (1, 2, max(1, n // 2), n) if k <= n}):
            conf = rng.integers(0, 3, size=(300, n)).astype(np.float32) / 2
            conf[rng.random((300, n)) < 0.2] = -np.inf
            conf[rng.random((300, n)) < 0.05] = np.nan
            z = rng.random((300, n)) < 0.1
            conf[z] = np.where(rng.random(z.sum()) < 0.5, 0.0, -0.0)
            conf[rng.random((300, n)) < 0.03] = np.inf
            p, s = gpu_unmask(conf, k)
            op, os_ = orc.unmask(conf, k)
            assert np.array_equal(p, op) and np.array_equal(s, os_), (n, k)


def test_unmask_workload_confidences(orc):
    for name, cfg in W.WORKLOADS.items():
        wl = W.make_workload(name, seed=0, batch=min(cfg["batch"], 16),
                             prefix_override=[64] * min(cfg["batch"], 16))
        for conf in wl.conf:
            for k in wl.unmask_k:
                big = np.concatenate([conf, W.make_confidences(np.random.default_rng(5), 500, cfg["bl"], cfg["conf"])])
                assert all(np.array_equal(a, b) for a, b in zip(gpu_unmask(big, k), orc.unmask(big, k)))


def test_unmask_denoising_chain(orc):
    """Four successive top-8 steps on a 32-position block; committed positions
    become -inf (the 14B-shape diffusion steps). Each side chains its own result."""
    rng = np.random.default_rng(14)
    B, n, k = 16, 32, 8
    conf_steps = [W.make_confidences(rng, B, n, "uniform") for _ in range(4)]
    committed_g = np.zeros((B, n), dtype=bool)
    committed_o = np.zeros((B, n), dtype=bool)
    for c in conf_steps:
        cg = np.where(committed_g, -np.inf, c).astype(np.float32)
        co = np.where(committed_o, -np.inf, c).astype(np.float32)
        pg, sg = gpu_unmask(cg, k)
        po, so = orc.unmask(co, k)
        assert np.array_equal(pg, po) and np.array_equal(sg, so)
        for b in range(B):
            committed_g[b, pg[b][pg[b] >= 0]] = True
            committed_o[b, po[b][po[b] >= 0]] = True
    assert committed_g.all(), "4 x top-8 fills the 32-token block"


# ---------------------------------------------------------------------------
# split combine
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("S,D", [(1, 128), (2, 64), (7, 128), (64, 128), (128, 64)])
def test_combine_matches_oracle(orc, S, D):
    rng = np.random.default_rng(S * 1000 + D)
    B, Hq, bl = 3, 8, 5
    # partial rows in bf16 (the workspace format); the oracle merges the same
    # bf16 values in fp64
    o_bits = W.f32_to_bf16_bits(rng.standard_normal((S, B, Hq, bl, D)).astype(np.float32))
    l = (rng.standard_normal((S, B, Hq, bl)) * 3).astype(np.float32)
    l[rng.random(l.shape) < 0.3] = -np.inf
    l[:, 0, 0, 0] = -np.inf  # a row with no keys at all
    o_bits[np.broadcast_to((l == -np.inf)[..., None], o_bits.shape)] = 0x7FC0  # NaN, never read
    o = W.bf16_bits_to_f32(o_bits)
    out = torch.empty((B, bl, Hq, D), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((B, Hq, bl), dtype=torch.float32, device="cuda")
    o_dev = torch.from_numpy(np.ascontiguousarray(o_bits).view(np.int16)).view(torch.bfloat16).cuda()
    nld.nld_split_kv_combine(o_dev, torch.from_numpy(l).cuda(), out, lse)
    ro, rl = orc.combine(np.nan_to_num(o, nan=0.0).reshape(S, -1, D), l.reshape(S, -1))
    ro = ro.reshape(B, Hq, bl, D).transpose(0, 2, 1, 3)
    rl = rl.reshape(B, Hq, bl)
    got = out.float().cpu().numpy()
    assert np.all(np.isfinite(got))
    # bf16 round-to-nearest of the exact value (half an ulp, at most 2^-8 relative)
    # plus fp32 accumulation error
    assert np.all(np.abs(got - ro) <= 2.0 ** -8 * np.abs(ro) + 1e-5)
    gl = lse.cpu().numpy()
    assert np.array_equal(np.isinf(gl), np.isinf(rl))
    fin = np.isfinite(rl)
    assert np.max(np.abs(gl[fin] - rl[fin])) <= 1e-4


# ---------------------------------------------------------------------------
# attention: small cases, every row
# ---------------------------------------------------------------------------

SMALL = [
    # name, B, Hq, Hkv, D, P, bl, prefix lens
    ("tinyshape", 1, 4, 1, 64, 256, 8, [256]),
    ("d128_g4_bl16", 2, 8, 2, 128, 16, 16, [300, 77]),
    ("d64_g2_bl5_ragged", 3, 4, 2, 64, 32, 5, [0, 13, 200]),
    ("d128_g5_bl32", 1, 10, 2, 128, 16, 32, [500]),
    ("d128_mha_bl1", 2, 4, 4, 128, 64, 1, [63, 64]),
    ("d128_g8_bl20_p128", 2, 16, 2, 128, 128, 20, [129, 1000]),
    ("d64_g1_bl32_p16", 1, 2, 2, 64, 16, 32, [31]),
    ("prefix0_bl32", 2, 8, 2, 128, 16, 32, [0, 0]),
    ("d128_g8_bl32_256rows", 2, 16, 2, 128, 16, 32, [700, 33]),
    ("d64_g6_bl30_180rows", 1, 6, 1, 64, 32, 30, [150]),
    # 96 packed rows: one M tile without row copies, several tiles per split
    ("d128_g3_bl32_96rows", 2, 6, 2, 128, 16, 32, [450, 190]),
    ("d64_g4_bl24_96rows", 1, 8, 2, 64, 32, 24, [230]),
    # two M tiles: the rows past 128 copied 2 or 4 times, or not at all
    ("d128_g6_bl30_180rows", 1, 6, 1, 128, 32, 30, [260]),
    ("d64_g5_bl32_160rows", 2, 10, 2, 64, 16, 32, [300, 45]),
    ("d64_g8_bl32_256rows", 1, 16, 2, 64, 16, 32, [100]),
    # two softmax groups over an odd number of tiles longer than the ring
    # (one split: 15 and 17 tiles): the group without the last tile reaches
    # the epilogue early and must wait for every PV product
    ("d128_g3_bl32_96rows_15tiles", 1, 6, 2, 128, 16, 32, [900]),
    ("d128_g4_bl32_128rows_17tiles", 1, 8, 2, 128, 16, 32, [1060]),
    # more than 128 rows with an odd block length: one CTA with two M tiles
    # (an even block length splits the slots over two CTAs instead)
    ("d128_g5_bl29_145rows", 1, 10, 2, 128, 16, 29, [300]),
    ("d64_g8_bl31_248rows", 2, 16, 2, 64, 16, 31, [100, 37]),
]


@pytest.mark.parametrize("spec", SMALL, ids=[s[0] for s in SMALL])
@pytest.mark.parametrize("mode", [DIFF, VER], ids=["diffusion", "verify"])
@pytest.mark.parametrize("splits", [0, 1, 3])
def test_attention_small_all_rows(orc, spec, mode, splits):
    name, B, Hq, Hkv, D, P, bl, prefix = spec
    case = W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix,
                                  seed=sum(prefix) + bl)
    dc = DeviceCase(case)
    out, lse = dc.run(mode, num_splits=splits)
    ro, rl = oracle_full(orc, case, mode)
    compare_attn(out, lse, ro, rl, f"{name} mode={mode} S={splits}")


@pytest.mark.parametrize("mode", [DIFF, VER], ids=["diffusion", "verify"])
@pytest.mark.parametrize("D", [64, 128])
def test_attention_multiwave_longest_first(orc, mode, D):
    """More (sequence, KV head) units than SMs with one split each: the CTAs
    take the sequences longest first (a permutation by prefix length, ties by
    index); every row still lands in its own sequence's output."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    B, Hq, Hkv, bl, P = 48, 16, 4, 8, 16
    assert B * Hkv > sms
    rng = np.random.Generator(np.random.PCG64(2024 + D))
    prefix = [int(x) for x in rng.integers(0, 400, size=B)]
    prefix[5] = prefix[17] = prefix[30] = 257  # ties
    prefix[0] = 0
    case = W.make_block_attn_case("multiwave", B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix,
                                  seed=77 + D)
    dc = DeviceCase(case)
    assert nld.nld_block_attn_num_splits(dc.params(0), bl) == 1
    ro, rl = oracle_full(orc, case, mode)
    for splits in (0, 1):
        out, lse = dc.run(mode, num_splits=splits)
        compare_attn(out, lse, ro, rl, f"multiwave D={D} mode={mode} S={splits}")
    for flags in (0, nld.NLD_ATTN_PREFIX_READY):
        o2, l2 = dc.run(mode, 0, flags=flags)
        compare_attn(o2, l2, ro, rl, f"multiwave D={D} mode={mode} flags={flags}")


# Two softmax groups with a lane quadrant of padding rows (80 rows per
# block-slot chunk, 96 rows) over splits longer than the ring: the warps of
# the empty quadrant do no exponentials, so they are the first to hand each
# score product over. A hand-off that let one of them run two products ahead
# released a PV product before the other warps had written their P (the
# output went wrong while the log-sum-exp stayed right). That interleaving
# showed only under a slower softmax step (an experimental build), never with
# the kernel as it was, so this test cannot prove its absence; it runs the
# shapes that expose it repeatedly, after the other plans have run, both
# passes, and the kernel now keeps every warp within one product of the
# others by construction.
HANDOFF = [
    ("d128_g8_bl20_p128", 2, 16, 2, 128, 128, 20, [129, 1000]),
    ("d128_g3_bl32_96rows", 1, 6, 2, 128, 16, 32, [900]),
    ("d64_g5_bl32_160rows", 1, 10, 2, 64, 16, 32, [1500]),
]


@pytest.mark.parametrize("spec", HANDOFF, ids=[s[0] for s in HANDOFF])
def test_two_group_handoff_repeated(orc, spec):
    name, B, Hq, Hkv, D, P, bl, prefix = spec
    case = W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix,
                                  seed=sum(prefix) + bl + 5)
    dc = DeviceCase(case)
    ref = {mode: oracle_full(orc, case, mode) for mode in (DIFF, VER)}
    for rep in range(6):
        for splits in (0, 1, 3):
            for mode in (DIFF, VER):
                out, lse = dc.run(mode, num_splits=splits)
                ro, rl = ref[mode]
                compare_attn(out, lse, ro, rl, f"{name} mode={mode} S={splits} rep={rep}")


@pytest.mark.parametrize("spec", SMALL, ids=[s[0] for s in SMALL])
def test_prefix_ready_flag_same_result(orc, spec):
    """NLD_ATTN_PREFIX_READY only moves prefix loads before the dependency
    wait: results are bit-identical to the unflagged call and match the oracle."""
    name, B, Hq, Hkv, D, P, bl, prefix = spec
    case = W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix,
                                  seed=sum(prefix) + 2 * bl)
    dc = DeviceCase(case)
    for mode in (DIFF, VER):
        for splits in (0, 1, 3):
            o0, l0 = dc.run(mode, splits)
            o1, l1 = dc.run(mode, splits, flags=nld.NLD_ATTN_PREFIX_READY)
            assert torch.equal(o0, o1) and torch.equal(l0, l1)
            ro, rl = oracle_full(orc, case, mode)
            compare_attn(o1, l1, ro, rl, f"{name} flag mode={mode} S={splits}")


@pytest.mark.parametrize("spec", [SMALL[1], SMALL[3], SMALL[10]], ids=[SMALL[1][0], SMALL[3][0], SMALL[10][0]])
@pytest.mark.parametrize("splits", [3, 19])
def test_partials_entry_point_then_combine(orc, spec, splits):
    """nld_block_attn_partials + nld_split_kv_combine run the same kernels as
    nld_block_attn: bit-identical result, within tolerance of the oracle."""
    name, B, Hq, Hkv, D, P, bl, prefix = spec
    case = W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix,
                                  seed=sum(prefix) + 5 * bl)
    dc = DeviceCase(case)
    p = dc.params(splits)
    if nld.nld_block_attn_num_splits(p, bl) < 2:
        pytest.skip("plan merges on chip: no partials")
    for mode in (DIFF, VER):
        ref_out, ref_lse = dc.run(mode, splits)
        ws = torch.zeros(nld.nld_block_attn_workspace_size(p, bl), dtype=torch.uint8, device="cuda")
        out = torch.full_like(ref_out, float("nan"))
        lse = torch.full_like(ref_lse, float("nan"))
        nld.nld_block_attn_partials(p, dc.q[mode], dc.k, dc.v, dc.table, dc.prefix, bl, mode, out, lse, ws)
        assert torch.isnan(out).all(), "the partials call leaves out untouched"
        o_part, lse_part = nld.workspace_views(p, bl, ws)
        nld.nld_split_kv_combine(o_part, lse_part, out, lse)
        assert torch.equal(out, ref_out) and torch.equal(lse, ref_lse)
        ro, rl = oracle_full(orc, case, mode)
        compare_attn(out, lse, ro, rl, f"{name} partials mode={mode} S={splits}")


# ---------------------------------------------------------------------------
# table-mask attention (quadratic self-speculation)
# ---------------------------------------------------------------------------

def run_masked(dc, table, splits=0, q=None):
    c = dc.case
    p = dc.params(splits)
    q = dc.q[DIFF] if q is None else q
    out = torch.empty((c.batch, c.block_len, c.num_q_heads, c.head_dim), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((c.batch, c.num_q_heads, c.block_len), dtype=torch.float32, device="cuda")
    ws = torch.zeros(max(16, nld.nld_block_attn_workspace_size(p, c.block_len)), dtype=torch.uint8, device="cuda")
    bm = torch.from_numpy(np.asarray(table, dtype=np.uint32).view(np.int32)).cuda()
    nld.nld_block_attn_masked(p, q, dc.k, dc.v, dc.table, dc.prefix, c.block_len, bm, out, lse, ws)
    return out, lse


@pytest.mark.parametrize("spec", [SMALL[1], SMALL[3], SMALL[10], SMALL[8]], ids=[SMALL[i][0] for i in (1, 3, 10, 8)])
def test_masked_tables_reduce_to_modes(spec):
    """An all-ones table runs the draft pass and the lower-triangular table
    the verify pass: bit-identical to nld_block_attn."""
    name, B, Hq, Hkv, D, P, bl, prefix = spec
    case = W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix,
                                  seed=sum(prefix) + 3 * bl)
    dc = DeviceCase(case)
    full = np.full(bl, (1 << bl) - 1, dtype=np.uint64).astype(np.uint32)
    tril = np.array([(2 << i) - 1 for i in range(bl)], dtype=np.uint64).astype(np.uint32)
    for splits in (0, 1, 3):
        for table, mode in ((full, DIFF), (tril, VER)):
            ref_o, ref_l = dc.run(mode, splits)
            got_o, got_l = run_masked(dc, table, splits, q=dc.q[mode])
            assert torch.equal(got_o, ref_o) and torch.equal(got_l, ref_l), f"{name} mode={mode} S={splits}"


@pytest.mark.parametrize("k,G,D,prefix", [(1, 4, 128, [100]), (2, 8, 64, [0, 37]), (3, 4, 128, [300, 5]),
                                          (4, 6, 128, [64]), (5, 4, 128, [1000, 17]), (5, 8, 64, [250])])
def test_quadss_attention_matches_oracle(orc, k, G, D, prefix):
    bl = 1 + k + k * k
    Hkv = 2
    case = W.make_block_attn_case(f"quadss{k}", len(prefix), G * Hkv, Hkv, D, block_len=bl, page_size=16,
                                  prefix_lens=prefix, seed=90 + k + G)
    dc = DeviceCase(case)
    table = nld.nld_quadss_block_mask(k)
    ro, rl, _ = orc.block_attn_masked(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                      case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, bl, table, case.scale)
    for splits in (0, 1, 3):
        out, lse = run_masked(dc, table, splits)
        compare_attn(out, lse, ro, rl, f"quadss k={k} G={G} S={splits}")


def test_masked_random_tables_and_empty_row(orc):
    rng = np.random.default_rng(91)
    for prefix in ([0, 0], [33, 7]):
        case = W.make_block_attn_case("randmask", 2, 8, 2, 128, block_len=20, page_size=16, prefix_lens=prefix,
                                      seed=sum(prefix) + 91)
        dc = DeviceCase(case)
        table = rng.integers(0, 1 << 20, size=20, dtype=np.uint64).astype(np.uint32)
        table[3] = 0  # with no prefix this row sees nothing
        ro, rl, _ = orc.block_attn_masked(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                          case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, 20, table,
                                          case.scale)
        for splits in (0, 2):
            out, lse = run_masked(dc, table, splits)
            o = out.float().cpu().numpy()
            l = lse.cpu().numpy()
            if prefix[0] == 0:
                assert np.all(o[0, 3] == 0) and np.all(l[0, :, 3] == -np.inf)
            fin = np.isfinite(rl)
            assert np.array_equal(np.isfinite(l), fin)
            compare_attn(out, None, ro, rl, f"random table prefix={prefix} S={splits}")
            assert np.max(np.abs(l[fin] - rl[fin])) <= 2e-3


def test_attention_tail_slots_hold_nan(orc):
    """Cache slots past the block inside the last page may be uninitialised;
    NaN there must not reach the output."""
    case = W.make_block_attn_case("nan_tail", 2, 8, 2, 128, block_len=7, page_size=16, prefix_lens=[37, 100], seed=3)
    kv = case.kv
    k_bits, v_bits = kv.k_bits.copy(), kv.v_bits.copy()
    nan = np.uint16(0x7FC0)
    for b, L in enumerate(kv.prefix_lens):
        N = int(L) + case.block_len
        for t in range(N, ((N + 15) // 16) * 16):  # rest of the last page
            page, slot = kv.page_table[b, t // kv.page_size], t % kv.page_size
            k_bits[page, :, slot, :] = nan
            v_bits[page, :, slot, :] = nan
    case2 = W.BlockAttnCase(case.name, case.batch, case.num_q_heads, case.num_kv_heads, case.head_dim,
                            case.block_len, case.scale, case.q_draft_bits, case.q_verify_bits,
                            W.PagedKV(k_bits, v_bits, kv.page_table, kv.prefix_lens, kv.page_size,
                                      kv.num_pages, kv.max_pages))
    dc = DeviceCase(case2)
    for mode in (DIFF, VER):
        for splits in (1, 2):
            out, lse = dc.run(mode, num_splits=splits)
            ro, rl = oracle_full(orc, case2, mode)
            compare_attn(out, lse, ro, rl, f"nan tail mode={mode} S={splits}")


def test_attention_split_sweep(orc):
    case = W.make_block_attn_case("sweep", 1, 8, 2, 128, 16, 16, [1000], seed=9)
    dc = DeviceCase(case)
    ro, rl = oracle_full(orc, case, VER)
    for S in (1, 2, 3, 4, 8, 16, 32, 64, 128):
        out, lse = dc.run(VER, num_splits=S)
        compare_attn(out, lse, ro, rl, f"S={S}")


_CLUSTER_SPECS = [SMALL[0], SMALL[8], SMALL[10], SMALL[13], SMALL[11]]


@pytest.mark.parametrize("spec", _CLUSTER_SPECS, ids=[s[0] for s in _CLUSTER_SPECS])
def test_attention_cluster_merges(orc, spec):
    """Explicit split counts of 2/4/8 (one thread-block cluster merging
    through distributed shared memory) and 16 (clusters of 8, two partials):
    row copies, one and two M tiles, D = 64 and 128, both passes."""
    name, B, Hq, Hkv, D, P, bl, prefix = spec
    case = W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix,
                                  seed=sum(prefix) + 11 * bl)
    dc = DeviceCase(case)
    for mode in (DIFF, VER):
        ro, rl = oracle_full(orc, case, mode)
        for S in (2, 4, 8, 16):
            out, lse = dc.run(mode, num_splits=S)
            compare_attn(out, lse, ro, rl, f"{name} cluster mode={mode} S={S}")


# ---------------------------------------------------------------------------
# attention: self-consistency on the GPU
# ---------------------------------------------------------------------------

def test_page_permutation_is_bit_identical():
    case = W.make_block_attn_case("perm", 2, 8, 2, 128, 16, 16, [333, 90], seed=4)
    kv = case.kv
    perm = np.random.default_rng(1).permutation(kv.num_pages)
    k2, v2 = np.empty_like(kv.k_bits), np.empty_like(kv.v_bits)
    k2[perm], v2[perm] = kv.k_bits, kv.v_bits
    t2 = np.where(kv.page_table >= 0, perm[np.maximum(kv.page_table, 0)], -1).astype(np.int32)
    case2 = W.BlockAttnCase(case.name, case.batch, case.num_q_heads, case.num_kv_heads, case.head_dim,
                            case.block_len, case.scale, case.q_draft_bits, case.q_verify_bits,
                            W.PagedKV(k2, v2, t2, kv.prefix_lens, kv.page_size, kv.num_pages, kv.max_pages))
    a, b = DeviceCase(case), DeviceCase(case2)
    for mode in (DIFF, VER):
        for S in (1, 4):
            oa, la = a.run(mode, S)
            ob, lb = b.run(mode, S)
            assert torch.equal(oa, ob) and torch.equal(la, lb)


def test_block_len_one_modes_agree():
    case = W.make_block_attn_case("bl1", 3, 32, 8, 128, block_len=1, page_size=16, prefix_lens=[5, 700, 4096], seed=5)
    dc = DeviceCase(case)
    q = dc.q[DIFF]
    for S in (1, 0):
        od, ld = dc.run(DIFF, S, q=q)
        ov, lv = dc.run(VER, S, q=q)
        assert torch.equal(od, ov) and torch.equal(ld, lv)


def test_device_clamps_bad_prefix_and_page_ids():
    """Out-of-range device values are clamped (no access leaves the buffers)
    and flagged in the device error word."""
    case = W.make_block_attn_case("bad", 2, 8, 2, 64, block_len=8, page_size=16, prefix_lens=[40, 10], seed=6)
    dc = DeviceCase(case)
    nld.nld_device_error(clear=True)
    dc.prefix = torch.tensor([10 ** 6, -5], dtype=torch.int32, device="cuda")
    dc.run(VER, 2)
    torch.cuda.synchronize()
    assert nld.nld_device_error(clear=True) & nld.NLD_DEVERR_PREFIX_RANGE
    dc = DeviceCase(case)
    dc.table[0, 0] = 10 ** 6
    dc.table[1, 0] = -3
    dc.run(DIFF, 1)
    torch.cuda.synchronize()
    assert nld.nld_device_error(clear=True) & nld.NLD_DEVERR_PAGE_RANGE


def test_wait_timeout_is_reported_and_context_survives(orc):
    """Failure detection without a fault: a bounded wait that nothing
    completes gives up, sets NLD_DEVERR_WAIT_TIMEOUT and returns; the next
    attention call on the same context is correct and raises no error."""
    nld.nld_device_error(clear=True)
    nld.nld_check_wait_timeout(2_000_000)  # 2 ms
    torch.cuda.synchronize()
    assert nld.nld_device_error(clear=True) & nld.NLD_DEVERR_WAIT_TIMEOUT
    name, B, Hq, Hkv, D, P, bl, prefix = SMALL[1]
    case = W.make_block_attn_case(name, B, Hq, Hkv, D, block_len=bl, page_size=P, prefix_lens=prefix, seed=5)
    dc = DeviceCase(case)
    out, lse = dc.run(VER)
    torch.cuda.synchronize()
    assert nld.nld_device_error(clear=True) == 0
    ro, rl = oracle_full(orc, case, VER)
    compare_attn(out, lse, ro, rl, "after a wait timeout")


def test_workspace_too_small_launches_nothing():
    case = W.make_block_attn_case("ws", 1, 8, 2, 128, 16, 16, [500], seed=7)
    dc = DeviceCase(case)
    p = dc.params(3)  # 3 pieces: no cluster, three partials in the workspace
    need = nld.nld_block_attn_workspace_size(p, 16)
    out = torch.zeros((1, 16, 8, 128), dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(need - 16, dtype=torch.uint8, device="cuda")
    with pytest.raises(nld.NldError) as e:
        nld.nld_block_attn(p, dc.q[VER], dc.k, dc.v, dc.table, dc.prefix, 16, VER, out, None, ws)
    assert e.value.status == 3
    torch.cuda.synchronize()
    assert torch.count_nonzero(out) == 0


# ---------------------------------------------------------------------------
# attention: the named workloads at full size
# ---------------------------------------------------------------------------

# every row of both passes where the oracle takes seconds; elsewhere four
# rows of every (sequence, KV head), so every CTA group's output is checked
FULL_ALL_ROWS = ["tiny_b1_h4x1_d64_L256_bl8", "8b_b1_h32x8_d128_L4096_bl16", "long_b1_h32x8_d128_L32768_bl32"]
FULL = FULL_ALL_ROWS + ["14b_b16_h40x8_d128_L8k-16k_bl32", "conc_b8_h32x8_d128_L512-8192_bl8",
                        "conc_b32_h32x8_d128_L512-8192_bl8", "conc_b64_h32x8_d128_L512-8192_bl8",
                        "conc_b128_h32x8_d128_L512-8192_bl8"]


@pytest.mark.parametrize("name", FULL)
def test_full_size_workload(orc, name):
    wl = W.make_workload(name, seed=0)
    case = wl.attn
    dc = DeviceCase(case)
    for mode in (DIFF, VER):
        if mode == DIFF and "diffusion" not in wl.steps:
            continue
        # automatic split count and the prefix-ready flag, as the bench runs it
        out, lse = dc.run(mode, flags=nld.NLD_ATTN_PREFIX_READY)
        if name in FULL_ALL_ROWS:
            ro, rl = oracle_full(orc, case, mode)
            compare_attn(out, lse, ro, rl, f"{name} mode={mode} all rows")
            continue
        rows = rows_per_unit(case, 4, seed=mode + 1)
        qb = dc.q_bits(mode)
        ro, rl = orc.block_attn_rows(qb, case.kv.k_bits, case.kv.v_bits, case.kv.page_table, case.kv.prefix_lens,
                                     case.num_q_heads, case.num_kv_heads, case.block_len, mode, case.scale, rows)
        o = out[rows[:, 0], rows[:, 1], rows[:, 2]]
        l = lse[rows[:, 0], rows[:, 2], rows[:, 1]]
        compare_attn(o, l, ro, rl, f"{name} mode={mode}")
        assert torch.isfinite(out.float()).all()


def test_long_context_split_sweep_sampled(orc):
    wl = W.make_workload("long_b1_h32x8_d128_L32768_bl32", seed=1)
    case = wl.attn
    dc = DeviceCase(case)
    rows = sample_rows(case, 24, seed=3)
    ro, rl = orc.block_attn_rows(case.q_verify_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                 case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, case.block_len, VER,
                                 case.scale, rows)
    for S in (1, 2, 4, 8, 16, 32, 64):
        out, lse = dc.run(VER, S)
        compare_attn(out[rows[:, 0], rows[:, 1], rows[:, 2]], lse[rows[:, 0], rows[:, 2], rows[:, 1]], ro, rl,
                     f"long S={S}")
