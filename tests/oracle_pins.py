"""Pins for the fp64 oracle: checks against things other than the oracle itself.

Each ``pin_*`` takes an oracle handle and raises AssertionError on a mismatch.
They are run on the real oracle (tests/test_oracle_pins.py) and on copies of
the oracle with a planted mistake (tests/test_oracle_mutations.py), which
must each fail at least one pin.

What pins what:
  - torch's scaled_dot_product_attention (fp64, CPU): bl = 1 decode, the
    diffusion pass as full attention over prefix + block, the verify pass as
    the last rows of causal attention, GQA as MHA with repeated KV heads.
  - scipy.special.logsumexp: the lse output.
  - Hand-derived golden values (tests/golden/attn_uniform_q0.txt).
  - Closed forms: constant V, identical keys, one visible key.
  - Invariants: softmax rows sum to 1, page permutation, block permutation.
  - Split / combine against the unsplit result.
  - Brute force and hand-written cases for accept and unmask.
"""
from __future__ import annotations

import math
import os

import numpy as np
import scipy.special
import torch

from paper_2607_05722_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
DIFF, VER = W.MODE_DIFFUSION, W.MODE_VERIFY


# --------------------------------------------------------------------------
# helpers (independent of the oracle)
# --------------------------------------------------------------------------

def small_case(seed, B=2, Hq=4, Hkv=2, D=16, P=4, bl=5, prefix=(7, 12), shuffle=True):
    return W.make_block_attn_case("pin", B, Hq, Hkv, D, bl, P, list(prefix), seed, shuffle_pages=shuffle)


def gather_contiguous(case, b):
    """K, V of sequence b as fp64 [Hkv, L+bl, D], read through the page table
    with numpy indexing."""
    kv = case.kv
    N = int(kv.prefix_lens[b]) + case.block_len
    t = np.arange(N)
    pages = kv.page_table[b, t // kv.page_size]
    slots = t % kv.page_size
    k = W.bf16_bits_to_f32(kv.k_bits[pages, :, slots, :]).astype(np.float64)  # [N, Hkv, D]
    v = W.bf16_bits_to_f32(kv.v_bits[pages, :, slots, :]).astype(np.float64)
    return np.transpose(k, (1, 0, 2)), np.transpose(v, (1, 0, 2))


def q_f64(bits):
    return W.bf16_bits_to_f32(bits).astype(np.float64)


def sdpa(q, k, v, scale, causal=False):
    """torch SDPA in fp64 on CPU. q [H, M, D], k/v [H, N, D]."""
    out = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q)[None], torch.from_numpy(k)[None], torch.from_numpy(v)[None],
        is_causal=causal, scale=scale)
    return out[0].numpy()


def repeat_heads(x, G):
    return np.repeat(x, G, axis=0)


def assert_close(a, b, tol, what):
    err = float(np.max(np.abs(np.asarray(a) - np.asarray(b)))) if np.size(a) else 0.0
    assert err <= tol, f"{what}: max abs err {err:.3e} > {tol:.1e}"


# --------------------------------------------------------------------------
# attention pins
# --------------------------------------------------------------------------

def pin_decode_bl1(orc):
    """bl = 1: both modes are single-token decode attention over L + 1 keys."""
    case = small_case(11, bl=1, prefix=(6, 13))
    G = case.num_q_heads // case.num_kv_heads
    for mode in (DIFF, VER):
        out, lse = orc.block_attn(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                  case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, 1, mode, case.scale)
        for b in range(case.batch):
            k, v = gather_contiguous(case, b)
            q = np.transpose(q_f64(case.q_draft_bits[b]), (1, 0, 2))  # [Hq, 1, D]
            ref = sdpa(q, repeat_heads(k, G), repeat_heads(v, G), case.scale)
            assert_close(np.transpose(out[b], (1, 0, 2)), ref, 1e-12, f"decode mode={mode}")


def pin_diffusion_full_attention(orc):
    """Diffusion pass = unmasked attention over prefix + block (L = 0 included)."""
    for prefix, seed in (((0, 0), 3), ((9, 0), 4), ((7, 12), 5)):
        case = small_case(seed, prefix=prefix)
        G = case.num_q_heads // case.num_kv_heads
        out, _ = orc.block_attn(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, case.block_len,
                                DIFF, case.scale)
        for b in range(case.batch):
            k, v = gather_contiguous(case, b)
            q = np.transpose(q_f64(case.q_draft_bits[b]), (1, 0, 2))
            ref = sdpa(q, repeat_heads(k, G), repeat_heads(v, G), case.scale)
            assert_close(np.transpose(out[b], (1, 0, 2)), ref, 1e-12, f"diffusion prefix={prefix}")


def pin_verify_causal_tail(orc):
    """Verify pass = the last bl rows of causal attention over the L + bl sequence."""
    rng = np.random.default_rng(77)
    for prefix, seed in (((0, 3), 6), ((7, 12), 8)):
        case = small_case(seed, prefix=prefix)
        G = case.num_q_heads // case.num_kv_heads
        out, _ = orc.block_attn(case.q_verify_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, case.block_len,
                                VER, case.scale)
        for b in range(case.batch):
            L = int(case.kv.prefix_lens[b])
            k, v = gather_contiguous(case, b)
            qb = np.transpose(q_f64(case.q_verify_bits[b]), (1, 0, 2))  # [Hq, bl, D]
            qpre = rng.standard_normal((case.num_q_heads, L, case.head_dim))
            qfull = np.concatenate([qpre, qb], axis=1)
            ref = sdpa(qfull, repeat_heads(k, G), repeat_heads(v, G), case.scale, causal=True)[:, L:, :]
            assert_close(np.transpose(out[b], (1, 0, 2)), ref, 1e-12, f"verify prefix={prefix}")


def pin_lse_logsumexp(orc):
    """lse = logsumexp of the scaled scores over the visible keys."""
    case = small_case(21, prefix=(5, 10))
    G = case.num_q_heads // case.num_kv_heads
    for mode, qbits in ((DIFF, case.q_draft_bits), (VER, case.q_verify_bits)):
        _, lse = orc.block_attn(qbits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, case.block_len,
                                mode, case.scale)
        for b in range(case.batch):
            L = int(case.kv.prefix_lens[b])
            k, _ = gather_contiguous(case, b)
            q = q_f64(qbits[b])  # [bl, Hq, D]
            for h in range(case.num_q_heads):
                scores = q[:, h, :] @ k[h // G].T * case.scale  # [bl, N]
                for i in range(case.block_len):
                    n_vis = L + (case.block_len if mode == DIFF else i + 1)
                    ref = scipy.special.logsumexp(scores[i, :n_vis])
                    assert abs(lse[b, h, i] - ref) <= 1e-12, f"lse b={b} h={h} i={i} mode={mode}"


def pin_softmax_rows(orc):
    """Probabilities are >= 0, sum to 1 per row, and are 0 on masked keys."""
    case = small_case(31, prefix=(4, 9))
    for mode in (DIFF, VER):
        _, _, p = orc.block_attn(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                 case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, case.block_len,
                                 mode, case.scale, want_probs=True)
        assert np.all(p >= 0.0)
        assert_close(p.sum(axis=-1), 1.0, 1e-12, "row sums")
        for b in range(case.batch):
            L = int(case.kv.prefix_lens[b])
            for i in range(case.block_len):
                n_vis = L + (case.block_len if mode == DIFF else i + 1)
                assert np.all(p[b, :, i, n_vis:] == 0.0), "probability on a masked key"
                assert np.all(p[b, :, i, :n_vis] > 0.0), "visible key with zero probability"


def pin_page_permutation(orc):
    """Relabelling physical pages (and moving their contents) changes nothing, bit for bit."""
    case = small_case(41, prefix=(10, 3))
    kv = case.kv
    rng = np.random.default_rng(5)
    perm = rng.permutation(kv.num_pages)  # new physical index of old page p is perm[p]
    k2 = np.empty_like(kv.k_bits)
    v2 = np.empty_like(kv.v_bits)
    k2[perm] = kv.k_bits
    v2[perm] = kv.v_bits
    table2 = np.where(kv.page_table >= 0, perm[np.maximum(kv.page_table, 0)], -1).astype(np.int32)
    for mode in (DIFF, VER):
        a = orc.block_attn(case.q_draft_bits, kv.k_bits, kv.v_bits, kv.page_table, kv.prefix_lens,
                           case.num_q_heads, case.num_kv_heads, case.block_len, mode, case.scale)
        b = orc.block_attn(case.q_draft_bits, k2, v2, table2, kv.prefix_lens,
                           case.num_q_heads, case.num_kv_heads, case.block_len, mode, case.scale)
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def pin_block_permutation(orc):
    """Diffusion pass: permuting block tokens (queries and their K/V slots
    together) permutes the output rows."""
    case = small_case(51, B=1, prefix=(6,), P=4, bl=5, shuffle=False)
    kv = case.kv
    L = int(kv.prefix_lens[0])
    bl = case.block_len
    perm = np.random.default_rng(9).permutation(bl)
    q2 = case.q_draft_bits.copy()
    q2[0] = case.q_draft_bits[0][perm]
    k2, v2 = kv.k_bits.copy(), kv.v_bits.copy()
    P = kv.page_size
    for j in range(bl):  # slot L + j gets the content of old slot L + perm[j]
        dst, src = L + j, L + perm[j]
        dp, ds = kv.page_table[0, dst // P], dst % P
        sp, ss = kv.page_table[0, src // P], src % P
        k2[dp, :, ds, :] = kv.k_bits[sp, :, ss, :]
        v2[dp, :, ds, :] = kv.v_bits[sp, :, ss, :]
    a, la = orc.block_attn(case.q_draft_bits, kv.k_bits, kv.v_bits, kv.page_table, kv.prefix_lens,
                           case.num_q_heads, case.num_kv_heads, bl, DIFF, case.scale)
    b, lb = orc.block_attn(q2, k2, v2, kv.page_table, kv.prefix_lens,
                           case.num_q_heads, case.num_kv_heads, bl, DIFF, case.scale)
    assert_close(b[0], a[0][perm], 1e-12, "block permutation (out)")
    assert_close(lb[0], la[0][:, perm], 1e-12, "block permutation (lse)")


def pin_closed_forms(orc):
    """Constant V gives o = V; identical keys give the mean of the visible V;
    a single visible key (L = 0, bl = 1) gives that key's V and lse = score."""
    case = small_case(61, prefix=(5, 11))
    kv = case.kv
    G = case.num_q_heads // case.num_kv_heads
    c_bits = W.f32_to_bf16_bits(np.full(kv.v_bits.shape, 0.75, dtype=np.float32))
    for mode in (DIFF, VER):
        out, _ = orc.block_attn(case.q_draft_bits, kv.k_bits, c_bits, kv.page_table, kv.prefix_lens,
                                case.num_q_heads, case.num_kv_heads, case.block_len, mode, case.scale)
        assert_close(out, 0.75, 1e-14, "constant V")
    same_k = np.broadcast_to(kv.k_bits[:1, :, :1, :], kv.k_bits.shape).copy()
    for mode in (DIFF, VER):
        out, lse = orc.block_attn(case.q_draft_bits, same_k, kv.v_bits, kv.page_table, kv.prefix_lens,
                                  case.num_q_heads, case.num_kv_heads, case.block_len, mode, case.scale)
        for b in range(case.batch):
            L = int(kv.prefix_lens[b])
            _, v = gather_contiguous(case, b)
            k0 = W.bf16_bits_to_f32(kv.k_bits[0, :, 0, :]).astype(np.float64)  # [Hkv, D]
            q = q_f64(case.q_draft_bits[b])
            for i in range(case.block_len):
                n_vis = L + (case.block_len if mode == DIFF else i + 1)
                for h in range(case.num_q_heads):
                    ref = v[h // G, :n_vis].mean(axis=0)
                    assert_close(out[b, i, h], ref, 1e-12, "identical keys")
                    s = float(q[i, h] @ k0[h // G]) * case.scale
                    assert abs(lse[b, h, i] - (s + math.log(n_vis))) <= 1e-12, "identical keys lse"
    one = small_case(62, B=1, prefix=(0,), bl=1)
    out, lse = orc.block_attn(one.q_draft_bits, one.kv.k_bits, one.kv.v_bits, one.kv.page_table,
                              one.kv.prefix_lens, one.num_q_heads, one.num_kv_heads, 1, VER, one.scale)
    k, v = gather_contiguous(one, 0)
    q = q_f64(one.q_draft_bits[0, 0])
    G1 = one.num_q_heads // one.num_kv_heads
    for h in range(one.num_q_heads):
        assert_close(out[0, 0, h], v[h // G1, 0], 0.0, "single key")
        assert abs(lse[0, h, 0] - float(q[h] @ k[h // G1, 0]) * one.scale) <= 1e-12


def read_golden_uniform():
    rows = []
    with open(os.path.join(GOLDEN, "attn_uniform_q0.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            mode, i, o, cnt = [x.strip() for x in line.split("|")]
            rows.append((DIFF if mode == "diffusion" else VER, int(i),
                         np.array([float(x) for x in o.split()]), int(cnt)))
    return rows


def golden_uniform_inputs():
    B, Hq, Hkv, D, P, L, bl = 1, 2, 1, 4, 4, 6, 3
    table = np.array([[2, 0, 1]], dtype=np.int32)
    v = np.full((3, Hkv, P, D), 1000.0, dtype=np.float32)
    for t in range(L + bl):
        page, slot = table[0, t // P], t % P
        v[page, 0, slot] = [t, 2 * t, -t, 1]
    k = np.random.default_rng(0).standard_normal((3, Hkv, P, D)).astype(np.float32)
    q = np.zeros((B, bl, Hq, D), dtype=np.float32)
    return (W.f32_to_bf16_bits(q), W.f32_to_bf16_bits(k), W.f32_to_bf16_bits(v), table,
            np.array([L], dtype=np.int32), Hq, Hkv, bl)


def pin_golden_uniform(orc):
    """Hand-derived outputs for all-zero queries (tests/golden/attn_uniform_q0.txt)."""
    q, k, v, table, pl, Hq, Hkv, bl = golden_uniform_inputs()
    res = {m: orc.block_attn(q, k, v, table, pl, Hq, Hkv, bl, m, 0.5) for m in (DIFF, VER)}
    for mode, i, o_ref, cnt in read_golden_uniform():
        out, lse = res[mode]
        for h in range(Hq):
            assert_close(out[0, i, h], o_ref, 1e-12, f"golden mode={mode} i={i}")
            assert abs(lse[0, h, i] - math.log(cnt)) <= 1e-12


def pin_split_combine(orc):
    """Attention over S disjoint key ranges, merged by the combine rule, equals
    the unsplit result; empty ranges (lse = -inf) are ignored."""
    case = small_case(71, prefix=(9, 14), bl=6)
    kv = case.kv
    Nmax = int(np.max(kv.prefix_lens)) + case.block_len
    for mode in (DIFF, VER):
        full, lse_full = orc.block_attn(case.q_verify_bits, kv.k_bits, kv.v_bits, kv.page_table,
                                        kv.prefix_lens, case.num_q_heads, case.num_kv_heads,
                                        case.block_len, mode, case.scale)
        for cuts in ([0, 4, 11, Nmax], [0, 1, 2, 3, 15, 16, Nmax + 8], [0, Nmax]):
            parts_o, parts_l = [], []
            for a, b in zip(cuts[:-1], cuts[1:]):
                o, l = orc.block_attn(case.q_verify_bits, kv.k_bits, kv.v_bits, kv.page_table,
                                      kv.prefix_lens, case.num_q_heads, case.num_kv_heads,
                                      case.block_len, mode, case.scale, key_begin=a, key_end=b)
                parts_o.append(o.reshape(-1, case.head_dim))
                # lse is [B, Hq, bl]; reorder to the out row order [B, bl, Hq]
                parts_l.append(np.transpose(l, (0, 2, 1)).reshape(-1))
            out, lse = orc.combine(np.stack(parts_o), np.stack(parts_l))
            assert_close(out, full.reshape(-1, case.head_dim), 1e-12, f"split {cuts}")
            assert_close(lse, np.transpose(lse_full, (0, 2, 1)).reshape(-1), 1e-12, "split lse")


def _sdpa_row(case, qbits, mode, b, i, h):
    """One output row (b, i, h) and its lse, from torch SDPA in fp64 over the
    keys the row sees (Sec. 2.2: the whole prefix, then every block slot in
    the draft pass or block slots 0..i in the verify pass)."""
    G = case.num_q_heads // case.num_kv_heads
    L = int(case.kv.prefix_lens[b])
    k, v = gather_contiguous(case, b)
    n_vis = L + (case.block_len if mode == DIFF else i + 1)
    q = q_f64(qbits[b, i, h])[None, None, :]  # [1, 1, D]
    kk, vv = k[h // G, :n_vis][None], v[h // G, :n_vis][None]
    o = sdpa(q, kk, vv, case.scale)[0, 0]
    lse = scipy.special.logsumexp(q[0, 0] @ kk[0].T * case.scale)
    return o, lse


def pin_block_attn_rows(orc):
    """The selected-rows entry (the oracle of every full-size GPU parity run):
    rows listed as (b, i, h) triples, in any order and with repeats, each
    equal to torch SDPA over the keys that row sees, bit-identical to the
    same row of the all-rows entry, and written at its own list position."""
    rng = np.random.default_rng(91)
    # ragged batch, G = 3 (query head h reads KV head h // 3), bl = Hq so that
    # a swapped (i, h) stays in range and is caught by value, not by bounds
    case = W.make_block_attn_case("rows", 3, 6, 2, 16, 6, 4, [0, 9, 14], 92, shuffle_pages=True)
    B, bl, Hq = case.batch, case.block_len, case.num_q_heads
    trip = np.array([(b, i, h) for b in range(B) for i in range(bl) for h in range(Hq)], np.int32)
    sel = np.concatenate([trip[rng.permutation(len(trip))[:40]], trip[[5, 5, len(trip) - 1]]])
    kv = case.kv
    for mode, qbits in ((DIFF, case.q_draft_bits), (VER, case.q_verify_bits)):
        full, lse_full = orc.block_attn(qbits, kv.k_bits, kv.v_bits, kv.page_table, kv.prefix_lens, Hq,
                                        case.num_kv_heads, bl, mode, case.scale)
        out, lse = orc.block_attn_rows(qbits, kv.k_bits, kv.v_bits, kv.page_table, kv.prefix_lens, Hq,
                                       case.num_kv_heads, bl, mode, case.scale, sel)
        assert out.shape == (len(sel), case.head_dim) and lse.shape == (len(sel),)
        for r, (b, i, h) in enumerate(sel):
            o_ref, l_ref = _sdpa_row(case, qbits, mode, b, i, h)
            assert_close(out[r], o_ref, 1e-12, f"rows mode={mode} r={r} (b,i,h)=({b},{i},{h})")
            assert abs(lse[r] - l_ref) <= 1e-12, f"rows lse mode={mode} r={r}"
            assert np.array_equal(out[r], full[b, i, h]), f"rows vs all rows mode={mode} r={r}"
            assert lse[r] == lse_full[b, h, i], f"rows lse vs all rows mode={mode} r={r}"


# --------------------------------------------------------------------------
# decision pins
# --------------------------------------------------------------------------

def read_golden(name):
    cases = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                cases.append([x.strip() for x in line.split("|")])
    return cases


def pin_accept_golden(orc):
    for d, v, acc in read_golden("accept_cases.txt"):
        d = np.array([[int(x) for x in d.split()]], dtype=np.int32)
        v = np.array([[int(x) for x in v.split()]], dtype=np.int32)
        got = orc.accept(d, v)
        assert int(got[0]) == int(acc), f"accept {d} {v}: {got[0]} != {acc}"


def brute_accept(d, v):
    out = []
    for row_d, row_v in zip(d.tolist(), v.tolist()):
        acc = len(row_d)
        for j, (a, b) in enumerate(zip(row_d, row_v)):
            if a != b:
                acc = j
                break
        out.append(acc)
    return np.array(out, dtype=np.int32)


def pin_accept_brute(orc):
    rng = np.random.default_rng(3)
    for n in (1, 2, 7, 8, 16, 31, 32):
        for p in (0.0, 0.5, 0.9, 1.0):
            d, v = W.make_accept_ids(rng, 64, n, 50, p)
            assert np.array_equal(orc.accept(d, v), brute_accept(d, v)), f"n={n} p={p}"


def pin_accept_statistics(orc):
    """E[accepted_len] = p (1 - p^n) / (1 - p) for independent agreement with prob p."""
    rng = np.random.default_rng(2024)
    for n, p in ((8, 0.8), (16, 0.75), (8, 0.7), (32, 0.75)):
        B = 40000
        d, v = W.make_accept_ids(rng, B, n, 131072, p)
        acc = orc.accept(d, v).astype(np.float64)
        mean_ref = p * (1 - p ** n) / (1 - p)
        se = acc.std() / math.sqrt(B)
        assert abs(acc.mean() - mean_ref) < 5 * se, f"n={n} p={p}: {acc.mean()} vs {mean_ref}"


def pin_unmask_golden(orc):
    for c, k, pos, nsel in read_golden("unmask_cases.txt"):
        conf = np.array([[float(x) for x in c.split()]], dtype=np.float32)
        k = int(k)
        p, s = orc.unmask(conf, k)
        assert p[0].tolist() == [int(x) for x in pos.split()], f"unmask {c} k={k}: {p[0]}"
        assert int(s[0]) == int(nsel)


def brute_unmask(conf, k):
    B, n = conf.shape
    pos = np.full((B, k), -1, dtype=np.int32)
    nsel = np.zeros(B, dtype=np.int32)
    for b in range(B):
        c = [float(x) for x in conf[b]]
        elig = [i for i in range(n) if not (math.isnan(c[i]) or c[i] == -math.inf)]
        order = sorted(elig, key=lambda i: (-c[i], i))[:k]
        pos[b, :len(order)] = order
        nsel[b] = len(order)
    return pos, nsel


def pin_unmask_brute(orc):
    rng = np.random.default_rng(8)
    for n in (1, 2, 8, 16, 32):
        for k in sorted({1, 2, min(4, n), min(8, n), n}):
            # few distinct values -> many ties; sprinkle -inf / nan / signed zeros
            conf = rng.integers(0, 4, size=(50, n)).astype(np.float32) / 4
            conf[rng.random((50, n)) < 0.15] = -np.inf
            conf[rng.random((50, n)) < 0.05] = np.nan
            z = rng.random((50, n)) < 0.1
            conf[z] = np.where(rng.random(z.sum()) < 0.5, 0.0, -0.0)
            p, s = orc.unmask(conf, k)
            bp, bs = brute_unmask(conf, k)
            assert np.array_equal(p, bp) and np.array_equal(s, bs), f"n={n} k={k}"


def pin_unmask_lexsort(orc):
    """Against numpy's lexsort (key: confidence descending, then index)."""
    rng = np.random.default_rng(12)
    conf = rng.random((200, 32), dtype=np.float32)
    for k in (1, 4, 8, 32):
        p, s = orc.unmask(conf, k)
        for b in range(conf.shape[0]):
            order = np.lexsort((np.arange(32), -conf[b].astype(np.float64)))[:k]
            assert p[b].tolist() == order.tolist()
        assert np.all(s == k)
    p, _ = orc.unmask(conf, 32)
    assert all(sorted(row) == list(range(32)) for row in p.tolist()), "k = n is a permutation"


def _nums(text, dtype):
    return np.array([[float(x) for x in text.split()]], dtype=dtype)


def pin_threshold_golden(orc):
    for c, thr, pos, nsel in read_golden("unmask_threshold_cases.txt"):
        p, s = orc.unmask_threshold(_nums(c, np.float32), np.float32(float(thr)))
        assert p[0].tolist() == [int(x) for x in pos.split()], f"threshold {c} | {thr}: {p[0]}"
        assert int(s[0]) == int(nsel)


def brute_threshold(conf, thr):
    B, n = conf.shape
    pos = np.full((B, n), -1, dtype=np.int32)
    nsel = np.zeros(B, dtype=np.int32)
    for b in range(B):
        c = [float(x) for x in conf[b]]
        elig = [i for i in range(n) if not (math.isnan(c[i]) or c[i] == -math.inf)]
        chosen = [i for i in elig if c[i] > float(thr)]
        if not chosen and elig:
            chosen = [sorted(elig, key=lambda i: (-c[i], i))[0]]
        pos[b, :len(chosen)] = chosen
        nsel[b] = len(chosen)
    return pos, nsel


def _tied_confidences(rng, B, n):
    conf = rng.integers(0, 5, size=(B, n)).astype(np.float32) / 4
    conf[rng.random((B, n)) < 0.2] = -np.inf
    conf[rng.random((B, n)) < 0.05] = np.nan
    return conf


def pin_threshold_brute(orc):
    rng = np.random.default_rng(21)
    for n in (1, 2, 8, 16, 32):
        conf = _tied_confidences(rng, 60, n)
        for thr in (-1.0, 0.0, 0.25, 0.5, 0.75, 1.0, 2.0):
            p, s = orc.unmask_threshold(conf, thr)
            bp, bs = brute_threshold(conf, thr)
            assert np.array_equal(p, bp) and np.array_equal(s, bs), f"n={n} thr={thr}"


def pin_threshold_limits(orc):
    """A threshold of -inf commits every masked position (numpy's flatnonzero);
    +inf always falls back to the single top-1 position of the pinned top-k rule."""
    rng = np.random.default_rng(22)
    conf = _tied_confidences(rng, 100, 32)
    p, s = orc.unmask_threshold(conf, -np.inf)
    for b in range(conf.shape[0]):
        idx = np.flatnonzero(~np.isnan(conf[b]) & (conf[b] != -np.inf))
        assert p[b][:s[b]].tolist() == idx.tolist() and np.all(p[b][s[b]:] == -1)
    p, s = orc.unmask_threshold(conf, np.inf)
    top, ts = orc.unmask(conf, 1)
    assert np.array_equal(s, ts) and np.array_equal(p[:, 0], top[:, 0])
    assert np.all(p[:, 1:] == -1)


def pin_greedy_golden(orc):
    for pr, tg, c, pos, nsel in read_golden("greedy_accept_cases.txt"):
        p, s = orc.greedy_accept(_nums(pr, np.int32), _nums(tg, np.int32), _nums(c, np.float32))
        assert p[0].tolist() == [int(x) for x in pos.split()], f"greedy {pr} | {tg} | {c}: {p[0]}"
        assert int(s[0]) == int(nsel)


def brute_greedy(pred, target, conf):
    B, n = conf.shape
    pos = np.full((B, n), -1, dtype=np.int32)
    nsel = np.zeros(B, dtype=np.int32)
    for b in range(B):
        c = [float(x) for x in conf[b]]
        masked = [j for j in range(n) if not (math.isnan(c[j]) or c[j] == -math.inf)]
        chosen = [j for j in masked if int(pred[b, j]) == int(target[b, j])]
        if not chosen and masked:
            chosen = [max(masked, key=lambda j: (c[j], -j))]
        pos[b, :len(chosen)] = chosen
        nsel[b] = len(chosen)
    return pos, nsel


def pin_greedy_brute(orc):
    rng = np.random.default_rng(23)
    for n in (1, 2, 8, 16, 32):
        conf = _tied_confidences(rng, 60, n)
        for p_match in (0.0, 0.1, 0.5, 1.0):
            target = rng.integers(0, 100, size=(60, n)).astype(np.int32)
            pred = np.where(rng.random((60, n)) < p_match, target, target + 1).astype(np.int32)
            p, s = orc.greedy_accept(pred, target, conf)
            bp, bs = brute_greedy(pred, target, conf)
            assert np.array_equal(p, bp) and np.array_equal(s, bs), f"n={n} p={p_match}"


def pin_greedy_chain(orc):
    """Iterating greedy acceptance unmasks a block in K <= n iterations, at least
    one position each (TPF = n / K, Sec. 5). When no prediction ever matches,
    every iteration commits one position and the order is the serial
    denoising order: the pinned top-k ranking of the confidences. When every
    prediction matches, one iteration commits the whole block."""
    rng = np.random.default_rng(24)
    B, n = 40, 32
    base = rng.random((B, n), dtype=np.float32)
    target = rng.integers(0, 1000, size=(B, n)).astype(np.int32)
    order, _ = orc.unmask(base, n)
    never = target + 1
    conf = base.copy()
    seq = []
    for _ in range(n):
        p, s = orc.greedy_accept(never, target, conf)
        assert np.all(s == 1)
        seq.append(p[:, 0].copy())
        conf[np.arange(B), p[:, 0]] = -np.inf
    assert np.array_equal(np.stack(seq, axis=1), order)
    p, s = orc.greedy_accept(target, target, base)
    assert np.all(s == n) and np.all(p == np.arange(n))
    for p_match in (0.3, 0.7):
        conf = base.copy()
        iters = np.zeros(B, dtype=np.int64)
        for _ in range(n):
            pred = np.where(rng.random((B, n)) < p_match, target, target + 1).astype(np.int32)
            p, s = orc.greedy_accept(pred, target, conf)
            live = ~np.all(conf == -np.inf, axis=1)
            assert np.all(s[live] >= 1) and np.all(s[~live] == 0)
            iters += live
            for b in range(B):
                conf[b, p[b, :s[b]]] = -np.inf
        assert np.all(conf == -np.inf) and np.all((iters >= 1) & (iters <= n))


# --------------------------------------------------------------------------
# logits -> (argmax, confidence) pins
# --------------------------------------------------------------------------

def _bf16_rows(x):
    return W.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def pin_logits_golden(orc):
    for lg, idx, cf in read_golden("logits_argmax_cases.txt"):
        x = np.array([[float(v) for v in lg.split()]], dtype=np.float32)
        ids, conf = orc.logits_argmax(_bf16_rows(x))
        assert int(ids[0]) == int(idx), f"argmax of {lg}: {ids[0]}"
        want = float(cf)
        if math.isnan(want):
            assert math.isnan(conf[0]), f"confidence of {lg}: {conf[0]}"
        else:
            assert abs(conf[0] - want) <= 1e-15 * max(1.0, want), f"confidence of {lg}: {conf[0]} vs {want}"


def pin_logits_scipy(orc):
    """Against scipy.special.softmax (max probability) and numpy's argmax (first
    index of the max) on the same bf16 values, up to the full vocabulary."""
    rng = np.random.default_rng(31)
    for rows, V in ((64, 1), (64, 7), (32, 1000), (4, 131072)):
        bits = W.f32_to_bf16_bits((rng.standard_normal((rows, V)) * 3.0).astype(np.float32))
        vals = W.bf16_bits_to_f32(bits).astype(np.float64)
        ids, conf = orc.logits_argmax(bits)
        assert np.array_equal(ids, np.argmax(vals, axis=1))
        ref = scipy.special.softmax(vals, axis=1).max(axis=1)
        assert np.allclose(conf, ref, rtol=1e-12, atol=0), f"V={V}"


def pin_logits_closed_forms(orc):
    """One logit c above V-1 zeros: conf = 1 / (1 + (V-1) e^-c), id its index.
    Equal logits: conf = 1/V, id 0. Ties between maxima: the lowest index."""
    for V, c, at in ((2, 1.0, 1), (100, 4.0, 57), (131072, 16.0, 131071), (5, -3.0, 2)):
        x = np.zeros((1, V), dtype=np.float32)
        x[0, at] = c
        ids, conf = orc.logits_argmax(_bf16_rows(x))
        bound = V * 2.0 ** -52  # a plain fp64 sum of V terms
        if c > 0:
            assert int(ids[0]) == at
            assert abs(conf[0] - 1.0 / (1.0 + (V - 1) * math.exp(-c))) <= bound
        else:
            assert int(ids[0]) == (1 if at == 0 else 0)
            assert abs(conf[0] - 1.0 / (V - 1 + math.exp(c))) <= bound
    for V in (1, 3, 1024):
        ids, conf = orc.logits_argmax(_bf16_rows(np.full((1, V), 0.5, np.float32)))
        assert int(ids[0]) == 0 and abs(conf[0] - 1.0 / V) < 1e-15
    rng = np.random.default_rng(32)
    x = rng.integers(-4, 4, size=(200, 50)).astype(np.float32)  # many tied maxima
    ids, _ = orc.logits_argmax(_bf16_rows(x))
    assert all(int(ids[r]) == x[r].tolist().index(max(x[r].tolist())) for r in range(200))


def pin_logits_brute(orc):
    rng = np.random.default_rng(33)
    x = rng.standard_normal((40, 33)).astype(np.float32) * 4
    x[rng.random(x.shape) < 0.1] = -np.inf
    x[5, :] = -np.inf
    bits = _bf16_rows(x)
    vals = W.bf16_bits_to_f32(bits).astype(np.float64).tolist()
    ids, conf = orc.logits_argmax(bits)
    for r, row in enumerate(vals):
        m = max(row)
        if m == -math.inf:
            assert int(ids[r]) == 0 and conf[r] == 0.0
            continue
        assert int(ids[r]) == row.index(m)
        assert abs(conf[r] - 1.0 / sum(math.exp(v - m) for v in row)) < 1e-14


# --------------------------------------------------------------------------
# block KV commit pins
# --------------------------------------------------------------------------

def _commit_inputs(rng, case):
    kv = case.kv
    shape = (case.batch, case.block_len, case.num_kv_heads, case.head_dim)
    k_new = W.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
    v_new = W.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
    return kv, k_new, v_new


def pin_commit_gather(orc):
    """Committed rows read back through the page table with numpy indexing
    equal the new rows; every other slot keeps its bits; the prefix advances
    by the committed count (or stays, without advance)."""
    rng = np.random.default_rng(51)
    for seed, prefix in ((1, (7, 12)), (2, (0, 3)), (3, (16, 1))):
        case = small_case(seed, prefix=prefix)
        kv, k_new, v_new = _commit_inputs(rng, case)
        P, bl = kv.page_size, case.block_len
        for counts, advance in ((None, True), (rng.integers(0, bl + 1, case.batch).astype(np.int32), True),
                                (np.array([0, bl], np.int32), False)):
            kp, vp, pl = orc.kv_commit(k_new, v_new, counts, kv.page_table, kv.prefix_lens, kv.k_bits, kv.v_bits,
                                       advance)
            cnt = np.full(case.batch, bl, np.int32) if counts is None else counts
            written = np.zeros(kv.k_bits.shape[:3], dtype=bool)  # [page, head, slot]
            for b in range(case.batch):
                L = int(kv.prefix_lens[b])
                t = L + np.arange(cnt[b])
                pages, slots = kv.page_table[b, t // P], t % P
                assert np.array_equal(kp[pages, :, slots, :], k_new[b, :cnt[b]])
                assert np.array_equal(vp[pages, :, slots, :], v_new[b, :cnt[b]])
                written[pages, :, slots] = True
            assert np.array_equal(kp[~written], kv.k_bits[~written]) and np.array_equal(vp[~written], kv.v_bits[~written])
            assert np.array_equal(pl, kv.prefix_lens + cnt if advance else kv.prefix_lens)


def pin_commit_then_attention(orc):
    """A block staged by the commit (all bl rows, no advance) is what the
    attention reads as the block's own keys: the result equals fp64 SDPA over
    the prefix K/V followed by the new block K/V (both passes)."""
    rng = np.random.default_rng(52)
    case = small_case(9, prefix=(6, 13))
    kv, k_new, v_new = _commit_inputs(rng, case)
    kp, vp, _ = orc.kv_commit(k_new, v_new, None, kv.page_table, kv.prefix_lens, kv.k_bits, kv.v_bits, False)
    G = case.num_q_heads // case.num_kv_heads
    for mode, qbits in ((DIFF, case.q_draft_bits), (VER, case.q_verify_bits)):
        out, _ = orc.block_attn(qbits, kp, vp, kv.page_table, kv.prefix_lens, case.num_q_heads,
                                case.num_kv_heads, case.block_len, mode, case.scale)
        for b in range(case.batch):
            L = int(kv.prefix_lens[b])
            k_pre, v_pre = gather_contiguous(case, b)  # the original pools: the prefix part is untouched
            kb = np.transpose(W.bf16_bits_to_f32(k_new[b]).astype(np.float64), (1, 0, 2))
            vb = np.transpose(W.bf16_bits_to_f32(v_new[b]).astype(np.float64), (1, 0, 2))
            k = np.concatenate([k_pre[:, :L], kb], axis=1)
            v = np.concatenate([v_pre[:, :L], vb], axis=1)
            q = np.transpose(q_f64(qbits[b]), (1, 0, 2))
            if mode == DIFF:
                ref = sdpa(q, repeat_heads(k, G), repeat_heads(v, G), case.scale)
            else:
                qfull = np.concatenate([rng.standard_normal((case.num_q_heads, L, case.head_dim)), q], axis=1)
                ref = sdpa(qfull, repeat_heads(k, G), repeat_heads(v, G), case.scale, causal=True)[:, L:, :]
            assert_close(np.transpose(out[b], (1, 0, 2)), ref, 1e-12, f"commit + attention mode={mode}")


def pin_commit_rollback_chain(orc):
    """Linear self-speculation steps: commit the accepted rows (accepted_len
    from the pinned accept rule) and advance; the next step's block lands
    right after them, over the rejected rows (the cache rebuilt at the
    rejection point, Sec. 3 Mode 3)."""
    rng = np.random.default_rng(53)
    case = small_case(11, B=3, prefix=(4, 9, 0))
    kv = case.kv
    P, bl = kv.page_size, case.block_len
    kp, vp, pl = kv.k_bits.copy(), kv.v_bits.copy(), kv.prefix_lens.copy()
    history = [[] for _ in range(case.batch)]  # committed rows in order, per sequence
    for step in range(3):
        _, k_new, v_new = _commit_inputs(rng, case)
        d, v = W.make_accept_ids(rng, case.batch, bl, 50, 0.6)
        acc = orc.accept(d, v)
        room = (kv.page_table.shape[1] * P - pl).astype(np.int32)
        acc = np.minimum(acc, room).astype(np.int32)
        kp, vp, pl_new = orc.kv_commit(k_new, v_new, acc, kv.page_table, pl, kp, vp, True)
        assert np.array_equal(pl_new, pl + acc)
        for b in range(case.batch):
            history[b] += [k_new[b, j] for j in range(acc[b])]
        pl = pl_new
    for b in range(case.batch):
        L0 = int(kv.prefix_lens[b])
        t = L0 + np.arange(len(history[b]))
        got = kp[kv.page_table[b, t // P], :, t % P, :]
        assert np.array_equal(got, np.array(history[b]).reshape(got.shape))


# --------------------------------------------------------------------------
# table-mask attention and the quadratic self-speculation mask
# --------------------------------------------------------------------------

def pin_quadss_layout(orc):
    """Eq. quad_input: 1 + k + k^2 block slots, k^2 of them masks. Chain slots
    (the AR token and the k speculative tokens) see only chain slots, causally;
    the masks of a group see the chain through their speculative token and
    exactly the k masks of their group; every slot sees itself."""
    for k in range(1, 6):
        m = orc.quadss_mask(k)
        n = 1 + k + k * k
        assert len(m) == n
        bits = [[(int(m[i]) >> j) & 1 for j in range(n)] for i in range(n)]
        spec = [0] + [1 + (g - 1) * (k + 1) for g in range(1, k + 1)]
        masks = [j for j in range(n) if j not in spec]
        assert len(masks) == k * k
        for i in range(n):
            assert bits[i][i] == 1
            if i in spec:
                assert [j for j in range(n) if bits[i][j]] == [j for j in spec if j <= i]
            else:
                g = (i - 1) // (k + 1) + 1
                own = [spec[g] + r for r in range(1, k + 1)]
                assert [j for j in masks if bits[i][j]] == own
                assert [j for j in spec if bits[i][j]] == spec[:g + 1]
    assert all(orc.quadss_mask(5) < 2 ** 31) and len(orc.quadss_mask(5)) == 31
    try:
        orc.quadss_mask(6)
        raise AssertionError("k=6 (43 slots) must be refused")
    except ValueError:
        pass


def pin_masked_reduces_to_modes(orc):
    """A table of all ones is the diffusion pass; the lower-triangular table
    is the verify pass (bit-identical: same arithmetic in the same order)."""
    for seed, prefix in ((41, (7, 12)), (42, (0, 5))):
        case = small_case(seed, prefix=prefix)
        bl = case.block_len
        full = np.full(bl, (1 << bl) - 1, dtype=np.uint32)
        tril = np.array([(2 << i) - 1 for i in range(bl)], dtype=np.uint32)
        for table, mode, qb in ((full, DIFF, case.q_draft_bits), (tril, VER, case.q_verify_bits)):
            ref, rl = orc.block_attn(qb, case.kv.k_bits, case.kv.v_bits, case.kv.page_table, case.kv.prefix_lens,
                                     case.num_q_heads, case.num_kv_heads, bl, mode, case.scale)
            got, gl, _ = orc.block_attn_masked(qb, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                               case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, bl,
                                               table, case.scale)
            assert np.array_equal(got, ref) and np.array_equal(gl, rl), f"mode {mode}"


def pin_quadss_against_sdpa(orc):
    """Quadratic-SS attention row by row against fp64 SDPA on exactly the keys
    the reading names: a chain row = causal attention along the prefix and
    the chain; a mask row of group g = unmasked attention over the prefix, the
    chain through its speculative token and its group's masks."""
    for k, prefix in ((2, (5, 9)), (3, (0, 14)), (5, (6, 1))):
        bl = 1 + k + k * k
        case = W.make_block_attn_case("quadss", 2, 4, 2, 16, bl, 4, list(prefix), 60 + k, shuffle_pages=True)
        table = orc.quadss_mask(k)
        out, _, _ = orc.block_attn_masked(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                          case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, bl, table,
                                          case.scale)
        G = case.num_q_heads // case.num_kv_heads
        for b in range(case.batch):
            L = int(case.kv.prefix_lens[b])
            kf, vf = gather_contiguous(case, b)  # [Hkv, L + bl, D]
            q = np.transpose(q_f64(case.q_draft_bits[b]), (1, 0, 2))  # [Hq, bl, D]
            for i in range(bl):
                keys = list(range(L)) + [L + j for j in range(bl) if (int(table[i]) >> j) & 1]
                ref = sdpa(q[:, i:i + 1], repeat_heads(kf[:, keys], G), repeat_heads(vf[:, keys], G), case.scale)
                assert_close(out[b, i], ref[:, 0], 1e-12, f"quadss k={k} b={b} row {i}")


def pin_masked_empty_row(orc):
    """With no prefix, a row whose table entry is empty sees no key: o = 0, lse = -inf."""
    case = small_case(43, prefix=(0, 0))
    bl = case.block_len
    table = np.array([(2 << i) - 1 for i in range(bl)], dtype=np.uint32)
    table[2] = 0
    out, lse, _ = orc.block_attn_masked(case.q_draft_bits, case.kv.k_bits, case.kv.v_bits, case.kv.page_table,
                                        case.kv.prefix_lens, case.num_q_heads, case.num_kv_heads, bl, table,
                                        case.scale)
    assert np.all(out[:, 2] == 0) and np.all(lse[:, :, 2] == -np.inf)
    assert np.all(np.isfinite(lse[:, :, [0, 1, 3]]))


# --------------------------------------------------------------------------
# AR-diffusion ensemble verifier pins
# --------------------------------------------------------------------------

def pin_ensemble_golden(orc):
    for ar, df, lam, idx, cf in read_golden("ensemble_cases.txt"):
        a = _bf16_rows(np.array([[float(v) for v in ar.split()]], np.float32))
        d = _bf16_rows(np.array([[float(v) for v in df.split()]], np.float32))
        ids, conf = orc.ensemble_argmax(a, d, float(lam))
        assert int(ids[0]) == int(idx) and abs(conf[0] - float(cf)) < 1e-15, f"{ar} | {df} | {lam}: {ids[0]} {conf[0]}"


def pin_ensemble_limits(orc):
    """lambda = 1 is the AR verifier alone, lambda = 0 the diffusion one: the
    pinned logits rule on each input."""
    rng = np.random.default_rng(71)
    a = _bf16_rows(rng.standard_normal((20, 500)).astype(np.float32) * 3)
    d = _bf16_rows(rng.standard_normal((20, 500)).astype(np.float32) * 3)
    for lam, src in ((1.0, a), (0.0, d)):
        ids, conf = orc.ensemble_argmax(a, d, lam)
        ri, rc = orc.logits_argmax(src)
        assert np.array_equal(ids, ri) and np.allclose(conf, rc, rtol=1e-14, atol=0)


def pin_ensemble_scipy(orc):
    """Against scipy.special.softmax mixtures (ids where the top two are apart)."""
    rng = np.random.default_rng(72)
    for V, lam in ((7, 0.3), (1000, 0.5), (32000, 0.8)):
        a = _bf16_rows(rng.standard_normal((16, V)).astype(np.float32) * 3)
        d = _bf16_rows(rng.standard_normal((16, V)).astype(np.float32) * 3)
        p = (lam * scipy.special.softmax(W.bf16_bits_to_f32(a).astype(np.float64), axis=1)
             + (1 - lam) * scipy.special.softmax(W.bf16_bits_to_f32(d).astype(np.float64), axis=1))
        ids, conf = orc.ensemble_argmax(a, d, lam)
        assert np.allclose(conf, p.max(axis=1), rtol=1e-12, atol=0)
        top2 = np.sort(p, axis=1)[:, -2:]
        clear = top2[:, 1] - top2[:, 0] > 1e-12
        assert np.array_equal(ids[clear], np.argmax(p, axis=1)[clear])


def pin_ensemble_empty_side(orc):
    """A distribution with nothing above -inf contributes nothing."""
    rng = np.random.default_rng(73)
    d = _bf16_rows(rng.standard_normal((8, 64)).astype(np.float32))
    a = _bf16_rows(np.full((8, 64), -np.inf, np.float32))
    ids, conf = orc.ensemble_argmax(a, d, 0.3)
    ri, rc = orc.logits_argmax(d)
    assert np.array_equal(ids, ri) and np.allclose(conf, 0.7 * rc, rtol=1e-14, atol=0)


ATTENTION_PINS = [pin_decode_bl1, pin_diffusion_full_attention, pin_verify_causal_tail, pin_lse_logsumexp,
                  pin_softmax_rows, pin_page_permutation, pin_block_permutation, pin_closed_forms,
                  pin_golden_uniform, pin_split_combine, pin_block_attn_rows]
DECISION_PINS = [pin_accept_golden, pin_accept_brute, pin_accept_statistics, pin_unmask_golden,
                 pin_unmask_brute, pin_unmask_lexsort, pin_threshold_golden, pin_threshold_brute,
                 pin_threshold_limits, pin_greedy_golden, pin_greedy_brute, pin_greedy_chain]
LOGITS_PINS = [pin_logits_golden, pin_logits_scipy, pin_logits_closed_forms, pin_logits_brute]
COMMIT_PINS = [pin_commit_gather, pin_commit_then_attention, pin_commit_rollback_chain]
MASK_PINS = [pin_quadss_layout, pin_masked_reduces_to_modes, pin_quadss_against_sdpa, pin_masked_empty_row]
ENSEMBLE_PINS = [pin_ensemble_golden, pin_ensemble_limits, pin_ensemble_scipy, pin_ensemble_empty_side]
ALL_PINS = ATTENTION_PINS + DECISION_PINS + LOGITS_PINS + COMMIT_PINS + MASK_PINS + ENSEMBLE_PINS
