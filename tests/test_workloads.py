"""The seeded input generator: determinism, bf16 rounding, page tables."""
import numpy as np
import torch

from paper_2607_05722_gb300 import workloads as W


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32),
                        rng.standard_normal(1000).astype(np.float32) * 1e-30,
                        np.array([0.0, -0.0, 1.0, -1.5, 3.0e38, 1.00390625, 1.01171875], dtype=np.float32)])
    ours = W.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    back = W.bf16_bits_to_f32(ours)
    assert np.array_equal(back, torch.from_numpy(ours.view(np.int16)).view(torch.bfloat16).float().numpy())


def test_workloads_deterministic_and_well_formed():
    for name in W.WORKLOADS:
        small = {"batch": 2, "prefix_override": [37, 100]} if W.WORKLOADS[name]["batch"] > 1 else {
            "prefix_override": [64]}
        a = W.make_workload(name, seed=3, **small)
        b = W.make_workload(name, seed=3, **small)
        assert np.array_equal(a.attn.kv.k_bits, b.attn.kv.k_bits)
        assert np.array_equal(a.attn.q_verify_bits, b.attn.q_verify_bits)
        assert np.array_equal(a.verify_ids, b.verify_ids)
        kv = a.attn.kv
        used = []
        for bi, L in enumerate(kv.prefix_lens):
            need = -(-(int(L) + a.attn.block_len) // kv.page_size)
            row = kv.page_table[bi]
            assert np.all(row[:need] >= 0) and np.all(row[:need] < kv.num_pages)
            assert np.all(row[need:] == -1)
            used.extend(row[:need].tolist())
        assert len(used) == len(set(used)), "a physical page serves two logical pages"


def test_full_size_prefix_ranges():
    rng = np.random.Generator(np.random.PCG64(0))
    p = W.WORKLOADS["14b_b16_h40x8_d128_L8k-16k_bl32"]["prefix"](rng, 1000)
    assert p.min() >= 8192 and p.max() <= 16384
    p = W.WORKLOADS["conc_b8_h32x8_d128_L512-8192_bl8"]["prefix"](rng, 1000)
    assert p.min() >= 512 and p.max() <= 8192
