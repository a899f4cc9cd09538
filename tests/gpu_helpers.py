"""Helpers for GPU tests: upload seeded inputs, run the C ABI, compare."""
from __future__ import annotations

import numpy as np
import torch

from paper_2607_05722_gb300 import nld
from paper_2607_05722_gb300 import workloads as W

# Attention tolerance (bf16 inputs, fp32 accumulation, bf16 P and output).
MAX_ABS = 1e-2
REL_L2 = 5e-3
LSE_ABS = 2e-3


def bits_to_bf16(bits: np.ndarray, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


class DeviceCase:
    """A BlockAttnCase resident on the GPU."""

    def __init__(self, case: W.BlockAttnCase, device="cuda"):
        self.case = case
        kv = case.kv
        self.k = bits_to_bf16(kv.k_bits, device)
        self.v = bits_to_bf16(kv.v_bits, device)
        # -1 entries past each sequence are never read by the kernel; keep them
        self.table = torch.from_numpy(kv.page_table).to(device)
        self.prefix = torch.from_numpy(kv.prefix_lens).to(device)
        self.q = {W.MODE_DIFFUSION: bits_to_bf16(case.q_draft_bits, device),
                  W.MODE_VERIFY: bits_to_bf16(case.q_verify_bits, device)}

    def q_bits(self, mode):
        return self.case.q_draft_bits if mode == W.MODE_DIFFUSION else self.case.q_verify_bits

    def params(self, num_splits=0, flags=0, softmax_scale=0.0):
        c = self.case
        return nld.make_params(c.batch, c.num_q_heads, c.num_kv_heads, c.head_dim, c.page_size,
                               c.kv.num_pages, c.kv.max_pages, num_splits, softmax_scale, flags)

    def run(self, mode, num_splits=0, q=None, flags=0, softmax_scale=0.0):
        c = self.case
        p = self.params(num_splits, flags, softmax_scale)
        q = self.q[mode] if q is None else q
        out = torch.empty((c.batch, c.block_len, c.num_q_heads, c.head_dim), dtype=torch.bfloat16, device=q.device)
        lse = torch.empty((c.batch, c.num_q_heads, c.block_len), dtype=torch.float32, device=q.device)
        ws_bytes = nld.nld_block_attn_workspace_size(p, c.block_len)
        ws = torch.zeros(max(ws_bytes, 1), dtype=torch.uint8, device=q.device) if ws_bytes else None
        nld.nld_block_attn(p, q, self.k, self.v, self.table, self.prefix, c.block_len, mode, out, lse, ws)
        return out, lse


def oracle_full(orc, case: W.BlockAttnCase, mode):
    qb = case.q_draft_bits if mode == W.MODE_DIFFUSION else case.q_verify_bits
    return orc.block_attn(qb, case.kv.k_bits, case.kv.v_bits, case.kv.page_table, case.kv.prefix_lens,
                          case.num_q_heads, case.num_kv_heads, case.block_len, mode, case.scale)


def compare_attn(out_gpu: torch.Tensor, lse_gpu: torch.Tensor, out_ref: np.ndarray, lse_ref: np.ndarray, what="",
                 max_abs=MAX_ABS):
    o = out_gpu.float().cpu().numpy().astype(np.float64)
    err = np.abs(o - out_ref)
    bar = max_abs
    max_abs = float(err.max()) if err.size else 0.0
    rel = float(np.linalg.norm(o - out_ref) / max(np.linalg.norm(out_ref), 1e-30))
    assert np.all(np.isfinite(o)), f"{what}: non-finite output"
    assert max_abs <= bar, f"{what}: max abs err {max_abs:.3e}"
    assert rel <= REL_L2, f"{what}: rel L2 err {rel:.3e}"
    if lse_gpu is not None:
        l = lse_gpu.cpu().numpy().astype(np.float64)
        lerr = float(np.max(np.abs(l - lse_ref))) if l.size else 0.0
        assert lerr <= LSE_ABS, f"{what}: lse err {lerr:.3e}"
    return max_abs, rel


def rows_per_unit(case: W.BlockAttnCase, per_unit: int, seed: int):
    """(b, i, h) rows: `per_unit` random rows of every (sequence, KV head),
    i.e. of every CTA group of the launch, plus each sequence's first and
    last block rows."""
    rng = np.random.default_rng(seed)
    G = case.num_q_heads // case.num_kv_heads
    rows = set()
    for b in range(case.batch):
        rows.add((b, 0, 0))
        rows.add((b, case.block_len - 1, case.num_q_heads - 1))
        for g in range(case.num_kv_heads):
            for _ in range(per_unit):
                rows.add((b, int(rng.integers(case.block_len)), g * G + int(rng.integers(G))))
    return np.array(sorted(rows), dtype=np.int32)


def sample_rows(case: W.BlockAttnCase, n: int, seed: int):
    """(b, i, h) rows: random ones plus each sequence's first and last block rows."""
    rng = np.random.default_rng(seed)
    rows = {(int(rng.integers(case.batch)), int(rng.integers(case.block_len)), int(rng.integers(case.num_q_heads)))
            for _ in range(n)}
    for b in range(min(case.batch, 8)):
        rows.add((b, 0, 0))
        rows.add((b, case.block_len - 1, case.num_q_heads - 1))
    return np.array(sorted(rows), dtype=np.int32)
