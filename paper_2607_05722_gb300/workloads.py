"""Seeded synthetic inputs shaped like the paper's decoding workloads.

This module holds random draws only: normal / uniform / Beta samples, their
round-to-nearest-even conversion to bf16 bit patterns, page-table construction
and token-id draws. It contains none of the attention or token-decision
arithmetic, so both the CUDA path and the CPU oracle can read its output.

Shapes follow the decoding workloads of the paper (Sec. 3: a block of draft
tokens attends to a cached prefix; Sec. 6.5: 8B-class models served at
concurrency 1..128). Head counts and head_dim are those of the 3B/8B/14B
decoder shapes (32 or 40 query heads over 8 KV heads, head_dim 128), plus a
small single-KV-head case.

Draw order inside one workload (one ``numpy.random.Generator(PCG64(seed))``):
prefix lengths, page permutation, K pool, V pool, draft-pass queries,
verify-pass queries, draft ids, agreement flags, replacement ids,
confidences. Everything is a pure function of ``(config, seed)``.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np

# Mask modes, by their meaning in the paper (Sec. 2.2 and Sec. 3):
# the diffusion draft pass is bidirectional inside the block, the AR verify
# pass is causal inside the block. Values match include/nld.h.
MODE_DIFFUSION = 0
MODE_VERIFY = 1

_CHUNK = 1 << 24  # elements drawn per normal() call, bounds fp32 temporaries


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (round to nearest, ties to even); return bits.

    Inputs here are finite normal/uniform draws, so NaN handling is not needed.
    """
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16(rng: np.random.Generator, shape) -> np.ndarray:
    """N(0,1) draws in fp32, rounded to bf16 bits, drawn in bounded chunks."""
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.uint16)
    for s in range(0, n, _CHUNK):
        e = min(n, s + _CHUNK)
        out[s:e] = f32_to_bf16_bits(rng.standard_normal(e - s, dtype=np.float32))
    return out.reshape(shape)


@dataclasses.dataclass
class PagedKV:
    """A paged bf16 KV pool: ``[num_pages, Hkv, P, D]`` per K and V (bit patterns)."""

    k_bits: np.ndarray
    v_bits: np.ndarray
    page_table: np.ndarray  # int32 [B, max_pages]; -1 past each sequence's pages
    prefix_lens: np.ndarray  # int32 [B]
    page_size: int
    num_pages: int
    max_pages: int


@dataclasses.dataclass
class BlockAttnCase:
    """One block-attention workload: queries for both passes over one KV pool."""

    name: str
    batch: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    block_len: int
    scale: float
    q_draft_bits: np.ndarray  # [B, bl, Hq, D] bf16 bits, diffusion-draft pass
    q_verify_bits: np.ndarray  # [B, bl, Hq, D] bf16 bits, AR-verify pass
    kv: PagedKV

    @property
    def page_size(self) -> int:
        return self.kv.page_size

    def kv_bytes_per_pass(self) -> int:
        """Algorithmic KV bytes of one pass: every visible key and value once per (b, kv head)."""
        toks = int(np.sum(self.kv.prefix_lens.astype(np.int64) + self.block_len))
        return toks * self.num_kv_heads * self.head_dim * 2 * 2


def make_page_table(rng: np.random.Generator, prefix_lens: np.ndarray, block_len: int,
                    page_size: int, shuffle: bool, spare_pages: int = 0):
    """Give each sequence ceil((L_b + bl) / P) pages from one shared pool.

    With ``shuffle`` the pool order is a random permutation, so logical pages of
    one sequence land on scattered physical pages.
    """
    need = [int(math.ceil((int(L) + block_len) / page_size)) for L in prefix_lens]
    total = int(sum(need)) + spare_pages
    order = rng.permutation(total).astype(np.int32) if shuffle else np.arange(total, dtype=np.int32)
    max_pages = max(need)
    table = np.full((len(need), max_pages), -1, dtype=np.int32)
    pos = 0
    for b, nb in enumerate(need):
        table[b, :nb] = order[pos:pos + nb]
        pos += nb
    return table, total, max_pages


def make_block_attn_case(name: str, batch: int, num_q_heads: int, num_kv_heads: int,
                         head_dim: int, block_len: int, page_size: int,
                         prefix_lens, seed: int, shuffle_pages: bool = True,
                         rng: Optional[np.random.Generator] = None) -> BlockAttnCase:
    """Build Q (both passes) and a paged KV pool holding prefix + block slots.

    ``prefix_lens`` is a list/array of B ints, or a callable ``rng -> array``
    (drawn first from the generator).
    """
    if rng is None:
        rng = np.random.Generator(np.random.PCG64(seed))
    if callable(prefix_lens):
        prefix_lens = prefix_lens(rng)
    prefix_lens = np.asarray(prefix_lens, dtype=np.int32).reshape(batch)
    table, num_pages, max_pages = make_page_table(rng, prefix_lens, block_len, page_size, shuffle_pages)
    kshape = (num_pages, num_kv_heads, page_size, head_dim)
    k_bits = normal_bf16(rng, kshape)
    v_bits = normal_bf16(rng, kshape)
    qshape = (batch, block_len, num_q_heads, head_dim)
    q_draft = normal_bf16(rng, qshape)
    q_verify = normal_bf16(rng, qshape)
    kv = PagedKV(k_bits, v_bits, table, prefix_lens, page_size, num_pages, max_pages)
    return BlockAttnCase(name, batch, num_q_heads, num_kv_heads, head_dim, block_len,
                         1.0 / math.sqrt(head_dim), q_draft, q_verify, kv)


def make_accept_ids(rng: np.random.Generator, batch: int, n: int, vocab: int, p_agree: float):
    """Draft ids uniform over the vocabulary; each verify id equals its draft with
    probability ``p_agree``, else is uniform over the other vocab - 1 ids."""
    draft = rng.integers(0, vocab, size=(batch, n), dtype=np.int64)
    agree = rng.random(size=(batch, n)) < p_agree
    other = rng.integers(0, vocab - 1, size=(batch, n), dtype=np.int64)
    other = other + (other >= draft)
    verify = np.where(agree, draft, other)
    return draft.astype(np.int32), verify.astype(np.int32)


def make_confidences(rng: np.random.Generator, batch: int, n: int, dist: str = "uniform"):
    """fp32 confidences: ``uniform`` = U(0,1), ``beta22`` = Beta(2, 2)."""
    if dist == "uniform":
        return rng.random(size=(batch, n), dtype=np.float32)
    if dist == "beta22":
        return rng.beta(2.0, 2.0, size=(batch, n)).astype(np.float32)
    raise ValueError(dist)


# ---------------------------------------------------------------------------
# Named workloads. Each is described by what it is, with its sizes.
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class Workload:
    """A full decoding-step workload: attention case + decision inputs."""

    attn: BlockAttnCase
    draft_ids: np.ndarray
    verify_ids: np.ndarray
    conf: List[np.ndarray]  # one [B, bl] array per diffusion denoising step
    unmask_k: List[int]
    vocab: int
    p_agree: float
    steps: List[str]  # pass sequence, e.g. ["diffusion", "verify", "accept"]
    description: str


WORKLOADS: Dict[str, dict] = {
    # Single KV head, head_dim 64, one contiguous 256-token page of prefix and
    # the 8 block slots on a second page.
    "tiny_b1_h4x1_d64_L256_bl8": dict(
        batch=1, hq=4, hkv=1, d=64, bl=8, page=256, shuffle=False,
        prefix=lambda rng, B: np.full(B, 256), vocab=32000, p=0.8,
        conf="uniform", k=[2], denoise_steps=1,
        steps=["diffusion", "verify", "accept", "unmask"]),
    # 8B-class GQA decoder shape at concurrency 1 with a 4096-token prefix.
    "8b_b1_h32x8_d128_L4096_bl16": dict(
        batch=1, hq=32, hkv=8, d=128, bl=16, page=16, shuffle=True,
        prefix=lambda rng, B: np.full(B, 4096), vocab=131072, p=0.75,
        conf="uniform", k=[4], denoise_steps=1,
        steps=["diffusion", "unmask", "verify", "accept"]),
    # 8B shape, 32768-token prefix, block of 32.
    "long_b1_h32x8_d128_L32768_bl32": dict(
        batch=1, hq=32, hkv=8, d=128, bl=32, page=16, shuffle=True,
        prefix=lambda rng, B: np.full(B, 32768), vocab=131072, p=0.75,
        conf="beta22", k=[4, 8], denoise_steps=1,
        steps=["diffusion", "verify", "accept", "unmask"]),
    # 14B-class shape: 40 q / 8 kv heads, 16 sequences of 8192..16384 tokens,
    # four denoising steps of top-8 then one verify pass.
    "14b_b16_h40x8_d128_L8k-16k_bl32": dict(
        batch=16, hq=40, hkv=8, d=128, bl=32, page=16, shuffle=True,
        prefix=lambda rng, B: rng.integers(8192, 16384, size=B, endpoint=True), vocab=131072, p=0.75,
        conf="uniform", k=[8], denoise_steps=4,
        steps=["diffusion", "unmask"] * 4 + ["verify", "accept"]),
}
for _B in (8, 32, 64, 128):
    # Ragged concurrency sweep, verify pass only.
    WORKLOADS[f"conc_b{_B}_h32x8_d128_L512-8192_bl8"] = dict(
        batch=_B, hq=32, hkv=8, d=128, bl=8, page=16, shuffle=True,
        prefix=lambda rng, B: rng.integers(512, 8192, size=B, endpoint=True), vocab=131072, p=0.7,
        conf="uniform", k=[2], denoise_steps=0, steps=["verify", "accept"])

HEADLINE = "8b_b1_h32x8_d128_L4096_bl16"


def make_workload(name: str, seed: int = 0, batch: Optional[int] = None,
                  prefix_override=None) -> Workload:
    """Build a named workload. ``batch``/``prefix_override`` shrink it for tests."""
    cfg = WORKLOADS[name]
    B = cfg["batch"] if batch is None else batch
    rng = np.random.Generator(np.random.PCG64(seed))
    if prefix_override is not None:
        prefix = np.asarray(prefix_override, dtype=np.int32).reshape(B)
    else:
        prefix = np.asarray(cfg["prefix"](rng, B), dtype=np.int32)
    attn = make_block_attn_case(name, B, cfg["hq"], cfg["hkv"], cfg["d"], cfg["bl"], cfg["page"],
                                prefix, seed, shuffle_pages=cfg["shuffle"], rng=rng)
    draft, verify = make_accept_ids(rng, B, cfg["bl"], cfg["vocab"], cfg["p"])
    nconf = max(1, cfg["denoise_steps"])
    conf = [make_confidences(rng, B, cfg["bl"], cfg["conf"]) for _ in range(nconf)]
    return Workload(attn, draft, verify, conf, list(cfg["k"]), cfg["vocab"], cfg["p"],
                    list(cfg["steps"]), name)


# ---------------------------------------------------------------------------
# Device-side draws for timing the large workloads (up to ~2.2 GB of KV):
# the same shapes and distributions, drawn with a seeded torch generator on
# the GPU instead of numpy on the host. Parity tests use the numpy path.
# ---------------------------------------------------------------------------

def make_device_workload(name: str, seed: int, device, batch: Optional[int] = None):
    """A named workload with Q/K/V drawn on `device` (bf16 from N(0,1) fp32),
    prefix lengths, page table, ids and confidences drawn on the host.
    Returns a dict of device tensors plus the host-side metadata."""
    import torch

    cfg = WORKLOADS[name]
    B = cfg["batch"] if batch is None else batch
    rng = np.random.Generator(np.random.PCG64(seed))
    prefix = np.asarray(cfg["prefix"](rng, B), dtype=np.int32)
    table, num_pages, max_pages = make_page_table(rng, prefix, cfg["bl"], cfg["page"], cfg["shuffle"])
    draft, verify = make_accept_ids(rng, B, cfg["bl"], cfg["vocab"], cfg["p"])
    nconf = max(1, cfg["denoise_steps"])
    conf = [make_confidences(rng, B, cfg["bl"], cfg["conf"]) for _ in range(nconf)]
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)

    def normal(shape):
        return torch.randn(shape, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)

    kshape = (num_pages, cfg["hkv"], cfg["page"], cfg["d"])
    qshape = (B, cfg["bl"], cfg["hq"], cfg["d"])
    return {
        "name": name, "batch": B, "hq": cfg["hq"], "hkv": cfg["hkv"], "d": cfg["d"], "bl": cfg["bl"],
        "page": cfg["page"], "num_pages": num_pages, "max_pages": max_pages, "unmask_k": list(cfg["k"]),
        "denoise_steps": cfg["denoise_steps"], "steps": list(cfg["steps"]),
        "k": normal(kshape), "v": normal(kshape), "q_draft": normal(qshape), "q_verify": normal(qshape),
        "page_table": torch.from_numpy(table).to(device), "prefix_lens": torch.from_numpy(prefix).to(device),
        "draft_ids": torch.from_numpy(draft).to(device), "verify_ids": torch.from_numpy(verify).to(device),
        "conf": [torch.from_numpy(c).to(device) for c in conf],
        "kv_bytes_per_pass": int(np.sum(prefix.astype(np.int64) + cfg["bl"])) * cfg["hkv"] * cfg["d"] * 4,
    }
