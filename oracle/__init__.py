"""fp64 CPU oracle for paged block attention, split combine, accept, top-k,
threshold and greedy unmasking, logits -> (argmax, confidence), and the block
KV commit into the paged cache.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the CPU
baseline of ``bench.py`` use it. The product path never imports it. It shares
no code with the CUDA library; it reads the same seeded inputs (bf16 bit
patterns as uint16) that the CUDA path reads.

The arithmetic lives in ``nld_oracle.c`` (plain loops, fp64). This module only
compiles it on first use and marshals numpy arrays through ctypes.

Parity status per function: every function here is pinned by the
``-m "not gpu"`` tests in ``tests/test_oracle_pins.py`` (library routines,
closed forms, brute force, invariants, mutation checks).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "nld_oracle.c")
BUILD_DIR = os.path.join(_HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "libnld_oracle.so")

MODE_DIFFUSION = 0
MODE_VERIFY = 1

_lock = threading.Lock()
_default = None


def compile_oracle(source: str = SOURCE, out_path: str = LIB_PATH, openmp: bool = True) -> str:
    """Compile the oracle C source into a shared library; return its path."""
    os.makedirs(os.path.dirname(out_path), exist_ok=True)
    base = ["gcc", "-O2", "-ffp-contract=off", "-shared", "-fPIC", "-std=c11", source, "-o", out_path, "-lm"]
    if openmp:
        try:
            subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
            return out_path
        except subprocess.CalledProcessError:
            pass
    subprocess.run(base, check=True, capture_output=True)
    return out_path


class Oracle:
    """ctypes handle on one compiled oracle library."""

    def __init__(self, lib_path: str):
        lib = ctypes.CDLL(lib_path)
        P = ctypes.c_void_p
        I = ctypes.c_int
        Lg = ctypes.c_long
        D = ctypes.c_double
        lib.nldo_block_attn.argtypes = [P, P, P, P, P, I, I, I, I, I, I, I, I, I, D, Lg, Lg, P, P, P, Lg]
        lib.nldo_block_attn.restype = I
        lib.nldo_block_attn_rows.argtypes = [P, P, P, P, P, I, I, I, I, I, I, I, I, I, D, Lg, P, P, P]
        lib.nldo_block_attn_rows.restype = I
        lib.nldo_combine.argtypes = [P, P, I, Lg, I, P, P]
        lib.nldo_combine.restype = None
        lib.nldo_accept.argtypes = [P, P, I, I, P]
        lib.nldo_accept.restype = None
        lib.nldo_unmask.argtypes = [P, I, I, I, P, P]
        lib.nldo_unmask.restype = None
        lib.nldo_unmask_threshold.argtypes = [P, I, I, ctypes.c_float, P, P]
        lib.nldo_unmask_threshold.restype = None
        lib.nldo_greedy_accept.argtypes = [P, P, P, I, I, P, P]
        lib.nldo_greedy_accept.restype = None
        lib.nldo_logits_argmax.argtypes = [P, Lg, I, Lg, P, P]
        lib.nldo_logits_argmax.restype = None
        lib.nldo_kv_commit.argtypes = [P, P, P, P, P, I, P, P, I, I, I, I, I, I, I]
        lib.nldo_kv_commit.restype = None
        lib.nldo_block_attn_masked.argtypes = [P, P, P, P, P, I, I, I, I, I, I, I, I, P, D, P, P, P, Lg]
        lib.nldo_block_attn_masked.restype = I
        lib.nldo_quadss_mask.argtypes = [I, P]
        lib.nldo_quadss_mask.restype = I
        lib.nldo_ensemble_argmax.argtypes = [P, P, Lg, I, Lg, D, P, P]
        lib.nldo_ensemble_argmax.restype = None
        lib.nldo_max_threads.argtypes = []
        lib.nldo_max_threads.restype = I
        self.lib = lib
        self.path = lib_path

    @staticmethod
    def _p(a: Optional[np.ndarray]):
        return None if a is None else a.ctypes.data

    def max_threads(self) -> int:
        return int(self.lib.nldo_max_threads())

    def block_attn(self, q_bits, k_bits, v_bits, page_table, prefix_lens, num_q_heads, num_kv_heads,
                   block_len, mode, scale, key_begin=0, key_end=-1, want_probs=False):
        """All rows. Returns (out [B,bl,Hq,D] f64, lse [B,Hq,bl] f64[, probs [B,Hq,bl,maxN]])."""
        q = np.ascontiguousarray(q_bits, dtype=np.uint16)
        k = np.ascontiguousarray(k_bits, dtype=np.uint16)
        v = np.ascontiguousarray(v_bits, dtype=np.uint16)
        pt = np.ascontiguousarray(page_table, dtype=np.int32)
        pl = np.ascontiguousarray(prefix_lens, dtype=np.int32)
        B, bl, Hq, D = q.shape
        assert bl == block_len and Hq == num_q_heads
        num_pages, Hkv, P, Dk = k.shape
        assert Dk == D and Hkv == num_kv_heads and v.shape == k.shape
        out = np.zeros((B, bl, Hq, D), dtype=np.float64)
        lse = np.zeros((B, Hq, bl), dtype=np.float64)
        probs = None
        stride = 0
        if want_probs:
            stride = int(np.max(pl.astype(np.int64) + bl)) if B else 1
            probs = np.zeros((B, Hq, bl, stride), dtype=np.float64)
        rc = self.lib.nldo_block_attn(self._p(q), self._p(k), self._p(v), self._p(pt), self._p(pl),
                                      B, Hq, Hkv, D, P, num_pages, pt.shape[1], bl, int(mode),
                                      float(scale), int(key_begin), int(key_end),
                                      self._p(out), self._p(lse), self._p(probs), stride)
        if rc != 0:
            raise ValueError(f"oracle block_attn failed: {rc}")
        return (out, lse, probs) if want_probs else (out, lse)

    def block_attn_rows(self, q_bits, k_bits, v_bits, page_table, prefix_lens, num_q_heads,
                        num_kv_heads, block_len, mode, scale, rows):
        """Selected rows (b, i, h). Returns (out [n, D], lse [n])."""
        q = np.ascontiguousarray(q_bits, dtype=np.uint16)
        k = np.ascontiguousarray(k_bits, dtype=np.uint16)
        v = np.ascontiguousarray(v_bits, dtype=np.uint16)
        pt = np.ascontiguousarray(page_table, dtype=np.int32)
        pl = np.ascontiguousarray(prefix_lens, dtype=np.int32)
        r = np.ascontiguousarray(rows, dtype=np.int32).reshape(-1, 3)
        B, bl, Hq, D = q.shape
        num_pages, Hkv, P, _ = k.shape
        out = np.zeros((r.shape[0], D), dtype=np.float64)
        lse = np.zeros((r.shape[0],), dtype=np.float64)
        rc = self.lib.nldo_block_attn_rows(self._p(q), self._p(k), self._p(v), self._p(pt), self._p(pl),
                                           B, Hq, Hkv, D, P, num_pages, pt.shape[1], bl, int(mode),
                                           float(scale), r.shape[0], self._p(r), self._p(out), self._p(lse))
        if rc != 0:
            raise ValueError(f"oracle block_attn_rows failed: {rc}")
        return out, lse

    def combine(self, o_part, lse_part):
        """o_part [S, R, D], lse_part [S, R] -> (out [R, D], lse [R])."""
        o = np.ascontiguousarray(o_part, dtype=np.float64)
        l = np.ascontiguousarray(lse_part, dtype=np.float64)
        S, R, D = o.shape
        out = np.zeros((R, D), dtype=np.float64)
        lse = np.zeros((R,), dtype=np.float64)
        self.lib.nldo_combine(self._p(o), self._p(l), S, R, D, self._p(out), self._p(lse))
        return out, lse

    def accept(self, draft, verify):
        d = np.ascontiguousarray(draft, dtype=np.int32)
        v = np.ascontiguousarray(verify, dtype=np.int32)
        B, n = d.shape
        acc = np.zeros((B,), dtype=np.int32)
        self.lib.nldo_accept(self._p(d), self._p(v), B, n, self._p(acc))
        return acc

    def unmask(self, conf, k):
        c = np.ascontiguousarray(conf, dtype=np.float32)
        B, n = c.shape
        pos = np.zeros((B, k), dtype=np.int32)
        nsel = np.zeros((B,), dtype=np.int32)
        self.lib.nldo_unmask(self._p(c), B, n, int(k), self._p(pos), self._p(nsel))
        return pos, nsel

    def unmask_threshold(self, conf, threshold):
        """(positions [B, n] ascending then -1, num_selected [B]) of one
        threshold-unmasking step with the top-1 fallback."""
        c = np.ascontiguousarray(conf, dtype=np.float32)
        B, n = c.shape
        pos = np.zeros((B, n), dtype=np.int32)
        nsel = np.zeros((B,), dtype=np.int32)
        self.lib.nldo_unmask_threshold(self._p(c), B, n, float(np.float32(threshold)), self._p(pos), self._p(nsel))
        return pos, nsel

    def logits_argmax(self, logits_bits, vocab=None):
        """(ids [rows] int32, conf [rows] fp64) of bf16 logits [rows, ld] (bit
        patterns as uint16); the first `vocab` columns are used (default: all)."""
        lb = np.ascontiguousarray(logits_bits, dtype=np.uint16)
        rows, ld = lb.shape
        vocab = ld if vocab is None else int(vocab)
        ids = np.zeros((rows,), dtype=np.int32)
        conf = np.zeros((rows,), dtype=np.float64)
        self.lib.nldo_logits_argmax(self._p(lb), rows, vocab, ld, self._p(ids), self._p(conf))
        return ids, conf

    def ensemble_argmax(self, ar_bits, diff_bits, lam, vocab=None):
        """(ids [rows] int32, conf [rows] fp64) of lam * softmax(ar) + (1 - lam) * softmax(diff)."""
        a = np.ascontiguousarray(ar_bits, dtype=np.uint16)
        d = np.ascontiguousarray(diff_bits, dtype=np.uint16)
        rows, ld = a.shape
        vocab = ld if vocab is None else int(vocab)
        ids = np.zeros((rows,), dtype=np.int32)
        conf = np.zeros((rows,), dtype=np.float64)
        self.lib.nldo_ensemble_argmax(self._p(a), self._p(d), rows, vocab, ld, float(lam), self._p(ids), self._p(conf))
        return ids, conf

    def quadss_mask(self, k):
        """uint32 [1 + k + k^2] block masks of quadratic self-speculation (bit j: slot j visible)."""
        out = np.zeros((32,), dtype=np.uint32)
        n = self.lib.nldo_quadss_mask(int(k), self._p(out))
        if n < 0:
            raise ValueError(f"k={k}: block of 1 + k + k^2 slots exceeds 32")
        return out[:n].copy()

    def block_attn_masked(self, q_bits, k_bits, v_bits, page_table, prefix_lens, num_q_heads, num_kv_heads,
                          block_len, block_mask, scale, want_probs=False):
        """Block attention whose block part follows block_mask (uint32 [bl]);
        (out [B, bl, Hq, D], lse [B, Hq, bl], probs or None) in fp64."""
        q = np.ascontiguousarray(q_bits, dtype=np.uint16)
        k = np.ascontiguousarray(k_bits, dtype=np.uint16)
        v = np.ascontiguousarray(v_bits, dtype=np.uint16)
        table = np.ascontiguousarray(page_table, dtype=np.int32)
        pl = np.ascontiguousarray(prefix_lens, dtype=np.int32)
        bm = np.ascontiguousarray(block_mask, dtype=np.uint32)
        B, bl, Hq, D = q.shape
        num_pages, Hkv, P, _ = k.shape
        out = np.zeros((B, bl, Hq, D), dtype=np.float64)
        lse = np.zeros((B, Hq, bl), dtype=np.float64)
        stride = int(pl.max() + bl) if B else 1
        probs = np.zeros((B, Hq, bl, stride), dtype=np.float64) if want_probs else None
        rc = self.lib.nldo_block_attn_masked(self._p(q), self._p(k), self._p(v), self._p(table), self._p(pl),
                                             B, Hq, Hkv, D, P, num_pages, table.shape[1], bl, self._p(bm),
                                             float(scale), self._p(out), self._p(lse), self._p(probs), stride)
        if rc != 0:
            raise RuntimeError(f"nldo_block_attn_masked failed ({rc})")
        return out, lse, probs

    def kv_commit(self, k_new_bits, v_new_bits, counts, page_table, prefix_lens, k_bits, v_bits, advance):
        """Commit rows of a [B, bl, Hkv, D] K/V block into copies of the page
        pools; returns (k_pages, v_pages, prefix_lens) after the commit."""
        kn = np.ascontiguousarray(k_new_bits, dtype=np.uint16)
        vn = np.ascontiguousarray(v_new_bits, dtype=np.uint16)
        B, bl, Hkv, D = kn.shape
        kp = np.array(k_bits, dtype=np.uint16, copy=True, order="C")
        vp = np.array(v_bits, dtype=np.uint16, copy=True, order="C")
        P = kp.shape[2]
        table = np.ascontiguousarray(page_table, dtype=np.int32)
        pl = np.array(prefix_lens, dtype=np.int32, copy=True)
        cnt = None if counts is None else np.ascontiguousarray(counts, dtype=np.int32)
        self.lib.nldo_kv_commit(self._p(kn), self._p(vn), self._p(cnt), self._p(table), self._p(pl), int(bool(advance)),
                                self._p(kp), self._p(vp), B, Hkv, D, P, kp.shape[0], table.shape[1], bl)
        return kp, vp, pl

    def greedy_accept(self, pred, target, conf):
        """(positions [B, n] ascending then -1, num_selected [B]) of one greedy
        parallel acceptance iteration."""
        p = np.ascontiguousarray(pred, dtype=np.int32)
        t = np.ascontiguousarray(target, dtype=np.int32)
        c = np.ascontiguousarray(conf, dtype=np.float32)
        B, n = c.shape
        pos = np.zeros((B, n), dtype=np.int32)
        nsel = np.zeros((B,), dtype=np.int32)
        self.lib.nldo_greedy_accept(self._p(p), self._p(t), self._p(c), B, n, self._p(pos), self._p(nsel))
        return pos, nsel


def load(lib_path: Optional[str] = None) -> Oracle:
    """The default oracle (compiled on first use), or one from ``lib_path``."""
    global _default
    if lib_path is not None:
        return Oracle(lib_path)
    with _lock:
        if _default is None:
            if (not os.path.exists(LIB_PATH)
                    or os.path.getmtime(LIB_PATH) < os.path.getmtime(SOURCE)):
                compile_oracle()
            _default = Oracle(LIB_PATH)
    return _default
