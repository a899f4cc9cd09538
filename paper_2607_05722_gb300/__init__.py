"""GB300-native (sm_103a) block attention over a paged bf16 KV cache, fused
with the token decisions of tri-mode decoding (diffusion draft, AR verify,
longest-prefix acceptance, confidence-ranked unmasking).

Modules:
  build      compiles csrc/*.cu into _build/libnld.so (nvcc, sm_103a)
  nld        ctypes binding of the C ABI declared in include/nld.h
  workloads  seeded synthetic inputs shaped like the paper's workloads
"""
__all__ = ["build", "nld", "workloads"]
