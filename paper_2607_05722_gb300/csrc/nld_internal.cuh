// Internal declarations of libnld: kernel argument blocks, launch helpers and
// thin inline-PTX wrappers (mbarrier, TMA, ldmatrix, mma) used by the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "nld.h"

namespace nld {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kMaxSplits = 128;
constexpr int kMaxRows = 160;   // (Hq / Hkv) * block_len handled by one CTA
constexpr int kMaxBlock = 32;   // block_len and the decision width n
constexpr int kTileTok = 64;    // KV tokens per pipeline stage
constexpr int kGroupTok = 16;   // KV tokens per TMA box (never crosses a page: P % 16 == 0)

// Arguments of the block-attention kernel (one CTA per (split, kv head, sequence)).
struct AttnArgs {
  const __nv_bfloat16* q;      // [B, bl, Hq, D]
  const int32_t* page_table;   // [B, max_pages]
  const int32_t* prefix_lens;  // [B]
  __nv_bfloat16* out;          // [B, bl, Hq, D]       (unsplit)
  float* lse;                  // [B, Hq, bl] or null  (unsplit)
  float* o_part;               // [S, B, Hq, bl, D]    (split; null when unsplit)
  float* lse_part;             // [S, B, Hq, bl]
  unsigned int* err;           // device error word
  int B, Hq, Hkv, G, bl, R;    // R = G * bl query rows per CTA
  int page_size, log2_page, num_pages, max_pages;
  int num_splits, chunk;       // splits and tokens per split (multiple of 16)
  int mode, nstage, nwr;       // mask mode, pipeline depth, 16-row warp groups
  float scale_log2;            // softmax scale * log2(e)
};

// Launchers (defined next to their kernels). Return a CUDA error code.
cudaError_t launch_block_attn(const AttnArgs& a, const CUtensorMap& tmk, const CUtensorMap& tmv,
                              int head_dim, cudaStream_t stream);
cudaError_t launch_combine(const float* o_part, const float* lse_part, int S, int B, int Hq, int bl,
                           int D, __nv_bfloat16* out, float* lse, cudaStream_t stream);
cudaError_t launch_accept(const int32_t* draft, const int32_t* verify, int B, int n, int32_t* acc,
                          cudaStream_t stream);
cudaError_t launch_unmask(const float* conf, int B, int n, int k, int32_t* pos, int32_t* nsel,
                          cudaStream_t stream);

// Pipeline shape the attention launcher picks for R query rows (shared with
// the host-side checks so both agree).
struct AttnShape {
  int nwr;      // warps along rows (16 rows each)
  int nwt;      // warps along KV tokens of a tile
  int nstage;   // pipeline stages
  int threads;  // consumers + one producer warp
  size_t smem;  // dynamic shared memory bytes
};
AttnShape attn_shape(int R, int head_dim);
size_t max_smem_bytes(int head_dim);

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait for an mbarrier phase with a time limit. On timeout, records
// NLD_DEVERR_WAIT_TIMEOUT and returns false instead of spinning forever.
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s: microsecond kernels never get near it
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, unsigned int* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 255u && global_timer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, NLD_DEVERR_WAIT_TIMEOUT);
      return false;
    }
  }
}

// 4-D tiled TMA load into shared memory, completing on an mbarrier.
__device__ __forceinline__ void tma_load_4d(void* dst, const CUtensorMap* map, uint64_t* bar, int c0, int c1,
                                            int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D += A * B for one m16n8k16 bf16 tile with fp32 accumulators.
__device__ __forceinline__ void mma_16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Hardware base-2 exponential (MUFU.EX2): ex2(-inf) = +0.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Hardware base-2 logarithm (MUFU.LG2).
__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void named_bar_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

}  // namespace nld
