// Internal declarations of libnld: kernel argument blocks, launch helpers and
// thin inline-PTX wrappers (mbarrier, TMA, clusters, tcgen05) used by the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "nld.h"

namespace nld {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kMaxSplits = 128;
constexpr int kModeBlockMask = 2;  // block part of the mask from a per-row table
constexpr int kMaxRows = 256;   // (Hq / Hkv) * block_len handled by one CTA (two 128-row M tiles)
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
  __nv_bfloat16* o_part;       // [S, B, Hq, bl, D]    (split; null when unsplit), each row normalised
  float* lse_part;             // [S, B, Hq, bl]
  unsigned int* err;           // device error word
  unsigned long long* rescales;  // running-max rescale events (diagnostic counter)
  int B, Hq, Hkv, G, bl, R;    // R = G * bl_c query rows per CTA
  int nh, bl_c;                // block-slot chunks per (split, KV head, sequence) (1 or 2), slots per chunk
  int page_size, log2_page, num_pages, max_pages;
  int num_splits, chunk;       // splits and tokens per split (multiple of 16)
  int mode;                    // NLD_MODE_DIFFUSION, NLD_MODE_VERIFY or kModeBlockMask
  const uint32_t* block_mask;  // [bl] row masks over the block slots (kModeBlockMask only)
  float scale_log2;            // softmax scale * log2(e)
  int prefix_ready;            // NLD_ATTN_PREFIX_READY: prefix K/V may be read before the dependency wait
  int order_by_length;         // CTA z takes the sequence of rank z by prefix length (longest first)
  int csize;                   // thread-block cluster size along the splits (1 = no cluster)
  int num_partials;            // partials written per (b, h, i): num_splits / csize (1 = final output)
};

// Launchers (defined next to their kernels). Return a CUDA error code.
// tcgen05 kernel: query rows R <= 256 (one or two 128-row MMA tiles).
bool tc_supports(int R, int head_dim);
// Tensor maps of one call: k/v the K/V page pools; q the query block and o
// the output or, with split partials, the partial rows (bf16 both), in
// boxes of one CTA's rows.
struct TmaMaps {
  CUtensorMap k, v, o, q;
};
cudaError_t launch_block_attn_tc(const AttnArgs& a, const TmaMaps& maps, int head_dim, cudaStream_t stream);
// The same for a table mask (a.mode == kModeBlockMask; block_attn_tc_masked.cu).
cudaError_t launch_block_attn_tc_masked(const AttnArgs& a, const TmaMaps& maps, int head_dim, cudaStream_t stream);
// A kernel whose one mbarrier wait can never complete (decide.cu).
cudaError_t launch_wait_timeout_check(uint64_t limit_ns, unsigned int* err, cudaStream_t stream);
cudaError_t launch_combine(const __nv_bfloat16* o_part, const float* lse_part, int S, int B, int Hq, int bl,
                           int D, __nv_bfloat16* out, float* lse, int sm_count, cudaStream_t stream);
cudaError_t launch_accept(const int32_t* draft, const int32_t* verify, int B, int n, int32_t* acc,
                          cudaStream_t stream);
cudaError_t launch_unmask(const float* conf, int B, int n, int k, int32_t* pos, int32_t* nsel,
                          cudaStream_t stream);
cudaError_t launch_unmask_threshold(const float* conf, int B, int n, float threshold, int32_t* pos, int32_t* nsel,
                                    cudaStream_t stream);
cudaError_t launch_greedy_accept(const int32_t* pred, const int32_t* target, const float* conf, int B, int n,
                                 int32_t* pos, int32_t* nsel, cudaStream_t stream);
// Logits -> (argmax, confidence): `split` CTAs per row (a cluster when > 1).
cudaError_t launch_logits_argmax(const __nv_bfloat16* logits, int rows, int vocab, long ld, int split, int32_t* ids,
                                 float* conf, unsigned int* err, cudaStream_t stream);
int logits_split_vectors();  // 16-byte vectors a CTA streams per ring stage
// AR-diffusion ensemble verifier: `split` CTAs per row pair (a cluster when > 1).
cudaError_t launch_ensemble_argmax(const __nv_bfloat16* ar, const __nv_bfloat16* diff, int rows, int vocab, long ld,
                                   int split, float lambda, int32_t* ids, float* conf, cudaStream_t stream);
// Block KV commit (rows j < count_b to slots L_b + j), then L_b += count_b.
cudaError_t launch_kv_commit(const __nv_bfloat16* k_new, const __nv_bfloat16* v_new, const int32_t* counts,
                             const int32_t* page_table, int32_t* prefix_lens, __nv_bfloat16* k_pages,
                             __nv_bfloat16* v_pages, int B, int Hkv, int D, int P, int num_pages, int max_pages,
                             int bl, bool advance, unsigned int* err, cudaStream_t stream);

// Launch with programmatic stream serialization: the kernel may start while
// its predecessor in the stream is still running. Every kernel of this
// library releases its dependents at its start (they can only launch once
// all of this grid's CTAs are resident, so none of them can be starved) and
// calls grid_dependency_wait() before it touches data an earlier kernel may
// produce, so launch latency and prologue (barrier setup, descriptor
// prefetch, and with NLD_ATTN_PREFIX_READY the prefix K/V stream) overlap
// the predecessor. Set NLD_DISABLE_PDL=1 to launch plainly.
bool pdl_enabled();

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel_cluster(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                                  int cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int n = 0;
  if (pdl_enabled()) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                          Args&&... args) {
  return launch_kernel_cluster(kern, grid, block, smem, stream, 1, std::forward<Args>(args)...);
}

// Resident clusters of `csize` CTAs of the tcgen05 attention kernel on the
// current device (cached), for the split plan.
int tc_max_active_clusters(int csize, int head_dim, int rows);

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------

// Wait until the grids this one depends on have completed and their memory
// is visible (no-op without a programmatic dependency).
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Allow the next grid in the stream to be scheduled.
__device__ __forceinline__ void grid_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

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

// Non-blocking test of an mbarrier phase.
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
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
__device__ __forceinline__ bool mbar_wait_for(uint64_t* bar, uint32_t parity, unsigned int* err,
                                              uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 255u && global_timer_ns() - t0 > limit_ns) {
      atomicOr(err, NLD_DEVERR_WAIT_TIMEOUT);
      return false;
    }
  }
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, unsigned int* err) {
  return mbar_wait_for(bar, parity, err, kWaitLimitNs);
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

// 3-D tiled TMA load into shared memory, completing on an mbarrier.
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar, int c0, int c1,
                                            int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// Hardware base-2 exponential (MUFU.EX2): ex2(-inf) = +0.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Three-input maximum (one instruction on sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Paired fp32 arithmetic (one f32x2 instruction for two lanes of work).
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.ftz.f32x2 rd, ra, rb, rc;\n\t"
      "mov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.ftz.f32x2 rd, ra, rb;\n\t"
      "mov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

// Hardware base-2 logarithm (MUFU.LG2).
__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Two bf16 values (low half first) widened exactly to fp32.
__device__ __forceinline__ void unpack_bf16(uint32_t w, float& lo, float& hi) {
  lo = __uint_as_float(w << 16);
  hi = __uint_as_float(w & 0xFFFF0000u);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void named_bar_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Arrive on a named barrier without waiting (the other `threads` - 32*k
// participants wait with named_bar_sync).
__device__ __forceinline__ void named_bar_arrive(int id, int threads) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// ---------------------------------------------------------------------------
// Thread-block clusters and distributed shared memory
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// Whole-cluster barrier (every thread of every CTA of the cluster), with
// release/acquire ordering of shared-memory writes across the cluster.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t dsmem_addr(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}

__device__ __forceinline__ float ld_dsmem_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ float4 ld_dsmem_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// ---------------------------------------------------------------------------
// tcgen05 (5th-generation tensor core) and tensor memory
// ---------------------------------------------------------------------------

// Bulk copy (TMA engine) of `bytes` from global to this CTA's shared memory,
// completing on an mbarrier (expect_tx set by the caller); both addresses
// 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(void* sdst, const void* gsrc, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(sdst)),
               "l"(gsrc), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// Bulk copy (TMA engine) of `bytes` from this CTA's shared memory to global
// memory; both addresses 16-byte aligned, bytes a multiple of 16. The issuing
// thread must call bulk_store_wait_read() before the source is overwritten or
// the CTA exits.
__device__ __forceinline__ void bulk_store(void* gdst, const void* ssrc, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n\t"
               "cp.async.bulk.commit_group;" ::"l"(gdst), "r"(smem_u32(ssrc)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_store_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }

// Tiled TMA stores shared -> global (one box at coordinates {c0, c1[, c2]},
// the innermost coordinate a multiple of 16 bytes), in the issuing thread's
// bulk group: close it with bulk_commit() and wait with bulk_store_wait_read()
// before the source is overwritten or the CTA exits.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1)
               : "memory");
}
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* src, int c0, int c1, int c2) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1), "r"(c2)
               : "memory");
}
__device__ __forceinline__ void tma_store_4d(const CUtensorMap* map, const void* src, int c0, int c1, int c2,
                                             int c3) {
  asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.bulk_group [%0, {%2, %3, %4, %5}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Allocate `ncols` TMEM columns (a power of two >= 32); the base address is
// written to shared memory. Executed by one whole warp.
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Shared-memory matrix descriptor for a 128-byte-swizzled operand tile:
// start address, leading-dimension and stride-dimension byte offsets (16-byte
// units), descriptor version 1, swizzle mode 2 (128 B).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// Instruction descriptor of tcgen05.mma kind::f16 with bf16 A and B and an
// fp32 accumulator: M x N tile, A K-major, B K-major or MN-major.
__host__ __device__ constexpr uint32_t umma_idesc_bf16(int M, int N, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
         (static_cast<uint32_t>(N >> 3) << 17) | (static_cast<uint32_t>(M >> 4) << 24);
}

// D(tmem) (+)= A(smem) * B(smem), issued by one thread.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on an mbarrier once every tcgen05 operation this thread issued has completed.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// Warp-collective: each lane reads 32 consecutive fp32 columns of its TMEM
// lane (lanes 32*(warp%4) .. +31), then waits for the load.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* out) {
  uint32_t r[32];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
               "tcgen05.wait::ld.sync.aligned;"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
               : "r"(taddr)
               : "memory");
#pragma unroll
  for (int j = 0; j < 32; ++j) out[j] = __uint_as_float(r[j]);
}

// Warp-collective: each lane reads 16 (or 64) consecutive fp32 columns of its
// TMEM lane in one load and waits once.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* out) {
  uint32_t r[16];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];\n\t"
               "tcgen05.wait::ld.sync.aligned;"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
               : "r"(taddr)
               : "memory");
#pragma unroll
  for (int j = 0; j < 16; ++j) out[j] = __uint_as_float(r[j]);
}

__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float* out) {
  uint32_t r[64];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%64];\n\t"
               "tcgen05.wait::ld.sync.aligned;"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
               : "r"(taddr)
               : "memory");
#pragma unroll
  for (int j = 0; j < 64; ++j) out[j] = __uint_as_float(r[j]);
}

// Warp-collective: each lane writes 32 consecutive fp32 columns of its TMEM lane and waits.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float* in) {
  uint32_t r[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) r[j] = __float_as_uint(in[j]);
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};\n\t"
               "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
               : "memory");
}

// Warp-collective TMEM stores of packed 32-bit words (each lane: N
// consecutive columns of its TMEM lane); the caller waits with tmem_wait_st().
template <int N>
__device__ __forceinline__ void tmem_st_u32(uint32_t taddr, const uint32_t* r);
template <>
__device__ __forceinline__ void tmem_st_u32<8>(uint32_t taddr, const uint32_t* r) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
               : "memory");
}
template <>
__device__ __forceinline__ void tmem_st_u32<16>(uint32_t taddr, const uint32_t* r) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
               : "memory");
}
template <>
__device__ __forceinline__ void tmem_st_u32<32>(uint32_t taddr, const uint32_t* r) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
               : "memory");
}
template <int N>
__device__ __forceinline__ void tmem_st_zero(uint32_t taddr) {
  uint32_t z[N];
#pragma unroll
  for (int i = 0; i < N; ++i) z[i] = 0u;
  tmem_st_u32<N>(taddr, z);
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// D(tmem) (+)= A(tmem) * B(smem), issued by one thread. A: M = 128 rows in
// TMEM lanes 0..127, K = 16 bf16 values per row packed two to a column (8
// columns from a_tmem).
__device__ __forceinline__ void umma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                             uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// ---------------------------------------------------------------------------
// K/V tile staging shared by the attention kernels
// ---------------------------------------------------------------------------

// A stage holds the K tile then the V tile of 64 tokens; each is D/64 column
// blocks of 64 tokens x 128 bytes, written by TMA with the 128-byte swizzle
// (chunk c of row r at chunk position c ^ (r % 8) within each 1024-byte atom).
template <int D>
struct TileGeom {
  static constexpr int kColBlocks = D / 64;
  static constexpr int kColBlockBytes = kTileTok * 128;
  static constexpr int kTileBytes = kColBlocks * kColBlockBytes;
  static constexpr int kStageBytes = 2 * kTileBytes;
};

// Byte offset of (token r, 16-byte chunk c) inside a K or V tile.
__device__ __forceinline__ uint32_t kv_swz(int r, int c) {
  return static_cast<uint32_t>((c >> 3) * (kTileTok * 128) + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

// Page id of each 16-token group of a split, loaded ahead: lane j of the
// producer warp holds group j of a batch of 32 groups (8 tiles). The load
// does not depend on the prefix length (the index is clamped into the table
// row), so it can be issued before the length is known; validate() then
// marks groups past the split end as out of the pool (TMA zero fill) and
// clamps corrupt ids into range, flagging them.
struct PagePrefetch {
  int raw;
  __device__ __forceinline__ void load(const AttnArgs& a, int b, int t_begin, int batch, int lane) {
    const int t = t_begin + (batch * 32 + lane) * kGroupTok;
    const int lp = min(t >> a.log2_page, a.max_pages - 1);
    raw = __ldg(a.page_table + static_cast<size_t>(b) * a.max_pages + lp);
  }
  __device__ __forceinline__ int validate(const AttnArgs& a, int t_begin, int t_end, int batch, int lane) const {
    const int t = t_begin + (batch * 32 + lane) * kGroupTok;
    if (t >= t_end) return a.num_pages;
    if (raw < 0 || raw >= a.num_pages) {
      atomicOr(a.err, NLD_DEVERR_PAGE_RANGE);
      return min(max(raw, 0), a.num_pages - 1);
    }
    return raw;
  }
};

// Producer warp `pw` of `nprod`: streams its share of the TMA boxes of the
// K/V tiles of tokens [t_begin, t_end) of (sequence b, KV head g) into an
// nstage ring: K tiles at [column block][stage], so that the K of
// consecutive stages is contiguous per column block, then V tiles at
// [stage][column block]. A tile has 4 groups x D/64 column blocks x {K, V} boxes
// (16 tokens x 64 dims each); they are dealt to the producer warps in equal
// shares and, within a warp, one box per lane: the first half of the warps
// load K, the second half V. With kSplit, K and V slots fill and free on
// their own barriers (k_full/v_full, k_empty/v_empty), so a K slot is
// refilled as soon as the score product that read it has completed, before
// the PV product frees the V slot of the same tile; without it a stage's K
// and V fill on k_full and free on k_empty together. TMA issue cost is per
// warp, so more producer warps land a tile sooner. A warp's expect_tx covers
// only its own boxes, so a full barrier expects one arrival per warp (of its
// kind, with kSplit). `first` holds the page ids of the first 32 groups,
// already loaded. With kSplit the `early_tiles` leading tiles issued before
// the dependency wait go out K first: the V warps wait at a named barrier
// until the K warps have issued the early K boxes, so the first score
// products' operands are not queued behind V boxes that only the later PV
// products read. Returns tiles issued.
template <int D, bool kSplit>
__device__ __forceinline__ int produce_kv(const AttnArgs& a, const CUtensorMap* tmk, const CUtensorMap* tmv,
                                          uint8_t* stages, uint64_t* k_full, uint64_t* v_full, uint64_t* k_empty,
                                          uint64_t* v_empty, int nstage, int g, int b, int t_begin, int t_end,
                                          int ntiles, int lane, int pw, int nprod, const PagePrefetch& first,
                                          int early_tiles) {
  using Geo = TileGeom<D>;
  constexpr int kGroups = kTileTok / kGroupTok;
  constexpr int kOpsPerTile = kGroups * 2 * Geo::kColBlocks;  // 16 (D=128) or 8 (D=64)
  const int my_ops = kOpsPerTile / nprod;                     // nprod divides kOpsPerTile (and its halves)
  const bool warp_v = pw >= nprod / 2;                        // this warp's boxes are all V (else all K)
  uint64_t* full = kSplit && warp_v ? v_full : k_full;
  uint64_t* empty = kSplit && warp_v ? v_empty : k_empty;
  const uint32_t bytes = static_cast<uint32_t>(my_ops) * kGroupTok * 128;
  int page_cur = first.validate(a, t_begin, t_end, 0, lane);
  PagePrefetch nxt;
  nxt.raw = 0;
  if (ntiles > 8) nxt.load(a, b, t_begin, 1, lane);
  int issued = 0;
  // Named barrier 4: the nprod producer warps, once, before any wait of the
  // loop (early_tiles <= nstage, so the K warps reach their arrival without
  // waiting on a slot).
  constexpr int kKFirstBar = 4;
  if (kSplit && warp_v && early_tiles > 0) named_bar_sync(kKFirstBar, 32 * nprod);
  for (int k = 0; k < ntiles; ++k) {
    const int st = k % nstage;
    // The first `early_tiles` tiles hold prefix tokens only and may be issued
    // before the dependency wait (NLD_ATTN_PREFIX_READY); the rest wait.
    if (k == early_tiles && early_tiles > 0) grid_dependency_wait();
    if (k >= nstage) {
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&empty[st], ((k / nstage) - 1) & 1, a.err) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
    }
    if (k > 0 && (k & 7) == 0) {
      const int batch = k >> 3;
      page_cur = nxt.validate(a, t_begin, t_end, batch, lane);
      if ((k + 8) < ntiles) nxt.load(a, b, t_begin, batch + 1, lane);
    }
    if (lane == 0) mbar_arrive_expect_tx(&full[st], bytes);
    __syncwarp();
    // op -> (group, kind, column block): group fastest, so a warp's boxes
    // spread over the tile's pages.
    const int op = pw * my_ops + (lane < my_ops ? lane : 0);
    const int grp = op % kGroups;
    const int kind_cb = op / kGroups;  // 0 .. 2*kColBlocks-1
    const bool is_v = kind_cb >= Geo::kColBlocks;
    const int cb = kind_cb % Geo::kColBlocks;
    const int page = __shfl_sync(0xffffffffu, page_cur, ((k & 7) * kGroups + grp) & 31);
    if (lane < my_ops) {
      const int t = t_begin + k * kTileTok + grp * kGroupTok;
      const int slot = page < a.num_pages ? (t & (a.page_size - 1)) : 0;
      uint8_t* dst = (is_v ? stages + (nstage + st) * Geo::kTileBytes + cb * Geo::kColBlockBytes
                           : stages + (cb * nstage + st) * Geo::kColBlockBytes) +
                     grp * kGroupTok * 128;
      tma_load_4d(dst, is_v ? tmv : tmk, &full[st], cb * 64, slot, g, page);
    }
    issued = k + 1;
    if (kSplit && !warp_v && k == early_tiles - 1) named_bar_arrive(kKFirstBar, 32 * nprod);
  }
  return issued;
}

}  // namespace nld
