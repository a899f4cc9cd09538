// C ABI of libnld (include/nld.h): host-side argument checks, KV split choice,
// TMA descriptor encoding and kernel launches. Nothing here allocates device
// memory or synchronises, except nld_device_error().
#include <climits>
#include <math.h>
#include <stdio.h>
#include <stdlib.h>

#include <mutex>

#include "nld_internal.cuh"

namespace {

using nld::AttnArgs;

// Error word the kernels OR their NLD_DEVERR_* bits into, and the count of
// running-max rescales (a diagnostic).
__device__ unsigned int g_device_error;
__device__ unsigned long long g_rescale_count;

constexpr int kMaxDevices = 64;
unsigned int* g_err_ptr[kMaxDevices];
unsigned long long* g_rescale_ptr[kMaxDevices];
int g_sm_count[kMaxDevices];
std::mutex g_mu;

bool aligned(const void* p, size_t a) { return p != nullptr && (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Per-device state: addresses of the error word and the rescale counter and
// the SM count, looked up once.
nld_status_t device_state(unsigned int** err, int* sms, unsigned long long** rescales = nullptr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return NLD_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_err_ptr[dev] == nullptr) {
    void* p = nullptr;
    void* c = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) return NLD_ERR_CUDA;
    if (cudaGetSymbolAddress(&c, g_rescale_count) != cudaSuccess) return NLD_ERR_CUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return NLD_ERR_CUDA;
    g_sm_count[dev] = n;
    g_rescale_ptr[dev] = static_cast<unsigned long long*>(c);
    g_err_ptr[dev] = static_cast<unsigned int*>(p);
  }
  if (err) *err = g_err_ptr[dev];
  if (sms) *sms = g_sm_count[dev];
  if (rescales) *rescales = g_rescale_ptr[dev];
  return NLD_OK;
}

bool is_pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }

nld_status_t check_params(const nld_attn_params_t* p, int block_len) {
  if (p == nullptr) return NLD_ERR_INVALID_ARG;
  if (p->batch < 1 || p->num_q_heads < 1 || p->num_kv_heads < 1 || p->num_pages < 1 ||
      p->max_pages_per_seq < 1 || p->num_splits < 0 || p->softmax_scale < 0.f || !isfinite(p->softmax_scale))
    return NLD_ERR_INVALID_ARG;
  if (p->num_q_heads % p->num_kv_heads != 0) return NLD_ERR_INVALID_ARG;
  if (p->flags & ~(NLD_ATTN_PREFIX_READY | NLD_ATTN_NO_CLUSTER))
    return NLD_ERR_INVALID_ARG;
  if (block_len < 1 || block_len > nld::kMaxBlock) return NLD_ERR_INVALID_ARG;
  if (p->num_splits > nld::kMaxSplits) return NLD_ERR_INVALID_ARG;
  if (!is_pow2(p->page_size) || p->page_size < 16 || p->page_size > 256) return NLD_ERR_INVALID_ARG;
  if (p->batch > 65535 || p->num_kv_heads > 65535) return NLD_ERR_UNSUPPORTED;
  if (p->head_dim != 64 && p->head_dim != 128) return NLD_ERR_UNSUPPORTED;
  if ((p->num_q_heads / p->num_kv_heads) * block_len > nld::kMaxRows) return NLD_ERR_UNSUPPORTED;
  // logical token positions must fit in int
  if (static_cast<long long>(p->max_pages_per_seq) * p->page_size > (1ll << 30)) return NLD_ERR_UNSUPPORTED;
  if (static_cast<long long>(p->max_pages_per_seq) * p->page_size < block_len) return NLD_ERR_INVALID_ARG;
  return NLD_OK;
}

// Split plan: S splits of `chunk` tokens (a multiple of 16) over the longest
// possible sequence, max_pages_per_seq * page_size tokens. Splits past a
// shorter sequence's end do no work. With num_splits = 0 the count is
// chosen so that (splits x sequences x KV heads) covers the SMs once.
// On the tcgen05 kernel the splits of a (sequence, KV head) can run as one
// thread-block cluster that merges its results on chip and writes the final
// output, so no workspace and no combine launch are needed. An automatic plan
// takes floor(SMs / units) splits (one wave) and, when that is 2..8, rounds
// it down to 2, 4 or 8 and uses one cluster per unit if those clusters are
// resident at once. An explicit split count of 2, 4 or 8 uses one cluster; a
// larger count divisible by 8, 4 or 2 uses clusters of that size, leaving
// one partial per cluster for the combine.
constexpr long long kMaxAutoChunk = 2048;  // tokens per piece in an automatic plan (1 MiB of K+V at D=128)

struct SplitPlan {
  int splits;    // CTAs along the KV range per (sequence, KV head)
  int chunk;     // tokens per split
  int csize;     // cluster size (1 = none)
  int partials;  // splits / csize
  int nh;        // block-slot chunks: CTAs per (split, sequence, KV head) (1 or 2)
};

// 129..256 packed rows with an even block length run as two CTAs per
// (split, sequence, KV head), each with half of the block slots (at most 128
// rows: one M tile); the pair streams the same K/V tiles at the same time,
// so the second read is served by L2. An odd block length keeps one CTA with
// two M tiles.
int slot_chunks(int rows, int block_len) { return rows > 128 && block_len % 2 == 0 ? 2 : 1; }

// Longest split that still runs paired score products at both head sizes
// (the ring holds at least 6 tiles at head_dim 128).
constexpr long long kPairedChunk = 384;

// The plan for `sms` SMs; `clusters_resident(cs)` says how many clusters of
// cs CTAs can be resident at once (0: none considered).
template <typename ClustersResident>
void plan_splits_for(const nld_attn_params_t* p, int block_len, int sms, ClustersResident clusters_resident,
                     SplitPlan* out) {
  const long long max_tokens = static_cast<long long>(p->max_pages_per_seq) * p->page_size;
  const int rows = (p->num_q_heads / p->num_kv_heads) * block_len;
  const int nh = slot_chunks(rows, block_len);
  const long long units = static_cast<long long>(p->batch) * p->num_kv_heads * nh;  // CTAs per split
  const bool tc = nld::tc_supports(rows, p->head_dim);
  const bool clusters = tc && nh == 1 && !(p->flags & NLD_ATTN_NO_CLUSTER);
  const bool automatic = p->num_splits == 0;
  int want = p->num_splits;
  int csize = 1;
  if (automatic) {
    // Fill the SMs once; when the (sequence, KV head) units fit in one wave,
    // also cut long ranges into pieces of at most kMaxAutoChunk tokens: with
    // ragged lengths (not known on the host) the longest sequence would
    // otherwise set the time; pieces past a shorter sequence's end exit at
    // once. With more units than SMs the hardware scheduler balances them.
    long long s = sms / units;
    if (units < sms) {  // a single wave: the longest range would set the time
      const long long by_chunk = (max_tokens + kMaxAutoChunk - 1) / kMaxAutoChunk;
      if (s < by_chunk) s = by_chunk;
    }
    const long long by_tiles = (max_tokens + nld::kTileTok - 1) / nld::kTileTok;  // >= one tile per split
    if (s > by_tiles) s = by_tiles;
    if (s > nld::kMaxSplits) s = nld::kMaxSplits;
    if (s < 1) s = 1;
    want = static_cast<int>(s);
    if (clusters && want >= 2 && want <= 8) {
      const int cs = want >= 8 ? 8 : want >= 4 ? 4 : 2;
      if (units <= clusters_resident(cs)) {
        want = cs;
        csize = cs;
      }
    }
  } else if (clusters && want >= 2) {
    for (int cs = 8; cs >= 2; cs >>= 1)
      if (want % cs == 0) {
        csize = cs;
        break;
      }
  }
  long long chunk = (max_tokens + want - 1) / want;
  chunk = (chunk + nld::kGroupTok - 1) / nld::kGroupTok * nld::kGroupTok;
  if (automatic && csize == 1 && tc && chunk <= kPairedChunk) {
    // Splits short enough for paired score products take whole pairs (128
    // tokens) when that keeps at least 85% of the splits: no half-filled
    // product or tile in every CTA (8B shape: 19 splits of 224 tokens become
    // 17 of 256, measured faster).
    const long long c2 = (chunk + 2 * nld::kTileTok - 1) / (2 * nld::kTileTok) * (2 * nld::kTileTok);
    const long long s2 = (max_tokens + c2 - 1) / c2;
    if (s2 * 100 >= static_cast<long long>(want) * 85) chunk = c2;
  } else if (automatic && csize == 1 && tc) {
    // Streaming splits end on a whole tile when that keeps their number.
    const long long c1 = (chunk + nld::kTileTok - 1) / nld::kTileTok * nld::kTileTok;
    if ((max_tokens + c1 - 1) / c1 == (max_tokens + chunk - 1) / chunk) chunk = c1;
  }
  long long splits = (max_tokens + chunk - 1) / chunk;
  splits = (splits + csize - 1) / csize * csize;  // trailing empty splits complete a cluster
  out->chunk = static_cast<int>(chunk);
  out->splits = static_cast<int>(splits);
  out->csize = csize;
  out->partials = static_cast<int>(splits / csize);
  out->nh = nh;
}

nld_status_t plan_splits(const nld_attn_params_t* p, int block_len, SplitPlan* out) {
  int sms = 0;
  if (p->num_splits == 0) {
    nld_status_t st = device_state(nullptr, &sms);
    if (st != NLD_OK) return st;
  }
  const int rows = (p->num_q_heads / p->num_kv_heads) * block_len;
  plan_splits_for(
      p, block_len, sms, [&](int cs) { return static_cast<long long>(nld::tc_max_active_clusters(cs, p->head_dim, rows)); },
      out);
  return NLD_OK;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

size_t partial_o_bytes(const nld_attn_params_t* p, int block_len, int splits) {
  return static_cast<size_t>(splits) * p->batch * p->num_q_heads * block_len * p->head_dim * sizeof(__nv_bfloat16);
}
size_t partial_lse_bytes(const nld_attn_params_t* p, int block_len, int splits) {
  return static_cast<size_t>(splits) * p->batch * p->num_q_heads * block_len * sizeof(float);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(f);
  });
  return fn;
}

// 4-D map over a page pool [num_pages, Hkv, P, D] (innermost first: D, P, Hkv,
// pages); one box is 64 dims x 16 tokens of one (page, KV head), stored with
// the 128-byte swizzle. Boxes past num_pages read as zeros.
nld_status_t encode_pool_map(CUtensorMap* map, const void* base, const nld_attn_params_t* p) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return NLD_ERR_CUDA;
  const cuuint64_t D = static_cast<cuuint64_t>(p->head_dim);
  cuuint64_t dims[4] = {D, static_cast<cuuint64_t>(p->page_size), static_cast<cuuint64_t>(p->num_kv_heads),
                        static_cast<cuuint64_t>(p->num_pages)};
  cuuint64_t strides[3] = {D * 2, D * 2 * p->page_size, D * 2 * p->page_size * p->num_kv_heads};
  cuuint32_t box[4] = {64, static_cast<cuuint32_t>(nld::kGroupTok), 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? NLD_OK : NLD_ERR_CUDA;
}

// Map over a [B, bl, Hq, D] bf16 block (queries or output) whose box is one
// CTA's R = G * bl rows of 64 dims (G heads x bl slots), 128-byte swizzle.
nld_status_t encode_block_map(CUtensorMap* map, const void* base, const nld::AttnArgs& a, int D) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return NLD_ERR_CUDA;
  cuuint32_t estr[3] = {1, 1, 1};
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(a.Hq), static_cast<cuuint64_t>(a.B) * a.bl};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(D) * 2 * a.Hq};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(a.G), static_cast<cuuint32_t>(a.bl_c)};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? NLD_OK : NLD_ERR_CUDA;
}

// Map for the tiled output stores of one CTA's R = G * bl rows, 128-byte
// swizzle, rows in packed order (block slot major), box 64 dims x G heads x
// bl slots, bf16. Final output [B, bl, Hq, D]. Split partials [partials * B,
// Hq, bl, D]: the map walks dims, heads (stride bl * D), block slots (stride
// D), then (partial, sequence).
nld_status_t encode_out_map(CUtensorMap* map, const nld::AttnArgs& a, int D) {
  if (a.o_part == nullptr) return encode_block_map(map, a.out, a, D);
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return NLD_ERR_CUDA;
  const long long units = static_cast<long long>(a.num_partials) * a.B;
  if (units > INT_MAX) return NLD_ERR_UNSUPPORTED;  // coordinates are int
  const cuuint64_t row = static_cast<cuuint64_t>(D) * 2;
  cuuint32_t estr[4] = {1, 1, 1, 1};
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(a.Hq), static_cast<cuuint64_t>(a.bl),
                        static_cast<cuuint64_t>(units)};
  cuuint64_t strides[3] = {row * a.bl, row, row * a.bl * a.Hq};
  cuuint32_t box[4] = {64, static_cast<cuuint32_t>(a.G), static_cast<cuuint32_t>(a.bl_c), 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, a.o_part, dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? NLD_OK : NLD_ERR_CUDA;
}

}  // namespace

namespace nld {
bool pdl_enabled() {
  static const bool on = [] {
    const char* v = getenv("NLD_DISABLE_PDL");
    return !(v != nullptr && v[0] == '1');
  }();
  return on;
}
}  // namespace nld

extern "C" {

const char* nld_status_string(nld_status_t s) {
  switch (s) {
    case NLD_OK: return "NLD_OK";
    case NLD_ERR_INVALID_ARG: return "NLD_ERR_INVALID_ARG";
    case NLD_ERR_UNSUPPORTED: return "NLD_ERR_UNSUPPORTED";
    case NLD_ERR_WORKSPACE: return "NLD_ERR_WORKSPACE";
    case NLD_ERR_CUDA: return "NLD_ERR_CUDA";
  }
  return "NLD_ERR_UNKNOWN";
}

int nld_block_attn_plan(const nld_attn_params_t* params, int block_len, int sm_count, int32_t plan[4]) {
  if (plan == nullptr || sm_count < 1) return -1;
  if (check_params(params, block_len) != NLD_OK) return -1;
  SplitPlan sp;
  plan_splits_for(params, block_len, sm_count, [](int) { return 0LL; }, &sp);
  plan[0] = sp.splits;
  plan[1] = sp.chunk;
  plan[2] = sp.csize;
  plan[3] = sp.partials;
  return 0;
}

int nld_block_attn_num_splits(const nld_attn_params_t* params, int block_len) {
  if (check_params(params, block_len) != NLD_OK) return -1;
  SplitPlan plan;
  if (plan_splits(params, block_len, &plan) != NLD_OK) return -1;
  return plan.partials;
}

int nld_block_attn_kernels(const nld_attn_params_t* params, int block_len) {
  if (check_params(params, block_len) != NLD_OK) return -1;
  SplitPlan plan;
  if (plan_splits(params, block_len, &plan) != NLD_OK) return -1;
  return plan.partials <= 1 ? 1 : 2;
}

size_t nld_block_attn_workspace_size(const nld_attn_params_t* params, int block_len) {
  if (check_params(params, block_len) != NLD_OK) return static_cast<size_t>(-1);
  SplitPlan plan;
  if (plan_splits(params, block_len, &plan) != NLD_OK) return static_cast<size_t>(-1);
  if (plan.partials == 1) return 0;
  return align256(partial_o_bytes(params, block_len, plan.partials)) +
         partial_lse_bytes(params, block_len, plan.partials);
}

}  // extern "C"

namespace {

nld_status_t block_attn_impl(const nld_attn_params_t* params, const void* q_block, const void* k_pages,
                             const void* v_pages, const int32_t* page_table, const int32_t* prefix_lens,
                             int block_len, int mode, const uint32_t* block_mask, void* out, float* lse,
                             void* workspace, size_t workspace_bytes, bool run_combine, cudaStream_t stream) {
  nld_status_t st = check_params(params, block_len);
  if (st != NLD_OK) return st;
  if (mode != NLD_MODE_DIFFUSION && mode != NLD_MODE_VERIFY && mode != nld::kModeBlockMask)
    return NLD_ERR_INVALID_ARG;
  if (mode == nld::kModeBlockMask && !aligned(block_mask, 4)) return NLD_ERR_INVALID_ARG;
  if (!aligned(q_block, 16) || !aligned(k_pages, 16) || !aligned(v_pages, 16) || !aligned(out, 16) ||
      !aligned(page_table, 4) || !aligned(prefix_lens, 4))
    return NLD_ERR_INVALID_ARG;
  if (lse != nullptr && !aligned(lse, 4)) return NLD_ERR_INVALID_ARG;
  SplitPlan plan;
  st = plan_splits(params, block_len, &plan);
  if (st != NLD_OK) return st;
  size_t o_bytes = 0;
  if (plan.partials > 1) {
    o_bytes = align256(partial_o_bytes(params, block_len, plan.partials));
    const size_t need = o_bytes + partial_lse_bytes(params, block_len, plan.partials);
    if (workspace == nullptr || workspace_bytes < need) return NLD_ERR_WORKSPACE;
    if (!aligned(workspace, 16)) return NLD_ERR_INVALID_ARG;
  }
  unsigned int* err = nullptr;
  unsigned long long* rescales = nullptr;
  st = device_state(&err, nullptr, &rescales);
  if (st != NLD_OK) return st;

  nld::TmaMaps maps;
  if ((st = encode_pool_map(&maps.k, k_pages, params)) != NLD_OK) return st;
  if ((st = encode_pool_map(&maps.v, v_pages, params)) != NLD_OK) return st;

  const int G = params->num_q_heads / params->num_kv_heads;
  const float scale = params->softmax_scale > 0.f ? params->softmax_scale : 1.0f / sqrtf((float)params->head_dim);
  AttnArgs a{};
  a.q = static_cast<const __nv_bfloat16*>(q_block);
  a.page_table = page_table;
  a.prefix_lens = prefix_lens;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.lse = lse;
  a.err = err;
  a.rescales = rescales;
  a.B = params->batch;
  a.Hq = params->num_q_heads;
  a.Hkv = params->num_kv_heads;
  a.G = G;
  a.bl = block_len;
  a.nh = plan.nh;
  a.bl_c = block_len / plan.nh;
  a.R = G * a.bl_c;
  a.page_size = params->page_size;
  a.log2_page = __builtin_ctz(static_cast<unsigned>(params->page_size));
  a.num_pages = params->num_pages;
  a.max_pages = params->max_pages_per_seq;
  a.num_splits = plan.splits;
  a.chunk = plan.chunk;
  a.csize = plan.csize;
  a.num_partials = plan.partials;
  a.mode = mode;
  a.block_mask = mode == nld::kModeBlockMask ? block_mask : nullptr;
  a.scale_log2 = scale * nld::kLog2e;
  a.prefix_ready = (params->flags & NLD_ATTN_PREFIX_READY) ? 1 : 0;
  {
    // Longest sequences first when one split each leaves more units than SMs
    // (several waves): the last wave then holds the short sequences.
    int sms = 0;
    if ((st = device_state(nullptr, &sms)) != NLD_OK) return st;
    a.order_by_length = (plan.splits == 1 && plan.csize == 1 && a.B > 1 && a.B <= 1024 &&
                         static_cast<long long>(a.B) * a.Hkv * a.nh > sms)
                            ? 1
                            : 0;
  }
  if (plan.partials > 1) {
    a.o_part = static_cast<__nv_bfloat16*>(workspace);
    a.lse_part = reinterpret_cast<float*>(static_cast<char*>(workspace) + o_bytes);
  }
  if ((st = encode_out_map(&maps.o, a, params->head_dim)) != NLD_OK) return st;
  if ((st = encode_block_map(&maps.q, q_block, a, params->head_dim)) != NLD_OK) return st;
  if (nld::launch_block_attn_tc(a, maps, params->head_dim, stream) != cudaSuccess) return NLD_ERR_CUDA;
  if (plan.partials > 1 && run_combine) {
    int sms = 0;
    if ((st = device_state(nullptr, &sms)) != NLD_OK) return st;
    if (nld::launch_combine(a.o_part, a.lse_part, plan.partials, a.B, a.Hq, block_len, params->head_dim, a.out, lse,
                            sms, stream) != cudaSuccess)
      return NLD_ERR_CUDA;
  }
  return NLD_OK;
}

}  // namespace

extern "C" {

nld_status_t nld_block_attn(const nld_attn_params_t* params, const void* q_block, const void* k_pages,
                            const void* v_pages, const int32_t* page_table, const int32_t* prefix_lens,
                            int block_len, nld_mode_t mode, void* out, float* lse, void* workspace,
                            size_t workspace_bytes, cudaStream_t stream) {
  return block_attn_impl(params, q_block, k_pages, v_pages, page_table, prefix_lens, block_len, mode, nullptr, out,
                         lse, workspace, workspace_bytes, true, stream);
}

nld_status_t nld_block_attn_masked(const nld_attn_params_t* params, const void* q_block, const void* k_pages,
                                   const void* v_pages, const int32_t* page_table, const int32_t* prefix_lens,
                                   int block_len, const uint32_t* block_mask, void* out, float* lse, void* workspace,
                                   size_t workspace_bytes, cudaStream_t stream) {
  return block_attn_impl(params, q_block, k_pages, v_pages, page_table, prefix_lens, block_len, nld::kModeBlockMask,
                         block_mask, out, lse, workspace, workspace_bytes, true, stream);
}

int nld_quadss_block_mask(int k, uint32_t* masks) {
  // Slot order (Eq. quad_input): the AR token, then for each of the k
  // speculative tokens that token followed by its k masks. The chain (AR
  // and speculative tokens) is causal and sees no mask; the masks of a
  // speculative token see the chain up to it and their own k masks.
  const int n = 1 + k + k * k;
  if (k < 1 || n > nld::kMaxBlock || masks == nullptr) return -1;
  uint32_t chain = 1u;  // chain slots seen so far (the AR token, slot 0)
  masks[0] = chain;
  for (int g = 0; g < k; ++g) {
    const int spec = 1 + g * (k + 1);
    chain |= 1u << spec;
    masks[spec] = chain;
    const uint32_t group = ((1u << k) - 1u) << (spec + 1);  // this token's k masks
    for (int r = 1; r <= k; ++r) masks[spec + r] = chain | group;
  }
  return n;
}

nld_status_t nld_block_attn_partials(const nld_attn_params_t* params, const void* q_block, const void* k_pages,
                                     const void* v_pages, const int32_t* page_table, const int32_t* prefix_lens,
                                     int block_len, nld_mode_t mode, void* out, float* lse, void* workspace,
                                     size_t workspace_bytes, cudaStream_t stream) {
  return block_attn_impl(params, q_block, k_pages, v_pages, page_table, prefix_lens, block_len, mode, nullptr, out,
                         lse, workspace, workspace_bytes, false, stream);
}

nld_status_t nld_split_kv_combine(const void* o_part, const float* lse_part, int num_splits, int batch,
                                  int num_q_heads, int block_len, int head_dim, void* out, float* lse,
                                  cudaStream_t stream) {
  if (num_splits < 1 || num_splits > nld::kMaxSplits || batch < 1 || num_q_heads < 1 || block_len < 1 ||
      block_len > nld::kMaxBlock)
    return NLD_ERR_INVALID_ARG;
  if (head_dim != 64 && head_dim != 128) return NLD_ERR_UNSUPPORTED;
  if (!aligned(o_part, 16) || !aligned(lse_part, 4) || !aligned(out, 16)) return NLD_ERR_INVALID_ARG;
  if (lse != nullptr && !aligned(lse, 4)) return NLD_ERR_INVALID_ARG;
  int sms = 0;
  const nld_status_t st = device_state(nullptr, &sms);
  if (st != NLD_OK) return st;
  if (nld::launch_combine(static_cast<const __nv_bfloat16*>(o_part), lse_part, num_splits, batch, num_q_heads,
                          block_len, head_dim, static_cast<__nv_bfloat16*>(out), lse, sms, stream) != cudaSuccess)
    return NLD_ERR_CUDA;
  return NLD_OK;
}

nld_status_t nld_accept(const int32_t* draft_ids, const int32_t* verify_ids, int batch, int n,
                        int32_t* accepted_len, cudaStream_t stream) {
  if (batch < 1 || n < 1 || n > nld::kMaxBlock) return NLD_ERR_INVALID_ARG;
  if (!aligned(draft_ids, 4) || !aligned(verify_ids, 4) || !aligned(accepted_len, 4)) return NLD_ERR_INVALID_ARG;
  return nld::launch_accept(draft_ids, verify_ids, batch, n, accepted_len, stream) == cudaSuccess ? NLD_OK
                                                                                                   : NLD_ERR_CUDA;
}

nld_status_t nld_unmask(const float* confidences, int batch, int n, int k, int32_t* positions,
                        int32_t* num_selected, cudaStream_t stream) {
  if (batch < 1 || n < 1 || n > nld::kMaxBlock || k < 1 || k > n) return NLD_ERR_INVALID_ARG;
  if (!aligned(confidences, 4) || !aligned(positions, 4)) return NLD_ERR_INVALID_ARG;
  if (num_selected != nullptr && !aligned(num_selected, 4)) return NLD_ERR_INVALID_ARG;
  return nld::launch_unmask(confidences, batch, n, k, positions, num_selected, stream) == cudaSuccess
             ? NLD_OK
             : NLD_ERR_CUDA;
}

nld_status_t nld_unmask_threshold(const float* confidences, int batch, int n, float threshold, int32_t* positions,
                                  int32_t* num_selected, cudaStream_t stream) {
  if (batch < 1 || n < 1 || n > nld::kMaxBlock) return NLD_ERR_INVALID_ARG;
  if (!aligned(confidences, 4) || !aligned(positions, 4)) return NLD_ERR_INVALID_ARG;
  if (num_selected != nullptr && !aligned(num_selected, 4)) return NLD_ERR_INVALID_ARG;
  return nld::launch_unmask_threshold(confidences, batch, n, threshold, positions, num_selected, stream) ==
                 cudaSuccess
             ? NLD_OK
             : NLD_ERR_CUDA;
}

nld_status_t nld_greedy_accept(const int32_t* pred_ids, const int32_t* target_ids, const float* confidences,
                               int batch, int n, int32_t* positions, int32_t* num_selected, cudaStream_t stream) {
  if (batch < 1 || n < 1 || n > nld::kMaxBlock) return NLD_ERR_INVALID_ARG;
  if (!aligned(pred_ids, 4) || !aligned(target_ids, 4) || !aligned(confidences, 4) || !aligned(positions, 4))
    return NLD_ERR_INVALID_ARG;
  if (num_selected != nullptr && !aligned(num_selected, 4)) return NLD_ERR_INVALID_ARG;
  return nld::launch_greedy_accept(pred_ids, target_ids, confidences, batch, n, positions, num_selected, stream) ==
                 cudaSuccess
             ? NLD_OK
             : NLD_ERR_CUDA;
}

nld_status_t nld_logits_argmax(const void* logits, int rows, int vocab, int ld, int32_t* ids, float* conf,
                               cudaStream_t stream) {
  if (rows < 1 || vocab < 1 || ld < vocab || ld % 8 != 0) return NLD_ERR_INVALID_ARG;
  if (!aligned(logits, 16) || !aligned(ids, 4) || !aligned(conf, 4)) return NLD_ERR_INVALID_ARG;
  unsigned int* err = nullptr;
  int sms = 0;
  nld_status_t st = device_state(&err, &sms);
  if (st != NLD_OK) return st;
  // Pieces per row: fill the SMs once when there are fewer rows than SMs, at
  // least one ring stage of vectors a piece, at most one cluster of 8.
  int split = 1;
  if (rows < sms) {
    const int by_sms = sms / rows;
    const int by_len = (vocab / 8) / nld::logits_split_vectors();
    const int want = by_sms < by_len ? by_sms : by_len;
    while (split * 2 <= want && split * 2 <= 8) split *= 2;
  }
  return nld::launch_logits_argmax(static_cast<const __nv_bfloat16*>(logits), rows, vocab, ld, split, ids, conf, err,
                                   stream) == cudaSuccess
             ? NLD_OK
             : NLD_ERR_CUDA;
}

nld_status_t nld_logits_ensemble_argmax(const void* ar_logits, const void* diff_logits, int rows, int vocab, int ld,
                                        float lambda, int32_t* ids, float* conf, cudaStream_t stream) {
  if (rows < 1 || vocab < 1 || ld < vocab || ld % 8 != 0) return NLD_ERR_INVALID_ARG;
  if (!(lambda >= 0.f && lambda <= 1.f)) return NLD_ERR_INVALID_ARG;  // also rejects NaN
  if (!aligned(ar_logits, 16) || !aligned(diff_logits, 16) || !aligned(ids, 4) || !aligned(conf, 4))
    return NLD_ERR_INVALID_ARG;
  int sms = 0;
  nld_status_t st = device_state(nullptr, &sms);
  if (st != NLD_OK) return st;
  int split = 1;
  if (rows < sms) {
    const int by_sms = sms / rows;
    const int by_len = (vocab / 8) / nld::logits_split_vectors();
    const int want = by_sms < by_len ? by_sms : by_len;
    while (split * 2 <= want && split * 2 <= 8) split *= 2;
  }
  return nld::launch_ensemble_argmax(static_cast<const __nv_bfloat16*>(ar_logits),
                                     static_cast<const __nv_bfloat16*>(diff_logits), rows, vocab, ld, split, lambda,
                                     ids, conf, stream) == cudaSuccess
             ? NLD_OK
             : NLD_ERR_CUDA;
}

nld_status_t nld_kv_commit(const nld_attn_params_t* params, const void* k_new, const void* v_new,
                           const int32_t* counts, const int32_t* page_table, int32_t* prefix_lens, int block_len,
                           int advance, void* k_pages, void* v_pages, cudaStream_t stream) {
  nld_status_t st = check_params(params, block_len);
  if (st != NLD_OK) return st;
  if (!aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(k_pages, 16) || !aligned(v_pages, 16) ||
      !aligned(page_table, 4) || !aligned(prefix_lens, 4))
    return NLD_ERR_INVALID_ARG;
  if (counts != nullptr && !aligned(counts, 4)) return NLD_ERR_INVALID_ARG;
  unsigned int* err = nullptr;
  if ((st = device_state(&err, nullptr)) != NLD_OK) return st;
  return nld::launch_kv_commit(static_cast<const __nv_bfloat16*>(k_new), static_cast<const __nv_bfloat16*>(v_new),
                               counts, page_table, prefix_lens, static_cast<__nv_bfloat16*>(k_pages),
                               static_cast<__nv_bfloat16*>(v_pages), params->batch, params->num_kv_heads,
                               params->head_dim, params->page_size, params->num_pages, params->max_pages_per_seq,
                               block_len, advance != 0, err, stream) == cudaSuccess
             ? NLD_OK
             : NLD_ERR_CUDA;
}

nld_status_t nld_check_wait_timeout(uint64_t limit_ns, cudaStream_t stream) {
  if (limit_ns == 0 || limit_ns > nld::kWaitLimitNs) return NLD_ERR_INVALID_ARG;
  unsigned int* err = nullptr;
  nld_status_t st = device_state(&err, nullptr);
  if (st != NLD_OK) return st;
  return nld::launch_wait_timeout_check(limit_ns, err, stream) == cudaSuccess ? NLD_OK : NLD_ERR_CUDA;
}

nld_status_t nld_device_error(uint32_t* bits, int clear) {
  if (bits == nullptr) return NLD_ERR_INVALID_ARG;
  unsigned int* err = nullptr;
  nld_status_t st = device_state(&err, nullptr);
  if (st != NLD_OK) return st;
  unsigned int v = 0;
  if (cudaMemcpy(&v, err, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return NLD_ERR_CUDA;
  *bits = v;
  if (clear) {
    const unsigned int zero = 0;
    if (cudaMemcpy(err, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return NLD_ERR_CUDA;
  }
  return NLD_OK;
}

nld_status_t nld_rescale_count(uint64_t* count, int clear) {
  if (count == nullptr) return NLD_ERR_INVALID_ARG;
  unsigned long long* c = nullptr;
  nld_status_t st = device_state(nullptr, nullptr, &c);
  if (st != NLD_OK) return st;
  unsigned long long v = 0;
  if (cudaMemcpy(&v, c, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return NLD_ERR_CUDA;
  *count = static_cast<uint64_t>(v);
  if (clear) {
    const unsigned long long zero = 0;
    if (cudaMemcpy(c, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return NLD_ERR_CUDA;
  }
  return NLD_OK;
}

}  // extern "C"
