// nld_block_attn_static_scratch: block attention for callers that cannot
// allocate device memory.
//
// Some callers of this library have no way to obtain a workspace: a plugin
// running inside another runtime's enqueue callback, where allocating would
// synchronise the device or is forbidden; code that is not allowed to touch
// the process's allocator (a fixed memory budget accounted elsewhere); or a
// caller that only has raw pointers to its inputs and outputs. For them this
// entry point keeps the split-KV partials in a fixed array compiled into the
// library instead of a caller-provided workspace. It allocates nothing, frees
// nothing and calls no allocating library routine.
//
// The array is a file-scope __device__ variable of kStaticScratchBytes, so
// every GPU that loads the library holds it until the process exits. Its
// device address is looked up once per device, on the first call made with
// that device current (cudaGetSymbolAddress); make that first call before
// any stream capture. Every call on a device shares the one array and it
// keeps the previous call's contents; nothing in it needs to start at zero,
// because the attention kernel writes every partial that the combine reads.
// Two
// calls whose kernels overlap on the GPU (different streams without an
// ordering between them) race on the array.
#include <mutex>

#include "nld_internal.cuh"

namespace {

constexpr size_t kStaticScratchBytes = size_t(16) << 20;  // 16 MiB per device

__device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

constexpr int kMaxScratchDevices = 64;
void* g_scratch_addr[kMaxScratchDevices];
std::mutex g_scratch_mu;

// Device address of the array on the current device, looked up once.
nld_status_t static_scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxScratchDevices) return NLD_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_static_scratch) != cudaSuccess || ptr == nullptr) return NLD_ERR_CUDA;
    g_scratch_addr[dev] = ptr;
  }
  *out = g_scratch_addr[dev];
  return NLD_OK;
}

}  // namespace

extern "C" nld_status_t nld_block_attn_static_scratch(const nld_attn_params_t* params, const void* q_block,
                                                       const void* k_pages, const void* v_pages,
                                                       const int32_t* page_table, const int32_t* prefix_lens,
                                                       int block_len, nld_mode_t mode, void* out, float* lse,
                                                       cudaStream_t stream) {
  const size_t need = nld_block_attn_workspace_size(params, block_len);
  if (need == static_cast<size_t>(-1)) {
    // Let the regular entry point name the problem (it checks before launching).
    return nld_block_attn(params, q_block, k_pages, v_pages, page_table, prefix_lens, block_len, mode, out, lse,
                          nullptr, 0, stream);
  }
  if (need > kStaticScratchBytes) return NLD_ERR_WORKSPACE;  // plan needs more than the fixed array
  void* scratch = nullptr;
  if (need > 0) {
    const nld_status_t st = static_scratch_address(&scratch);
    if (st != NLD_OK) return st;
  }
  return nld_block_attn(params, q_block, k_pages, v_pages, page_table, prefix_lens, block_len, mode, out, lse,
                        scratch, need, stream);
}
