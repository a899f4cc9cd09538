// Block KV commit into the paged cache (Sec. 3 Mode 3: the accepted prefix is
// committed and the verifier's cache is rebuilt at the rejection point;
// Sec. 2: a completed block's KV cache is refreshed). Row j < count_b of the
// block's new K/V goes to logical slot L_b + j, i.e. page
// page_table[b][(L_b + j) / P], slot (L_b + j) mod P, for every KV head. One
// CTA per (row, sequence) moves the row's Hkv*D values of K and V in 16-byte
// vectors; a second kernel advances L_b by count_b, after every copy has read
// the old L_b (stream order; with PDL its dependency wait covers the copy).
#include "nld_internal.cuh"

namespace nld {
namespace {

constexpr int kCommitThreads = 256;

__global__ void __launch_bounds__(kCommitThreads)
    kv_commit_kernel(const __nv_bfloat16* __restrict__ k_new, const __nv_bfloat16* __restrict__ v_new,
                     const int32_t* __restrict__ counts, const int32_t* __restrict__ page_table,
                     const int32_t* __restrict__ prefix_lens, __nv_bfloat16* __restrict__ k_pages,
                     __nv_bfloat16* __restrict__ v_pages, int Hkv, int D, int P, int log2_page, int num_pages,
                     int max_pages, int bl, unsigned int* err) {
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();    // k_new, counts and prefix_lens come from earlier kernels
  const int j = blockIdx.x;
  const long b = blockIdx.y;
  int count = counts != nullptr ? __ldg(counts + b) : bl;
  if (count < 0 || count > bl) {
    if (threadIdx.x == 0 && j == 0) atomicOr(err, NLD_DEVERR_PREFIX_RANGE);
    count = min(max(count, 0), bl);
  }
  if (j >= count) return;
  const long t = static_cast<long>(__ldg(prefix_lens + b)) + j;
  if (t < 0 || t >= static_cast<long>(max_pages) * P) {
    if (threadIdx.x == 0) atomicOr(err, NLD_DEVERR_PREFIX_RANGE);
    return;
  }
  const int page = __ldg(page_table + b * max_pages + (t >> log2_page));
  if (page < 0 || page >= num_pages) {
    if (threadIdx.x == 0) atomicOr(err, NLD_DEVERR_PAGE_RANGE);
    return;
  }
  const long slot = t & (P - 1);
  const int vec_per_head = D / 8;
  const int nvec = Hkv * vec_per_head;
  const long src = (b * bl + j) * static_cast<long>(Hkv) * D;
  for (int v = threadIdx.x; v < 2 * nvec; v += kCommitThreads) {
    const bool is_v = v >= nvec;
    const int w = is_v ? v - nvec : v;
    const int g = w / vec_per_head, c = w - g * vec_per_head;
    const long dst = ((static_cast<long>(page) * Hkv + g) * P + slot) * D + c * 8;
    const uint4 x = __ldg(reinterpret_cast<const uint4*>((is_v ? v_new : k_new) + src) + w);
    *reinterpret_cast<uint4*>((is_v ? v_pages : k_pages) + dst) = x;
  }
}

__global__ void __launch_bounds__(kCommitThreads)
    advance_prefix_kernel(const int32_t* __restrict__ counts, int32_t* __restrict__ prefix_lens, int B, int bl) {
  grid_launch_dependents();
  grid_dependency_wait();  // every copy of the commit has read the old lengths
  const long b = static_cast<long>(blockIdx.x) * kCommitThreads + threadIdx.x;
  if (b >= B) return;
  const int count = counts != nullptr ? min(max(counts[b], 0), bl) : bl;
  prefix_lens[b] += count;
}

}  // namespace

cudaError_t launch_kv_commit(const __nv_bfloat16* k_new, const __nv_bfloat16* v_new, const int32_t* counts,
                             const int32_t* page_table, int32_t* prefix_lens, __nv_bfloat16* k_pages,
                             __nv_bfloat16* v_pages, int B, int Hkv, int D, int P, int num_pages, int max_pages,
                             int bl, bool advance, unsigned int* err, cudaStream_t stream) {
  const int log2_page = __builtin_ctz(static_cast<unsigned>(P));
  cudaError_t e = launch_kernel(kv_commit_kernel, dim3(bl, B), dim3(kCommitThreads), 0, stream, k_new, v_new, counts,
                                page_table, prefix_lens, k_pages, v_pages, Hkv, D, P, log2_page, num_pages, max_pages,
                                bl, err);
  if (e != cudaSuccess || !advance) return e;
  return launch_kernel(advance_prefix_kernel, dim3((B + kCommitThreads - 1) / kCommitThreads), dim3(kCommitThreads),
                       0, stream, counts, prefix_lens, B, bl);
}

}  // namespace nld
