// Split-KV combine: merge per-split softmax-normalised partial outputs and
// their log-sum-exps into the full attention result, one warp per output row
// (b, h, i); the row arithmetic is merge_split_row (split_merge.cuh), which
// the attention kernel's in-grid merge runs as well.
#include "split_merge.cuh"

namespace nld {
namespace {

constexpr int kCombineWarps = 8;

template <int D>
__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_kernel(const float* __restrict__ o_part, const float* __restrict__ lse_part, int S, int B, int Hq,
                   int bl, __nv_bfloat16* __restrict__ out, float* __restrict__ lse) {
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();
  const long row = static_cast<long>(blockIdx.x) * kCombineWarps + (threadIdx.x >> 5);
  const long R = static_cast<long>(B) * Hq * bl;
  if (row >= R) return;
  merge_split_row<D, false>(o_part, lse_part, S, R, row, Hq, bl, out, lse);
}

}  // namespace

cudaError_t launch_combine(const float* o_part, const float* lse_part, int S, int B, int Hq, int bl, int D,
                           __nv_bfloat16* out, float* lse, cudaStream_t stream) {
  const long R = static_cast<long>(B) * Hq * bl;
  const unsigned blocks = static_cast<unsigned>((R + kCombineWarps - 1) / kCombineWarps);
  if (D == 128)
    return launch_kernel(combine_kernel<128>, dim3(blocks), dim3(kCombineWarps * 32), 0, stream, o_part, lse_part,
                         S, B, Hq, bl, out, lse);
  return launch_kernel(combine_kernel<64>, dim3(blocks), dim3(kCombineWarps * 32), 0, stream, o_part, lse_part, S,
                       B, Hq, bl, out, lse);
}

}  // namespace nld
