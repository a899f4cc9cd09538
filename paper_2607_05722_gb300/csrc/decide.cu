// Token decisions of tri-mode decoding, one warp per sequence (n <= 32).
//  - accept (Sec. 3, Mode 3): ballot of draft != verify over the n positions;
//    the lowest set bit is the first mismatch j*, the accepted length.
//  - unmask (Sec. 3, Mode 2): lane i holds confidence c_i; its rank is
//    #{j eligible: c_j > c_i} + #{j < i eligible: c_j == c_i}, so ranks of
//    the eligible lanes are a permutation and the k smallest are written in
//    rank order. -inf and NaN are not eligible.
#include "nld_internal.cuh"

namespace nld {
namespace {

constexpr int kDecideWarps = 8;

__global__ void __launch_bounds__(kDecideWarps * 32)
    accept_kernel(const int32_t* __restrict__ draft, const int32_t* __restrict__ verify, int B, int n,
                  int32_t* __restrict__ accepted) {
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();
  const int lane = threadIdx.x & 31;
  const long b = static_cast<long>(blockIdx.x) * kDecideWarps + (threadIdx.x >> 5);
  if (b >= B) return;
  const bool differ = lane < n && __ldg(draft + b * n + lane) != __ldg(verify + b * n + lane);
  const unsigned mism = __ballot_sync(0xffffffffu, differ);
  if (lane == 0) accepted[b] = mism ? __ffs(mism) - 1 : n;
}

__global__ void __launch_bounds__(kDecideWarps * 32)
    unmask_kernel(const float* __restrict__ conf, int B, int n, int k, int32_t* __restrict__ positions,
                  int32_t* __restrict__ num_selected) {
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();
  const int lane = threadIdx.x & 31;
  const long b = static_cast<long>(blockIdx.x) * kDecideWarps + (threadIdx.x >> 5);
  if (b >= B) return;
  const float c = lane < n ? __ldg(conf + b * n + lane) : -INFINITY;
  const bool elig = lane < n && !isnan(c) && c != -INFINITY;
  int rank = 0;
  for (int j = 0; j < n; ++j) {
    const float cj = __shfl_sync(0xffffffffu, c, j);
    const bool ej = !isnan(cj) && cj != -INFINITY;  // j < n here
    rank += (ej && (cj > c || (cj == c && j < lane))) ? 1 : 0;
  }
  const int count = __popc(__ballot_sync(0xffffffffu, elig));
  const int sel = count < k ? count : k;
  int32_t* prow = positions + b * k;
  if (elig && rank < k) prow[rank] = lane;
  if (lane >= sel && lane < k) prow[lane] = -1;
  if (lane == 0 && num_selected != nullptr) num_selected[b] = sel;
}

}  // namespace

cudaError_t launch_accept(const int32_t* draft, const int32_t* verify, int B, int n, int32_t* acc,
                          cudaStream_t stream) {
  const unsigned blocks = static_cast<unsigned>((B + kDecideWarps - 1) / kDecideWarps);
  return launch_kernel(accept_kernel, dim3(blocks), dim3(kDecideWarps * 32), 0, stream, draft, verify, B, n, acc);
}

cudaError_t launch_unmask(const float* conf, int B, int n, int k, int32_t* pos, int32_t* nsel,
                          cudaStream_t stream) {
  const unsigned blocks = static_cast<unsigned>((B + kDecideWarps - 1) / kDecideWarps);
  return launch_kernel(unmask_kernel, dim3(blocks), dim3(kDecideWarps * 32), 0, stream, conf, B, n, k, pos, nsel);
}

}  // namespace nld
