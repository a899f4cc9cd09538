// Token decisions of tri-mode decoding, one warp per sequence (n <= 32).
//  - accept (Sec. 3, Mode 3): ballot of draft != verify over the n positions;
//    the lowest set bit is the first mismatch j*, the accepted length.
//  - unmask (Sec. 3, Mode 2): lane i holds confidence c_i as an unsigned key
//    in the order of the floats (ineligible lanes: 0); k rounds of a warp max
//    reduction each pick the largest key and the lowest lane holding it,
//    which writes its position at that rank and drops out, so positions come
//    out by (confidence descending, position ascending). -inf and NaN are not
//    eligible.
//  - threshold unmasking (Sec. 2, confidence-based sampling) and greedy
//    parallel acceptance (Sec. 5, diffusion SOL): the committed set is a
//    ballot (confidence > threshold; prediction == serial target), each member
//    writes its position at its popcount rank; an empty set falls back to a
//    warp argmax of the confidences.
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
  const int count = __popc(__ballot_sync(0xffffffffu, elig));
  const int sel = count < k ? count : k;
  int32_t* prow = positions + b * k;
  // Selection by warp max: each confidence as an unsigned key in the order
  // of the floats (+0 and -0 equal; ineligible lanes 0, below every eligible
  // key), then sel rounds of (max key, lowest lane holding it), the chosen
  // lane dropping out. Rank order: confidence descending, index ascending.
  const uint32_t bits = __float_as_uint(c == 0.f ? 0.f : c);
  uint32_t key = elig ? ((bits & 0x80000000u) ? ~bits : (bits | 0x80000000u)) : 0u;
  for (int r = 0; r < sel; ++r) {
    const uint32_t top = __reduce_max_sync(0xffffffffu, key);
    const int who = __ffs(__ballot_sync(0xffffffffu, key == top)) - 1;
    if (lane == who) {
      prow[r] = lane;
      key = 0u;
    }
  }
  if (lane >= sel && lane < k) prow[lane] = -1;
  if (lane == 0 && num_selected != nullptr) num_selected[b] = sel;
}

// Writes one step's committed set, given as a ballot over the n lanes: the
// set's lanes in ascending order into prow[0 .. count-1], -1 after. An empty
// set falls back to the single highest eligible confidence (the lower lane on
// ties; +0 and -0 tie), when any position is eligible. Warp-collective.
__device__ __forceinline__ void commit_set(unsigned chosen, float c, bool elig, int lane, int n, int32_t* prow,
                                           int32_t* nsel) {
  if (chosen == 0) {
    float bc = elig ? c : -INFINITY;  // eligible values are never -inf
    int bi = elig ? lane : 32;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float oc = __shfl_xor_sync(0xffffffffu, bc, off);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
      if (oc > bc || (oc == bc && oi < bi)) {
        bc = oc;
        bi = oi;
      }
    }
    if (bi < 32) chosen = 1u << bi;
  }
  const int count = __popc(chosen);
  if ((chosen >> lane) & 1u) prow[__popc(chosen & ((1u << lane) - 1u))] = lane;
  if (lane >= count && lane < n) prow[lane] = -1;
  if (lane == 0 && nsel != nullptr) *nsel = count;
}

__global__ void __launch_bounds__(kDecideWarps * 32)
    unmask_threshold_kernel(const float* __restrict__ conf, int B, int n, float threshold,
                            int32_t* __restrict__ positions, int32_t* __restrict__ num_selected) {
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();
  const int lane = threadIdx.x & 31;
  const long b = static_cast<long>(blockIdx.x) * kDecideWarps + (threadIdx.x >> 5);
  if (b >= B) return;
  const float c = lane < n ? __ldg(conf + b * n + lane) : -INFINITY;
  const bool elig = lane < n && !isnan(c) && c != -INFINITY;
  const unsigned above = __ballot_sync(0xffffffffu, elig && c > threshold);
  commit_set(above, c, elig, lane, n, positions + b * n, num_selected != nullptr ? num_selected + b : nullptr);
}

__global__ void __launch_bounds__(kDecideWarps * 32)
    greedy_accept_kernel(const int32_t* __restrict__ pred, const int32_t* __restrict__ target,
                         const float* __restrict__ conf, int B, int n, int32_t* __restrict__ positions,
                         int32_t* __restrict__ num_selected) {
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();
  const int lane = threadIdx.x & 31;
  const long b = static_cast<long>(blockIdx.x) * kDecideWarps + (threadIdx.x >> 5);
  if (b >= B) return;
  const float c = lane < n ? __ldg(conf + b * n + lane) : -INFINITY;
  const bool elig = lane < n && !isnan(c) && c != -INFINITY;  // still masked
  const bool match = elig && __ldg(pred + b * n + lane) == __ldg(target + b * n + lane);
  commit_set(__ballot_sync(0xffffffffu, match), c, elig, lane, n, positions + b * n,
             num_selected != nullptr ? num_selected + b : nullptr);
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

cudaError_t launch_unmask_threshold(const float* conf, int B, int n, float threshold, int32_t* pos, int32_t* nsel,
                                    cudaStream_t stream) {
  const unsigned blocks = static_cast<unsigned>((B + kDecideWarps - 1) / kDecideWarps);
  return launch_kernel(unmask_threshold_kernel, dim3(blocks), dim3(kDecideWarps * 32), 0, stream, conf, B, n,
                       threshold, pos, nsel);
}

// One thread initialises an mbarrier that expects one arrival, never
// arrives, and waits on it with the pipelines' bounded wait: the wait gives
// up after limit_ns and records NLD_DEVERR_WAIT_TIMEOUT, as any kernel's
// wait would, and the kernel returns.
__global__ void __launch_bounds__(32) wait_timeout_check_kernel(uint64_t limit_ns, unsigned int* err) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    mbar_wait_for(&bar, 0, err, limit_ns);
  }
}

cudaError_t launch_wait_timeout_check(uint64_t limit_ns, unsigned int* err, cudaStream_t stream) {
  wait_timeout_check_kernel<<<1, 32, 0, stream>>>(limit_ns, err);
  return cudaGetLastError();
}

cudaError_t launch_greedy_accept(const int32_t* pred, const int32_t* target, const float* conf, int B, int n,
                                 int32_t* pos, int32_t* nsel, cudaStream_t stream) {
  const unsigned blocks = static_cast<unsigned>((B + kDecideWarps - 1) / kDecideWarps);
  return launch_kernel(greedy_accept_kernel, dim3(blocks), dim3(kDecideWarps * 32), 0, stream, pred, target, conf,
                       B, n, pos, nsel);
}

}  // namespace nld
