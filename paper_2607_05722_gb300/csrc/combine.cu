// Split-KV combine: merge per-split softmax-normalised partial outputs (bf16)
// and their log-sum-exps (fp32) into the full attention result.
//   m = max_s lse_s, c_s = exp(lse_s - m), out = sum_s c_s o_s / sum_s c_s,
//   lse = m + ln sum_s c_s.
// One warp per output row (b, h, i); each lane owns D/32 consecutive dims, so
// every partial row is read as one coalesced 128/256-byte segment; lane j
// holds the lse of splits j, j+32, ... Partials of splits without keys
// (lse = -inf) are never read. The weights and sums are fp32.
#include "nld_internal.cuh"

namespace nld {
namespace {

// Row `row` of R = B*Hq*bl rows (partial row order [B, Hq, bl]); o_part
// [S, R, D] bf16, lse_part [S, R] (natural log). Warp-collective.
template <int D>
__device__ __forceinline__ void merge_split_row(const __nv_bfloat16* __restrict__ o_part,
                                                const float* __restrict__ lse_part,
                                                int S, long R, long row, int Hq, int bl,
                                                __nv_bfloat16* __restrict__ out, float* __restrict__ lse) {
  constexpr int V = D / 32;  // dims per lane (2 or 4)
  const int lane = threadIdx.x & 31;
  const int i = static_cast<int>(row % bl);
  const long bh = row / bl;
  const int h = static_cast<int>(bh % Hq);
  const long b = bh / Hq;

  // One memory round trip per 32 splits: each lane loads its share of the
  // partial rows at the same time as the lse values.
  constexpr int kMaxPerLane = kMaxSplits / 32;
  constexpr int kRound = 32;
  const long split_stride = R * static_cast<long>(D);
  const __nv_bfloat16* base = o_part + row * D + lane * V;
  float ls[kMaxPerLane];
#pragma unroll
  for (int u = 0; u < kMaxPerLane; ++u) {
    const int s = lane + 32 * u;
    ls[u] = s < S ? __ldg(lse_part + static_cast<long>(s) * R + row) : -INFINITY;
  }
  uint32_t x[kRound][V / 2];  // bf16 pairs
  auto load_round = [&](int s0) {
#pragma unroll
    for (int u = 0; u < kRound; ++u) {
      const int s = s0 + u;
      if (s < S) {
        const __nv_bfloat16* op = base + s * split_stride;
        if constexpr (V == 4) {
          const uint2 t = __ldg(reinterpret_cast<const uint2*>(op));
          x[u][0] = t.x;
          x[u][1] = t.y;
        } else {
          x[u][0] = __ldg(reinterpret_cast<const unsigned int*>(op));
        }
      }
    }
  };
  load_round(0);
  float m = -INFINITY;
#pragma unroll
  for (int u = 0; u < kMaxPerLane; ++u) m = fmaxf(m, ls[u]);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));

  float acc[V];
#pragma unroll
  for (int v = 0; v < V; ++v) acc[v] = 0.f;
  float csum = 0.f;
  if (m != -INFINITY) {
    const float m2 = m * kLog2e;
    float w[kMaxPerLane];  // weight of split lane + 32u; 0 for empty splits
#pragma unroll
    for (int u = 0; u < kMaxPerLane; ++u) {
      w[u] = ls[u] == -INFINITY ? 0.f : ex2(fmaf(ls[u], kLog2e, -m2));
      csum += w[u];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) csum += __shfl_xor_sync(0xffffffffu, csum, off);
    for (int s0 = 0; s0 < S; s0 += kRound) {
      if (s0 > 0) load_round(s0);
      const int blk = s0 >> 5;  // warp-uniform
      const float wsrc = blk == 0 ? w[0] : blk == 1 ? w[1] : blk == 2 ? w[2] : w[3];
#pragma unroll
      for (int u = 0; u < kRound; ++u) {
        const float wu = __shfl_sync(0xffffffffu, wsrc, u);
        if (s0 + u < S && wu > 0.f) {
#pragma unroll
          for (int v = 0; v < V / 2; ++v) {
            float lo, hi;
            unpack_bf16(x[u][v], lo, hi);
            acc[2 * v] = fmaf(wu, lo, acc[2 * v]);
            acc[2 * v + 1] = fmaf(wu, hi, acc[2 * v + 1]);
          }
        }
      }
    }
  }
  const float inv = csum > 0.f ? 1.f / csum : 0.f;
  __nv_bfloat16* orow = out + ((b * bl + i) * Hq + h) * D + lane * V;
#pragma unroll
  for (int v = 0; v < V; v += 2)
    *reinterpret_cast<uint32_t*>(orow + v) = pack_bf16(acc[v] * inv, acc[v + 1] * inv);
  if (lse != nullptr && lane == 0)
    lse[(b * Hq + h) * bl + i] = csum > 0.f ? fmaf(lg2(csum), kLn2, m) : -INFINITY;
}


constexpr int kCombineWarps = 8;

template <int D>
__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_kernel(const __nv_bfloat16* __restrict__ o_part, const float* __restrict__ lse_part, int S, int B, int Hq,
                   int bl, __nv_bfloat16* __restrict__ out, float* __restrict__ lse) {
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();
  const long row = static_cast<long>(blockIdx.x) * kCombineWarps + (threadIdx.x >> 5);
  const long R = static_cast<long>(B) * Hq * bl;
  if (row >= R) return;
  merge_split_row<D>(o_part, lse_part, S, R, row, Hq, bl, out, lse);
}

// The combine is bound by the rate at which an SM pulls partial rows from
// L2, so its CTAs should sit on as many SMs as possible. At 96 registers a
// thread two CTAs fit on one SM and the scheduler packs them; when the grid
// fits in one wave, a dynamic shared-memory request of more than half an SM
// (used for nothing) keeps it to one CTA per SM (measured at 17 partials x
// 512 rows: 3.0 -> 2.8 us). Larger grids launch without it.
constexpr int kSpreadSmemBytes = 120 * 1024;

template <int D>
cudaError_t configure_combine(int dev) {
  static int configured[64] = {0};
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!__atomic_load_n(&configured[dev], __ATOMIC_ACQUIRE)) {
    cudaError_t e =
        cudaFuncSetAttribute(combine_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSpreadSmemBytes);
    if (e != cudaSuccess) return e;
    __atomic_store_n(&configured[dev], 1, __ATOMIC_RELEASE);
  }
  return cudaSuccess;
}

template <int D>
cudaError_t launch_combine_d(const __nv_bfloat16* o_part, const float* lse_part, int S, int B, int Hq, int bl,
                             __nv_bfloat16* out, float* lse, int sm_count, cudaStream_t stream) {
  const long R = static_cast<long>(B) * Hq * bl;
  const unsigned blocks = static_cast<unsigned>((R + kCombineWarps - 1) / kCombineWarps);
  size_t smem = 0;
  if (static_cast<long>(blocks) <= sm_count) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if ((e = configure_combine<D>(dev)) != cudaSuccess) return e;
    smem = kSpreadSmemBytes;
  }
  return launch_kernel(combine_kernel<D>, dim3(blocks), dim3(kCombineWarps * 32), smem, stream, o_part, lse_part, S,
                       B, Hq, bl, out, lse);
}

}  // namespace

cudaError_t launch_combine(const __nv_bfloat16* o_part, const float* lse_part, int S, int B, int Hq, int bl, int D,
                           __nv_bfloat16* out, float* lse, int sm_count, cudaStream_t stream) {
  if (D == 128) return launch_combine_d<128>(o_part, lse_part, S, B, Hq, bl, out, lse, sm_count, stream);
  return launch_combine_d<64>(o_part, lse_part, S, B, Hq, bl, out, lse, sm_count, stream);
}

}  // namespace nld
