// Split-KV combine: merge per-split softmax-normalised partial outputs and
// their log-sum-exps into the full attention result.
//   m = max_s lse_s, c_s = exp(lse_s - m), out = sum_s c_s o_s / sum_s c_s,
//   lse = m + ln sum_s c_s.
// One warp per output row (b, h, i); each lane owns D/32 consecutive dims, so
// every partial row is read as one coalesced 256/512-byte segment.
#include "nld_internal.cuh"

namespace nld {
namespace {

constexpr int kCombineWarps = 8;

template <int D>
__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_kernel(const float* __restrict__ o_part, const float* __restrict__ lse_part, int S, int B, int Hq,
                   int bl, __nv_bfloat16* __restrict__ out, float* __restrict__ lse) {
  constexpr int V = D / 32;  // dims per lane (2 or 4)
  const int lane = threadIdx.x & 31;
  const long row = static_cast<long>(blockIdx.x) * kCombineWarps + (threadIdx.x >> 5);
  const long R = static_cast<long>(B) * Hq * bl;
  if (row >= R) return;
  // partial row order is [B, Hq, bl]
  const int i = static_cast<int>(row % bl);
  const long bh = row / bl;
  const int h = static_cast<int>(bh % Hq);
  const int b = static_cast<int>(bh / Hq);

  float m = -INFINITY;
  for (int s = lane; s < S; s += 32) m = fmaxf(m, __ldg(lse_part + static_cast<long>(s) * R + row));
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));

  float acc[V];
#pragma unroll
  for (int v = 0; v < V; ++v) acc[v] = 0.f;
  float csum = 0.f;
  if (m != -INFINITY) {
    const float m2 = m * kLog2e;
#pragma unroll 4
    for (int s = 0; s < S; ++s) {
      const float ls = __ldg(lse_part + static_cast<long>(s) * R + row);
      if (ls == -INFINITY) continue;  // no keys in this split: o_s is not read
      const float c = ex2(ls * kLog2e - m2);
      csum += c;
      const float* op = o_part + (static_cast<long>(s) * R + row) * D + lane * V;
      if constexpr (V == 4) {
        const float4 x = __ldg(reinterpret_cast<const float4*>(op));
        acc[0] += c * x.x; acc[1] += c * x.y; acc[2] += c * x.z; acc[3] += c * x.w;
      } else {
        const float2 x = __ldg(reinterpret_cast<const float2*>(op));
        acc[0] += c * x.x; acc[1] += c * x.y;
      }
    }
  }
  const float inv = csum > 0.f ? 1.f / csum : 0.f;
  __nv_bfloat16* orow = out + ((static_cast<long>(b) * bl + i) * Hq + h) * D + lane * V;
#pragma unroll
  for (int v = 0; v < V; v += 2)
    *reinterpret_cast<uint32_t*>(orow + v) = pack_bf16(acc[v] * inv, acc[v + 1] * inv);
  if (lse != nullptr && lane == 0)
    lse[(static_cast<long>(b) * Hq + h) * bl + i] = csum > 0.f ? m + lg2(csum) * kLn2 : -INFINITY;
}

}  // namespace

cudaError_t launch_combine(const float* o_part, const float* lse_part, int S, int B, int Hq, int bl, int D,
                           __nv_bfloat16* out, float* lse, cudaStream_t stream) {
  const long R = static_cast<long>(B) * Hq * bl;
  const unsigned blocks = static_cast<unsigned>((R + kCombineWarps - 1) / kCombineWarps);
  if (D == 128)
    combine_kernel<128><<<blocks, kCombineWarps * 32, 0, stream>>>(o_part, lse_part, S, B, Hq, bl, out, lse);
  else
    combine_kernel<64><<<blocks, kCombineWarps * 32, 0, stream>>>(o_part, lse_part, S, B, Hq, bl, out, lse);
  return cudaGetLastError();
}

}  // namespace nld
