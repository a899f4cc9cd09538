// Block attention over a paged bf16 KV cache (Sec. 2.2 mask; Sec. 3 Modes 2/3).
//
// One CTA serves one (KV split, KV head g, sequence b). Its G = Hq/Hkv query
// heads times the bl block tokens are packed into R = G*bl query rows, so each
// K/V page is read from HBM once per (b, g) and feeds every row of the group.
//
// This is the mma.sync variant, used when more than 128 query rows are packed
// (the tcgen05 kernel in block_attn_tc.cu covers up to 128).
// Warp roles: warps 0 .. nwr*nwt-1 compute, the last warp streams K/V.
//   - Producer (produce_kv): 4-D TMA loads (16 tokens x 64 dims per box,
//     128-byte swizzle) of the pages of each 64-token tile into an nstage-deep
//     ring of shared-memory stages, completing on a "full" mbarrier per stage;
//     it refills a stage after the compute warps release its "empty" mbarrier.
//   - Compute warp (wr, wt): 16 query rows (wr) x a 64/nwt-token slice (wt) of
//     every tile. S = Q K^T and O += P V run on mma.sync m16n8k16 (bf16 in,
//     fp32 accumulate) with ldmatrix reading the swizzled tiles; the online
//     softmax keeps a running max and sum per row in base 2.
// Warps that split a tile's tokens merge their (max, sum, O) in shared memory
// at the end. With one split the CTA writes bf16 O and the natural-log LSE;
// with several it writes fp32 partials for the split combine.
#include "nld_internal.cuh"

namespace nld {
namespace {

// Largest CTA per token split: nwt = 4 and 2 serve up to 2 and 4 row warps,
// nwt = 1 up to kMaxRows / 16; plus the producer warp.
template <int NWT>
struct MaxWarps {
  static constexpr int value = (NWT == 4 ? 8 : NWT == 2 ? 8 : kMaxRows / 16) + 1;
};

template <int D, int NWT>
__global__ void __launch_bounds__(MaxWarps<NWT>::value * 32, 1)
    block_attn_mma_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                          const AttnArgs a) {
  using Geo = TileGeom<D>;
  constexpr int TW = kTileTok / NWT;  // tokens per warp per tile
  constexpr int NT = TW / 8;          // S n-tiles per warp
  constexpr int KD = D / 16;          // k-steps over head_dim
  constexpr int ND = D / 8;           // O n-tiles

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int nstage = a.nstage;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + nstage * Geo::kStageBytes);
  uint64_t* empty = full + nstage;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int ncons = a.nwr * NWT;

  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  if (threadIdx.x == 0) {
    for (int s = 0; s < nstage; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], ncons);
    }
    fence_mbar_init();
  }
  if (warp == ncons && lane == 0) {
    prefetch_tensormap(&tmk);
    prefetch_tensormap(&tmv);
  }
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();
  __syncthreads();

  const int lmax = a.max_pages * a.page_size - a.bl;
  int L = __ldg(a.prefix_lens + b);
  if (L < 0 || L > lmax) {
    if (threadIdx.x == 0) atomicOr(a.err, NLD_DEVERR_PREFIX_RANGE);
    L = min(max(L, 0), lmax);
  }
  const int N = L + a.bl;
  const float scl = a.scale_log2;
  const bool diff_mode = a.mode == NLD_MODE_DIFFUSION;
  const int t_begin = split * a.chunk;
  const int t_end = min(t_begin + a.chunk, N);

  if (t_begin >= t_end) {
    // This split lies past the sequence: its partials carry no keys.
    for (int r = threadIdx.x; r < a.R; r += blockDim.x) {
      const int i = r / a.G, h = g * a.G + (r - i * a.G);
      a.lse_part[((static_cast<size_t>(split) * a.B + b) * a.Hq + h) * a.bl + i] = -INFINITY;
    }
    return;
  }
  const int ntiles = (t_end - t_begin + kTileTok - 1) / kTileTok;

  if (warp == ncons) {
    PagePrefetch first;
    first.load(a, b, t_begin, 0, lane);
    produce_kv<D>(a, &tmk, &tmv, smem, full, empty, nstage, g, b, t_begin, t_end, ntiles, lane, 0, 1, first, 0);
    return;
  }

  // ---------------- compute warps ----------------
  const int wr = warp / NWT, wt = warp % NWT;
  const int r0 = wr * 16;
  const int qlo = lane >> 2;       // row within the 8-row half of the m16 tile
  const int qc = (lane & 3) * 2;   // column pair within an 8-column n-tile

  int row_i[2], row_h[2];
  bool row_ok[2];
#pragma unroll
  for (int hf = 0; hf < 2; ++hf) {
    const int r = r0 + qlo + 8 * hf;
    row_ok[hf] = r < a.R;
    const int i = r / a.G;
    row_i[hf] = i;
    row_h[hf] = g * a.G + (r - i * a.G);
  }

  // Q fragments of this warp's 16 rows, kept in registers for the whole pass.
  uint32_t qa[KD][4];
#pragma unroll
  for (int kk = 0; kk < KD; ++kk) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int hf = e & 1;
      const int col = kk * 16 + qc + (e >> 1) * 8;
      uint32_t v = 0;
      if (row_ok[hf]) {
        const __nv_bfloat16* qp =
            a.q + ((static_cast<size_t>(b) * a.bl + row_i[hf]) * a.Hq + row_h[hf]) * D + col;
        v = __ldg(reinterpret_cast<const unsigned int*>(qp));
      }
      qa[kk][e] = v;
    }
  }

  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.f, 0.f};
  float o[ND][4];
#pragma unroll
  for (int dn = 0; dn < ND; ++dn)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[dn][e] = 0.f;

  const uint32_t smem_base = smem_u32(smem);
  for (int k = 0; k < ntiles; ++k) {
    const int st = k % nstage;
    if (!mbar_wait(&full[st], (k / nstage) & 1, a.err)) break;
    const uint32_t kbase = smem_base + st * Geo::kStageBytes;
    const uint32_t vbase = kbase + Geo::kTileBytes;
    const int tile_t0 = t_begin + k * kTileTok;
    const int valid = t_end - tile_t0;  // tokens of this tile inside the split (>= 1)

    // ---- S = Q K^T over this warp's token slice ----
    float s[NT][4];
#pragma unroll
    for (int j = 0; j < NT; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) s[j][e] = 0.f;
#pragma unroll
    for (int kk = 0; kk < KD; ++kk) {
#pragma unroll
      for (int jn = 0; jn < NT; jn += 2) {
        const int tok = wt * TW + jn * 8 + (lane & 7) + ((lane >> 4) << 3);
        const int chunk = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kbase + kv_swz(tok, chunk), b0, b1, b2, b3);
        mma_16816(s[jn], qa[kk], b0, b1);
        mma_16816(s[jn + 1], qa[kk], b2, b3);
      }
    }

    // ---- mask, scale (base 2), online softmax ----
    // The mask only matters on a tile that reaches the block or the split
    // end; there it is applied branch-free (a branch per element in these
    // unrolled loops is several times slower than the arithmetic).
    float mx[2] = {-INFINITY, -INFINITY};
    if ((tile_t0 + kTileTok <= L) && (valid >= kTileTok)) {
#pragma unroll
      for (int jn = 0; jn < NT; ++jn)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          s[jn][e] *= scl;
          mx[e >> 1] = fmaxf(mx[e >> 1], s[jn][e]);
        }
    } else {
#pragma unroll
      for (int jn = 0; jn < NT; ++jn)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int hf = e >> 1;
          const int col = wt * TW + jn * 8 + qc + (e & 1);
          const int t = tile_t0 + col;
          const bool vis = (col < valid) & ((t < L) | diff_mode | (t - L <= row_i[hf]));
          s[jn][e] = vis ? s[jn][e] * scl : -INFINITY;
          mx[hf] = fmaxf(mx[hf], s[jn][e]);
        }
    }
    float m_use[2];
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
      mx[hf] = fmaxf(mx[hf], __shfl_xor_sync(0xffffffffu, mx[hf], 1));
      mx[hf] = fmaxf(mx[hf], __shfl_xor_sync(0xffffffffu, mx[hf], 2));
      const float m_new = fmaxf(m_run[hf], mx[hf]);
      m_use[hf] = (m_new == -INFINITY) ? 0.f : m_new;
      const float alpha = ex2(m_run[hf] - m_use[hf]);
      m_run[hf] = m_new;
      l_run[hf] *= alpha;
#pragma unroll
      for (int dn = 0; dn < ND; ++dn) {
        o[dn][2 * hf] *= alpha;
        o[dn][2 * hf + 1] *= alpha;
      }
    }
#pragma unroll
    for (int jn = 0; jn < NT; ++jn) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = ex2(s[jn][e] - m_use[e >> 1]);
        s[jn][e] = p;
        l_run[e >> 1] += p;
      }
    }

    // ---- O += P V ----
    // Slots past the end of the sequence inside its last page may hold stale
    // or uninitialised cache data; their P is 0, but 0 * NaN = NaN, so the V
    // operand is zeroed for those tokens (only in a partial last group).
    const bool tail = (valid < kTileTok) && (valid & (kGroupTok - 1));
#pragma unroll
    for (int kt = 0; kt < TW / 16; ++kt) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kt][0], s[2 * kt][1]);
      pa[1] = pack_bf16(s[2 * kt][2], s[2 * kt][3]);
      pa[2] = pack_bf16(s[2 * kt + 1][0], s[2 * kt + 1][1]);
      pa[3] = pack_bf16(s[2 * kt + 1][2], s[2 * kt + 1][3]);
      const int tok_base = wt * TW + kt * 16;
#pragma unroll
      for (int dn = 0; dn < ND; dn += 2) {
        const int tok = tok_base + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int chunk = dn + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vbase + kv_swz(tok, chunk), b0, b1, b2, b3);
        if (tail) {
          // b0/b2 hold tokens tok_base + qc + {0,1}; b1/b3 the same + 8.
          const int t0 = tok_base + qc, t1 = t0 + 8;
          const uint32_t m0 = (t0 < valid ? 0x0000ffffu : 0u) | (t0 + 1 < valid ? 0xffff0000u : 0u);
          const uint32_t m1 = (t1 < valid ? 0x0000ffffu : 0u) | (t1 + 1 < valid ? 0xffff0000u : 0u);
          b0 &= m0;
          b2 &= m0;
          b1 &= m1;
          b3 &= m1;
        }
        mma_16816(o[dn], pa, b0, b1);
        mma_16816(o[dn + 1], pa, b2, b3);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[st]);
  }

#pragma unroll
  for (int hf = 0; hf < 2; ++hf) {
    l_run[hf] += __shfl_xor_sync(0xffffffffu, l_run[hf], 1);
    l_run[hf] += __shfl_xor_sync(0xffffffffu, l_run[hf], 2);
  }

  if constexpr (NWT > 1) {
    // Merge the token slices of warps (wr, 1..NWT-1) into warp (wr, 0).
    // The stage ring is free: every issued load has been consumed.
    constexpr int kSlot = 16 * D + 32;  // floats: O[16][D], m[16], l[16]
    float* mrg = reinterpret_cast<float*>(smem);
    named_bar_sync(1, ncons * 32);
    if (wt > 0) {
      float* slot = mrg + (wr * (NWT - 1) + (wt - 1)) * kSlot;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const int row = qlo + 8 * hf;
#pragma unroll
        for (int dn = 0; dn < ND; ++dn) {
          slot[row * D + dn * 8 + qc] = o[dn][2 * hf];
          slot[row * D + dn * 8 + qc + 1] = o[dn][2 * hf + 1];
        }
        if ((lane & 3) == 0) {
          slot[16 * D + row] = m_run[hf];
          slot[16 * D + 16 + row] = l_run[hf];
        }
      }
    }
    named_bar_sync(1, ncons * 32);
    if (wt > 0) return;
#pragma unroll
    for (int w2 = 1; w2 < NWT; ++w2) {
      const float* slot = mrg + (wr * (NWT - 1) + (w2 - 1)) * kSlot;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const int row = qlo + 8 * hf;
        const float m2 = slot[16 * D + row];
        const float l2 = slot[16 * D + 16 + row];
        const float m_new = fmaxf(m_run[hf], m2);
        const float mu = (m_new == -INFINITY) ? 0.f : m_new;
        const float f1 = ex2(m_run[hf] - mu), f2 = ex2(m2 - mu);
        m_run[hf] = m_new;
        l_run[hf] = l_run[hf] * f1 + l2 * f2;
#pragma unroll
        for (int dn = 0; dn < ND; ++dn) {
          o[dn][2 * hf] = o[dn][2 * hf] * f1 + slot[row * D + dn * 8 + qc] * f2;
          o[dn][2 * hf + 1] = o[dn][2 * hf + 1] * f1 + slot[row * D + dn * 8 + qc + 1] * f2;
        }
      }
    }
  }

  // ---------------- epilogue ----------------
  const bool split_out = a.o_part != nullptr;
#pragma unroll
  for (int hf = 0; hf < 2; ++hf) {
    if (!row_ok[hf]) continue;
    const int i = row_i[hf], h = row_h[hf];
    const float l = l_run[hf];
    const float inv = l > 0.f ? 1.f / l : 0.f;
    const float lse_v = l > 0.f ? (m_run[hf] + lg2(l)) * kLn2 : -INFINITY;
    if (!split_out) {
      __nv_bfloat16* orow = a.out + ((static_cast<size_t>(b) * a.bl + i) * a.Hq + h) * D;
#pragma unroll
      for (int dn = 0; dn < ND; ++dn)
        *reinterpret_cast<uint32_t*>(orow + dn * 8 + qc) = pack_bf16(o[dn][2 * hf] * inv, o[dn][2 * hf + 1] * inv);
      if (a.lse != nullptr && (lane & 3) == 0) a.lse[(static_cast<size_t>(b) * a.Hq + h) * a.bl + i] = lse_v;
    } else {
      const size_t prow = ((static_cast<size_t>(split) * a.B + b) * a.Hq + h) * a.bl + i;
      if (l > 0.f) {
        float* op = a.o_part + prow * D;
#pragma unroll
        for (int dn = 0; dn < ND; ++dn)
          *reinterpret_cast<float2*>(op + dn * 8 + qc) = make_float2(o[dn][2 * hf] * inv, o[dn][2 * hf + 1] * inv);
      }
      if ((lane & 3) == 0) a.lse_part[prow] = lse_v;
    }
  }
}

template <int D, int NWT>
cudaError_t launch_t(const AttnArgs& a, const CUtensorMap& tmk, const CUtensorMap& tmv, const AttnShape& sh,
                     cudaStream_t stream) {
  auto kern = block_attn_mma_kernel<D, NWT>;
  // Opt in to the largest dynamic shared memory any shape of this variant
  // uses, once per device (not inside a stream capture after the first call).
  static int configured[64] = {0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!__atomic_load_n(&configured[dev], __ATOMIC_ACQUIRE)) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(max_smem_bytes(D)));
    if (e != cudaSuccess) return e;
    __atomic_store_n(&configured[dev], 1, __ATOMIC_RELEASE);
  }
  dim3 grid(a.num_splits, a.Hkv, a.B);
  return launch_kernel(kern, grid, dim3(sh.threads), sh.smem, stream, tmk, tmv, a);
}

}  // namespace

size_t max_smem_bytes(int head_dim) {
  // the largest ring plus barriers and alignment slack (every nwt shares nstage)
  return 1024 + 4ull * 2 * kTileTok * head_dim * 2 + 2 * 4 * sizeof(uint64_t);
}

AttnShape attn_shape(int R, int head_dim) {
  AttnShape sh;
  sh.nwr = (R + 15) / 16;
  sh.nwt = sh.nwr >= 5 ? 1 : (sh.nwr >= 3 ? 2 : 4);
  sh.nstage = 4;
  sh.threads = (sh.nwr * sh.nwt + 1) * 32;
  const size_t stage_bytes = 2ull * kTileTok * head_dim * 2;
  const size_t merge_bytes = static_cast<size_t>(sh.nwt - 1) * sh.nwr * (16 * head_dim + 32) * 4;
  size_t ring = sh.nstage * stage_bytes;
  if (merge_bytes > ring) ring = merge_bytes;  // cannot happen for R <= 192, kept as a guard
  sh.smem = 1024 /*alignment slack*/ + ring + 2 * sh.nstage * sizeof(uint64_t);
  return sh;
}

cudaError_t launch_block_attn(const AttnArgs& a, const CUtensorMap& tmk, const CUtensorMap& tmv, int head_dim,
                              cudaStream_t stream) {
  const AttnShape sh = attn_shape(a.R, head_dim);
  AttnArgs args = a;
  args.nwr = sh.nwr;
  args.nstage = sh.nstage;
  if (head_dim == 128) {
    if (sh.nwt == 1) return launch_t<128, 1>(args, tmk, tmv, sh, stream);
    if (sh.nwt == 2) return launch_t<128, 2>(args, tmk, tmv, sh, stream);
    return launch_t<128, 4>(args, tmk, tmv, sh, stream);
  }
  if (sh.nwt == 1) return launch_t<64, 1>(args, tmk, tmv, sh, stream);
  if (sh.nwt == 2) return launch_t<64, 2>(args, tmk, tmv, sh, stream);
  return launch_t<64, 4>(args, tmk, tmv, sh, stream);
}

}  // namespace nld
