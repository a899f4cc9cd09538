// Logits -> (argmax id, confidence) per position: the inputs of the token
// decisions (Sec. 2 confidence-based sampling; Sec. 5 serial denoising
// commits the position with the highest peak probability).
//   m = max_v l_v, id = the lowest v with l_v = m,
//   conf = max_v softmax(l)_v = 1 / sum_v exp(l_v - m).
// A row is cut into `split` pieces, one CTA each (a thread-block cluster when
// split > 1). Pieces of at most 2048 vectors (a few rows over many SMs, as
// in a decode step) take logits_argmax_small_kernel: every thread loads its
// vectors at once and folds them in one pass. Larger pieces stream: in a CTA
// one producer warp streams the piece through a ring of
// 16 KB stages with bulk copies (TMA engine) and eight warps fold each 8-logit
// vector into a running (max, sum of exp(l - max), argmax): the vector max
// comes first, so the rare rescale happens once per vector, then one exp per
// logit. The partial states merge by the log-sum-exp rule (ties: the lower
// index) across the warps, the CTA and, through distributed shared memory,
// the cluster. NaN logits never win the argmax and make the sum NaN; a row
// with nothing above -inf gets id 0 and confidence 0.
#include "nld_internal.cuh"

namespace nld {
namespace {

constexpr int kLgConsumerWarps = 8;
constexpr int kLgThreads = 32 * (kLgConsumerWarps + 1);  // + the producer warp
constexpr int kLgStages = 4;
constexpr int kLgStageVecs = 1024;                       // 16-byte vectors (8 logits): 16 KB a stage
constexpr int kLgRingBytes = kLgStages * kLgStageVecs * 16;
constexpr int kLgSmemBytes = kLgRingBytes + 2 * kLgStages * 8 + 4 * 8 * 3 + 16 + 128;  // + alignment slack

// Merge (m2, s2, i2) into (m, s, i): the max, the sums rescaled to it, and
// the argmax (the lower index when the maxima are equal). A state whose max
// is still -inf has sum 0, or NaN if it met a NaN logit; it enters the merge
// as sum * 0, which keeps the NaN.
__device__ __forceinline__ void lg_merge(float& m, float& s, int& i, float m2, float s2, int i2) {
  const float mm = fmaxf(m, m2);
  i = m > m2 ? i : (m2 > m ? i2 : min(i, i2));
  const float a = m == -INFINITY ? s * 0.f : s * ex2((m - mm) * kLog2e);
  const float b = m2 == -INFINITY ? s2 * 0.f : s2 * ex2((m2 - mm) * kLog2e);
  m = mm;
  s = a + b;
}

// Fold x[0..n) (logits e0 .. e0+n-1, in index order) into (m, s, i).
template <int N>
__device__ __forceinline__ void lg_fold(const float (&x)[N], int e0, float& m, float& s, int& i) {
  float vm = x[0];
#pragma unroll
  for (int j = 1; j < N; ++j) vm = fmaxf(vm, x[j]);
  if (vm > m) {  // a new running max (NaN never is)
    s = m == -INFINITY ? s * 0.f : s * ex2((m - vm) * kLog2e);
    m = vm;
    int first = N - 1;
#pragma unroll
    for (int j = N - 1; j >= 0; --j)
      if (x[j] == vm) first = j;
    i = e0 + first;
  }
  if (m != -INFINITY) {
#pragma unroll
    for (int j = 0; j < N; ++j) s += ex2((x[j] - m) * kLog2e);  // a NaN logit makes s NaN
  } else {
#pragma unroll
    for (int j = 0; j < N; ++j)
      if (isnan(x[j])) s = NAN;  // nothing finite yet: the NaN must still reach the sum
  }
}

__global__ void __launch_bounds__(kLgThreads)
    logits_argmax_kernel(const __nv_bfloat16* __restrict__ logits, int vocab, long ld, int split,
                         int32_t* __restrict__ ids, float* __restrict__ conf, unsigned int* err) {
  extern __shared__ uint8_t lg_smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(lg_smem_raw) + 127) & ~uintptr_t(127));
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + kLgRingBytes);
  uint64_t* empty = full + kLgStages;
  float* red = reinterpret_cast<float*>(empty + kLgStages);  // [consumer warp][m, s, i]
  float* part = red + 3 * kLgConsumerWarps;                   // this CTA's merged state, for the cluster

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int piece = static_cast<int>(blockIdx.x % split);
  const long row = static_cast<long>(blockIdx.x / split);
  const int nvec = vocab >> 3, tail = vocab & 7;
  const int per = (nvec + split - 1) / split;
  const int v0 = min(nvec, piece * per), v1 = min(nvec, v0 + per);
  const int nst = (v1 - v0 + kLgStageVecs - 1) / kLgStageVecs;

  if (threadIdx.x == 0) {
    for (int st = 0; st < kLgStages; ++st) {
      mbar_init(&full[st], 1);
      mbar_init(&empty[st], kLgConsumerWarps);
    }
    fence_mbar_init();
  }
  __syncthreads();
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();    // the logits come from the previous kernel
  const uint8_t* grow = reinterpret_cast<const uint8_t*>(logits + row * ld);

  float m = -INFINITY, s = 0.f;
  int idx = 0;
  if (warp == kLgConsumerWarps) {
    // ---- producer: one lane issues the stages of this piece ----
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      for (int k = 0; k < nst; ++k) {
        const int st = k % kLgStages;
        if (k >= kLgStages && !mbar_wait(&empty[st], ((k / kLgStages) - 1) & 1, err)) {
          ok = false;
          break;
        }
        const uint32_t bytes = static_cast<uint32_t>(min(kLgStageVecs, v1 - v0 - k * kLgStageVecs)) * 16u;
        mbar_arrive_expect_tx(&full[st], bytes);
        bulk_load(ring + st * kLgStageVecs * 16, grow + static_cast<long>(v0 + k * kLgStageVecs) * 16, bytes,
                  &full[st]);
        issued = k + 1;
      }
      if (!ok) {
        // Gave up on a timeout: let the copies in flight land before exit (bounded).
        for (int k = max(0, issued - kLgStages); k < issued; ++k)
          mbar_wait(&full[k % kLgStages], (k / kLgStages) & 1, err);
      }
    }
  } else {
    // ---- consumers: thread t folds vectors t, t+256, ... of each stage ----
    const int t = threadIdx.x;
    for (int k = 0; k < nst; ++k) {
      const int st = k % kLgStages;
      if (!__all_sync(0xffffffffu, mbar_wait(&full[st], (k / kLgStages) & 1, err))) break;
      const int nv = min(kLgStageVecs, v1 - v0 - k * kLgStageVecs);
      const uint4* sv = reinterpret_cast<const uint4*>(ring + st * kLgStageVecs * 16);
      const int ebase = (v0 + k * kLgStageVecs) * 8;
      for (int j = t; j < nv; j += 32 * kLgConsumerWarps) {
        const uint4 w = sv[j];
        float x[8];
        unpack_bf16(w.x, x[0], x[1]);
        unpack_bf16(w.y, x[2], x[3]);
        unpack_bf16(w.z, x[4], x[5]);
        unpack_bf16(w.w, x[6], x[7]);
        lg_fold(x, ebase + j * 8, m, s, idx);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
    if (piece == split - 1 && t < tail) {  // the last vocab % 8 logits, after every vector
      const uint16_t bits = reinterpret_cast<const uint16_t*>(grow)[nvec * 8 + t];
      const float x[1] = {__uint_as_float(static_cast<uint32_t>(bits) << 16)};
      lg_fold(x, nvec * 8 + t, m, s, idx);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
      const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
      const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
      lg_merge(m, s, idx, m2, s2, i2);
    }
    if (lane == 0) {
      red[3 * warp] = m;
      red[3 * warp + 1] = s;
      red[3 * warp + 2] = __int_as_float(idx);
    }
  }
  __syncthreads();
  if (warp == 0) {
    m = lane < kLgConsumerWarps ? red[3 * lane] : -INFINITY;
    s = lane < kLgConsumerWarps ? red[3 * lane + 1] : 0.f;
    idx = lane < kLgConsumerWarps ? __float_as_int(red[3 * lane + 2]) : 0;
#pragma unroll
    for (int off = 4; off > 0; off >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
      const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
      const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
      lg_merge(m, s, idx, m2, s2, i2);
    }
    if (lane == 0) {
      if (split == 1) {
        ids[row] = idx;
        conf[row] = m == -INFINITY ? 0.f : 1.f / s;
      } else {
        part[0] = m;
        part[1] = s;
        part[2] = __int_as_float(idx);
      }
    }
  }
  if (split > 1) {
    // Merge the pieces of the row: rank 0 reads every CTA's state through
    // distributed shared memory; the second barrier keeps the peers' shared
    // memory alive until it has.
    cluster_sync();
    if (cluster_ctarank() == 0 && warp == 0) {
      const uint32_t pa = smem_u32(part);
      m = -INFINITY;
      s = 0.f;
      idx = 0;
      if (lane < split) {
        m = ld_dsmem_f32(dsmem_addr(pa, lane));
        s = ld_dsmem_f32(dsmem_addr(pa + 4, lane));
        idx = __float_as_int(ld_dsmem_f32(dsmem_addr(pa + 8, lane)));
      }
#pragma unroll
      for (int off = 4; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
        const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
        lg_merge(m, s, idx, m2, s2, i2);
      }
      if (lane == 0) {
        ids[row] = idx;
        conf[row] = m == -INFINITY ? 0.f : 1.f / s;
      }
    }
    cluster_sync();
  }
}

// Small pieces (at most kLsThreads * kLsMaxVecs 8-logit vectors per CTA: a
// few rows over many SMs, the decode-step case): no ring. Every thread loads
// all its vectors at once (one memory round trip), folds them in one pass
// (the max of its logits first, then one exp per logit against it), and
// the CTA merges the threads' states; the pieces of a row then push their
// states into rank 0's shared memory with a remote store and a release
// arrival on rank 0's mbarrier, and rank 0 merges them, so no peer waits
// for another. Same rules as logits_argmax_kernel (ties to the lower index;
// NaN never wins and makes the sum NaN; nothing above -inf: id 0, conf 0).
constexpr int kLsThreads = 256;  // light enough for two CTAs per SM, so every cluster of 8 is resident at once
constexpr int kLsMaxVecs = 8;  // vectors a thread holds in flight

__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.aligned;" ::: "memory"); }
__device__ __forceinline__ void st_dsmem_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void mbar_arrive_remote_release(uint32_t addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(addr) : "memory");
}
// Wait (bounded) with acquire at cluster scope, for arrivals made by peers.
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, unsigned int* err) {
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 0;; ++it) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (ok) return true;
    if ((it & 255u) == 255u && global_timer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, NLD_DEVERR_WAIT_TIMEOUT);
      return false;
    }
  }
}

__global__ void __launch_bounds__(kLsThreads)
    logits_argmax_small_kernel(const __nv_bfloat16* __restrict__ logits, int vocab, long ld, int split,
                               int32_t* __restrict__ ids, float* __restrict__ conf, unsigned int* err) {
  __shared__ float red[kLsThreads / 32][3];
  __shared__ float parts[8][3];  // rank 0: the pieces' (m, s, id)
  __shared__ __align__(8) uint64_t arrived;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, t = threadIdx.x;
  const int piece = static_cast<int>(blockIdx.x % split);
  const long row = static_cast<long>(blockIdx.x / split);
  const int nvec = vocab >> 3, tail = vocab & 7;
  const int per = (nvec + split - 1) / split;
  const int v0 = min(nvec, piece * per), v1 = min(nvec, v0 + per);
  if (split > 1) {
    if (t == 0) {
      mbar_init(&arrived, static_cast<uint32_t>(split));
      fence_mbar_init();
    }
    cluster_arrive_relaxed();  // rank 0's barrier is ready once every CTA has arrived (waited below)
  }
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  grid_dependency_wait();    // the logits come from the previous kernel
  const uint4* grow = reinterpret_cast<const uint4*>(logits + row * ld);
  uint4 w[kLsMaxVecs];
#pragma unroll
  for (int j = 0; j < kLsMaxVecs; ++j) {
    const int v = v0 + t + j * kLsThreads;
    w[j] = v < v1 ? __ldg(grow + v) : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);  // -inf
  }
  // max of this thread's logits and the lowest index holding it
  float m = -INFINITY;
  int idx = 0;
#pragma unroll
  for (int j = 0; j < kLsMaxVecs; ++j) {
    float x[8];
    unpack_bf16(w[j].x, x[0], x[1]);
    unpack_bf16(w[j].y, x[2], x[3]);
    unpack_bf16(w[j].z, x[4], x[5]);
    unpack_bf16(w[j].w, x[6], x[7]);
    const int e0 = (v0 + t + j * kLsThreads) * 8;
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (x[e] > m) {  // strictly greater: the first (lowest) index of the max stays; NaN never is
        m = x[e];
        idx = e0 + e;
      }
  }
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < kLsMaxVecs; ++j) {
    float x[8];
    unpack_bf16(w[j].x, x[0], x[1]);
    unpack_bf16(w[j].y, x[2], x[3]);
    unpack_bf16(w[j].z, x[4], x[5]);
    unpack_bf16(w[j].w, x[6], x[7]);
    if (m != -INFINITY) {
#pragma unroll
      for (int e = 0; e < 8; ++e) s += ex2((x[e] - m) * kLog2e);  // padding (-inf) adds 0; a NaN makes s NaN
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e)
        if (isnan(x[e])) s = NAN;
    }
  }
  if (piece == split - 1 && t < tail) {  // the last vocab % 8 logits
    const uint16_t bits = reinterpret_cast<const uint16_t*>(logits + row * ld)[nvec * 8 + t];
    const float x[1] = {__uint_as_float(static_cast<uint32_t>(bits) << 16)};
    lg_fold(x, nvec * 8 + t, m, s, idx);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
    const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
    lg_merge(m, s, idx, m2, s2, i2);
  }
  if (lane == 0) {
    red[warp][0] = m;
    red[warp][1] = s;
    red[warp][2] = __int_as_float(idx);
  }
  __syncthreads();
  if (warp == 0) {
    constexpr int kW = kLsThreads / 32;
    m = lane < kW ? red[lane][0] : -INFINITY;
    s = lane < kW ? red[lane][1] : 0.f;
    idx = lane < kW ? __float_as_int(red[lane][2]) : 0;
#pragma unroll
    for (int off = kW / 2; off > 0; off >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
      const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
      const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
      lg_merge(m, s, idx, m2, s2, i2);
    }
    if (split == 1 && lane == 0) {
      ids[row] = idx;
      conf[row] = m == -INFINITY ? 0.f : 1.f / s;
    }
  }
  if (split > 1) {
    cluster_wait();
    if (t == 0) {
      const uint32_t slot = smem_u32(&parts[piece][0]);
      st_dsmem_f32(dsmem_addr(slot, 0), m);
      st_dsmem_f32(dsmem_addr(slot + 4, 0), s);
      st_dsmem_f32(dsmem_addr(slot + 8, 0), __int_as_float(idx));
      mbar_arrive_remote_release(dsmem_addr(smem_u32(&arrived), 0));
    }
    if (cluster_ctarank() == 0 && warp == 0) {
      bool ok = true;
      if (lane == 0) ok = mbar_wait_cluster(&arrived, 0, err);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      m = -INFINITY;
      s = 0.f;
      idx = 0;
      if (ok && lane < split) {
        m = parts[lane][0];
        s = parts[lane][1];
        idx = __float_as_int(parts[lane][2]);
      }
#pragma unroll
      for (int off = 4; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
        const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
        lg_merge(m, s, idx, m2, s2, i2);
      }
      if (lane == 0 && ok) {
        ids[row] = idx;
        conf[row] = m == -INFINITY ? 0.f : 1.f / s;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// AR-diffusion ensemble verifier (appendix, verification with the ensemble):
// p = lambda softmax(ar) + (1 - lambda) softmax(diff); id = lowest argmax,
// conf = max p. Two passes over the row pair in one launch: the pieces of a
// row pair first fold both rows into (max, sum), merge them across the
// cluster (distributed shared memory), then re-read their pieces (now in L2)
// to evaluate p and keep its lowest-index maximum.
// ---------------------------------------------------------------------------

constexpr int kEnThreads = 256;

// (p, i) merge: the larger p, the lower index on ties.
__device__ __forceinline__ void en_merge(float& p, int& i, float p2, int i2) {
  if (p2 > p || (p2 == p && i2 < i)) {
    p = p2;
    i = i2;
  }
}

__global__ void __launch_bounds__(kEnThreads)
    ensemble_argmax_kernel(const __nv_bfloat16* __restrict__ ar, const __nv_bfloat16* __restrict__ diff, int vocab,
                           long ld, int split, float lambda, int32_t* __restrict__ ids, float* __restrict__ conf) {
  __shared__ float red[kEnThreads / 32][6];
  __shared__ float tot[4];  // rank 0: m_a, s_a, m_b, s_b of the row pair
  __shared__ float best[2];  // this CTA's (p, index)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, t = threadIdx.x;
  const int piece = static_cast<int>(blockIdx.x % split);
  const long row = static_cast<long>(blockIdx.x / split);
  const int nvec = vocab >> 3, tail = vocab & 7;
  const int per = (nvec + split - 1) / split;
  const int v0 = min(nvec, piece * per), v1 = min(nvec, v0 + per);
  const bool has_tail = piece == split - 1 && t < tail;
  grid_launch_dependents();
  grid_dependency_wait();  // the logits come from earlier kernels
  const uint4* ra = reinterpret_cast<const uint4*>(ar + row * ld);
  const uint4* rb = reinterpret_cast<const uint4*>(diff + row * ld);
  const uint16_t* ta = reinterpret_cast<const uint16_t*>(ar + row * ld) + nvec * 8;
  const uint16_t* tb = reinterpret_cast<const uint16_t*>(diff + row * ld) + nvec * 8;

  // ---- pass 1: (max, sum) of each row over this piece ----
  float ma = -INFINITY, sa = 0.f, mb = -INFINITY, sb = 0.f;
  int ia = 0, ib = 0;
  for (int v = v0 + t; v < v1; v += kEnThreads) {
    const uint4 wa = __ldg(ra + v), wb = __ldg(rb + v);
    float xa[8], xb[8];
    unpack_bf16(wa.x, xa[0], xa[1]); unpack_bf16(wa.y, xa[2], xa[3]);
    unpack_bf16(wa.z, xa[4], xa[5]); unpack_bf16(wa.w, xa[6], xa[7]);
    unpack_bf16(wb.x, xb[0], xb[1]); unpack_bf16(wb.y, xb[2], xb[3]);
    unpack_bf16(wb.z, xb[4], xb[5]); unpack_bf16(wb.w, xb[6], xb[7]);
    lg_fold(xa, v * 8, ma, sa, ia);
    lg_fold(xb, v * 8, mb, sb, ib);
  }
  if (has_tail) {
    const float xa[1] = {__uint_as_float(static_cast<uint32_t>(ta[t]) << 16)};
    const float xb[1] = {__uint_as_float(static_cast<uint32_t>(tb[t]) << 16)};
    lg_fold(xa, nvec * 8 + t, ma, sa, ia);
    lg_fold(xb, nvec * 8 + t, mb, sb, ib);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    lg_merge(ma, sa, ia, __shfl_xor_sync(0xffffffffu, ma, off), __shfl_xor_sync(0xffffffffu, sa, off),
             __shfl_xor_sync(0xffffffffu, ia, off));
    lg_merge(mb, sb, ib, __shfl_xor_sync(0xffffffffu, mb, off), __shfl_xor_sync(0xffffffffu, sb, off),
             __shfl_xor_sync(0xffffffffu, ib, off));
  }
  if (lane == 0) {
    red[warp][0] = ma; red[warp][1] = sa; red[warp][2] = mb; red[warp][3] = sb;
  }
  __syncthreads();
  if (warp == 0) {
    ma = lane < kEnThreads / 32 ? red[lane][0] : -INFINITY;
    sa = lane < kEnThreads / 32 ? red[lane][1] : 0.f;
    mb = lane < kEnThreads / 32 ? red[lane][2] : -INFINITY;
    sb = lane < kEnThreads / 32 ? red[lane][3] : 0.f;
#pragma unroll
    for (int off = 4; off > 0; off >>= 1) {
      lg_merge(ma, sa, ia, __shfl_xor_sync(0xffffffffu, ma, off), __shfl_xor_sync(0xffffffffu, sa, off), 0);
      lg_merge(mb, sb, ib, __shfl_xor_sync(0xffffffffu, mb, off), __shfl_xor_sync(0xffffffffu, sb, off), 0);
    }
    if (lane == 0) {
      tot[0] = ma; tot[1] = sa; tot[2] = mb; tot[3] = sb;
    }
  }
  if (split > 1) {
    cluster_sync();  // every piece's (max, sum) is in its shared memory
    if (cluster_ctarank() == 0 && warp == 0) {
      const uint32_t base = smem_u32(tot);
      ma = -INFINITY; sa = 0.f; mb = -INFINITY; sb = 0.f;
      if (lane < split) {
        ma = ld_dsmem_f32(dsmem_addr(base, lane));
        sa = ld_dsmem_f32(dsmem_addr(base + 4, lane));
        mb = ld_dsmem_f32(dsmem_addr(base + 8, lane));
        sb = ld_dsmem_f32(dsmem_addr(base + 12, lane));
      }
#pragma unroll
      for (int off = 4; off > 0; off >>= 1) {
        lg_merge(ma, sa, ia, __shfl_xor_sync(0xffffffffu, ma, off), __shfl_xor_sync(0xffffffffu, sa, off), 0);
        lg_merge(mb, sb, ib, __shfl_xor_sync(0xffffffffu, mb, off), __shfl_xor_sync(0xffffffffu, sb, off), 0);
      }
    }
    cluster_sync();  // every rank has read the pieces' states before rank 0 overwrites its own
    if (cluster_ctarank() == 0 && threadIdx.x == 0) {
      tot[0] = ma; tot[1] = sa; tot[2] = mb; tot[3] = sb;
    }
    cluster_sync();  // the row pair's totals are in rank 0's shared memory
    const uint32_t base0 = dsmem_addr(smem_u32(tot), 0);
    ma = ld_dsmem_f32(base0);
    sa = ld_dsmem_f32(base0 + 4);
    mb = ld_dsmem_f32(base0 + 8);
    sb = ld_dsmem_f32(base0 + 12);
  } else {
    __syncthreads();
    ma = tot[0]; sa = tot[1]; mb = tot[2]; sb = tot[3];
  }
  // An empty distribution (max -inf) gets weight 0 and a stand-in max of 0,
  // so its terms are exp(-inf) * 0 = 0.
  const float ca = ma == -INFINITY ? 0.f : lambda / sa;
  const float cb = mb == -INFINITY ? 0.f : (1.f - lambda) / sb;
  const float ma2 = (ma == -INFINITY ? 0.f : ma) * kLog2e;
  const float mb2 = (mb == -INFINITY ? 0.f : mb) * kLog2e;

  // ---- pass 2: p over this piece (re-read, now in L2), lowest-index max ----
  float pbest = -1.f;
  int ibest = 0;
  for (int v = v0 + t; v < v1; v += kEnThreads) {
    const uint4 wa = __ldg(ra + v), wb = __ldg(rb + v);
    float xa[8], xb[8];
    unpack_bf16(wa.x, xa[0], xa[1]); unpack_bf16(wa.y, xa[2], xa[3]);
    unpack_bf16(wa.z, xa[4], xa[5]); unpack_bf16(wa.w, xa[6], xa[7]);
    unpack_bf16(wb.x, xb[0], xb[1]); unpack_bf16(wb.y, xb[2], xb[3]);
    unpack_bf16(wb.z, xb[4], xb[5]); unpack_bf16(wb.w, xb[6], xb[7]);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float p = ca * ex2(fmaf(xa[j], kLog2e, -ma2)) + cb * ex2(fmaf(xb[j], kLog2e, -mb2));
      if (p > pbest) {
        pbest = p;
        ibest = v * 8 + j;
      }
    }
  }
  if (has_tail) {
    const float a = __uint_as_float(static_cast<uint32_t>(ta[t]) << 16);
    const float b = __uint_as_float(static_cast<uint32_t>(tb[t]) << 16);
    const float p = ca * ex2(fmaf(a, kLog2e, -ma2)) + cb * ex2(fmaf(b, kLog2e, -mb2));
    if (p > pbest) {
      pbest = p;
      ibest = nvec * 8 + t;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1)
    en_merge(pbest, ibest, __shfl_xor_sync(0xffffffffu, pbest, off), __shfl_xor_sync(0xffffffffu, ibest, off));
  if (lane == 0) {
    red[warp][4] = pbest;
    red[warp][5] = __int_as_float(ibest);
  }
  __syncthreads();
  if (warp == 0) {
    pbest = lane < kEnThreads / 32 ? red[lane][4] : -1.f;
    ibest = lane < kEnThreads / 32 ? __float_as_int(red[lane][5]) : 0;
#pragma unroll
    for (int off = 4; off > 0; off >>= 1)
      en_merge(pbest, ibest, __shfl_xor_sync(0xffffffffu, pbest, off), __shfl_xor_sync(0xffffffffu, ibest, off));
    if (lane == 0) {
      best[0] = pbest;
      best[1] = __int_as_float(ibest);
    }
  }
  if (split > 1) {
    cluster_sync();
    if (cluster_ctarank() == 0 && warp == 0) {
      const uint32_t base = smem_u32(best);
      pbest = -1.f;
      ibest = 0;
      if (lane < split) {
        pbest = ld_dsmem_f32(dsmem_addr(base, lane));
        ibest = __float_as_int(ld_dsmem_f32(dsmem_addr(base + 4, lane)));
      }
#pragma unroll
      for (int off = 4; off > 0; off >>= 1)
        en_merge(pbest, ibest, __shfl_xor_sync(0xffffffffu, pbest, off), __shfl_xor_sync(0xffffffffu, ibest, off));
      if (lane == 0) {
        ids[row] = ibest;
        conf[row] = pbest;
      }
    }
    cluster_sync();  // the peers keep their shared memory until rank 0 has read it
  } else if (threadIdx.x == 0) {
    ids[row] = ibest;
    conf[row] = pbest;
  }
}

}  // namespace

int logits_split_vectors() { return kLgStageVecs; }

cudaError_t launch_ensemble_argmax(const __nv_bfloat16* ar, const __nv_bfloat16* diff, int rows, int vocab, long ld,
                                   int split, float lambda, int32_t* ids, float* conf, cudaStream_t stream) {
  const dim3 grid(static_cast<unsigned>(static_cast<long>(rows) * split));
  return launch_kernel_cluster(ensemble_argmax_kernel, grid, dim3(kEnThreads), 0, stream, split, ar, diff, vocab, ld,
                               split, lambda, ids, conf);
}

cudaError_t launch_logits_argmax(const __nv_bfloat16* logits, int rows, int vocab, long ld, int split, int32_t* ids,
                                 float* conf, unsigned int* err, cudaStream_t stream) {
  static int configured[64] = {0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!__atomic_load_n(&configured[dev], __ATOMIC_ACQUIRE)) {
    e = cudaFuncSetAttribute(logits_argmax_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kLgSmemBytes);
    if (e != cudaSuccess) return e;
    __atomic_store_n(&configured[dev], 1, __ATOMIC_RELEASE);
  }
  const dim3 grid(static_cast<unsigned>(static_cast<long>(rows) * split));
  const long piece_vecs = ((vocab >> 3) + split - 1) / split;
  if (piece_vecs <= static_cast<long>(kLsThreads) * kLsMaxVecs)
    return launch_kernel_cluster(logits_argmax_small_kernel, grid, dim3(kLsThreads), 0, stream, split, logits, vocab,
                                 ld, split, ids, conf, err);
  return launch_kernel_cluster(logits_argmax_kernel, grid, dim3(kLgThreads), kLgSmemBytes, stream, split, logits,
                               vocab, ld, split, ids, conf, err);
}

}  // namespace nld
