// Block attention over a paged bf16 KV cache on the 5th-generation tensor
// cores (tcgen05, accumulators in tensor memory), for up to 256 packed query
// rows (Sec. 2.2 mask; Sec. 3 Modes 2 and 3).
//
// One CTA serves one (KV split, KV head g, sequence b): its G = Hq/Hkv query
// heads times the bl block tokens form R = G*bl <= 256 query rows in one or
// two 128-row MMA tiles, so each K/V page leaves HBM once per (b, g).
//
// Warp roles (5 + 4*MT*CG warps):
//   warps 0-2 and the last  TMA producers: the boxes of each 64-token K/V tile
//             (16 tokens x 64 dims each) dealt four ways into a ring of up to
//             8 stages (produce_kv), warps 0-1 the K boxes, the others the V
//             boxes (with two softmax groups each kind with its own full/empty
//             barriers, so that a K slot refills once its score product is
//             done); TMA issue cost is per warp, so four issuing warps land a
//             tile sooner.
//   warp 3    allocates the TMEM columns; lane 0 loads Q by TMA (one M tile)
//             and issues every MMA:
//               S_j = Q K^T     (M=128 rows, N=64*TPS tokens, K=D; double-buffered in TMEM)
//               O  += P_k V_k   (M=128 rows, N=D, K=64 tokens; V read MN-major)
//             S_{j+1} is issued before the PV products of S_j so the tensor
//             core computes the next scores while the softmax warps work.
//             Each MMA or commit instruction holds the issuing thread ~50
//             cycles (measured), so the one issuing thread is a serial
//             resource of the chain.
//   warps 4.. softmax: thread t owns TMEM lane 32*(warp%4)+lane, one query
//             row. It loads its S row, applies the mask and the base-2 scale,
//             keeps the running max and sum, writes P (bf16) back to TMEM
//             over the consumed S columns as the PV MMA's A operand, and at
//             the end reads O from TMEM, divides by the sum and stages its row
//             in the freed K/V ring in 128-byte-swizzled boxes, which one
//             thread writes with tiled TMA stores (the bf16 output or bf16
//             split partials, in packed row order).
//             With 33..64 packed rows, Q is replicated into the idle lane
//             quadrants (REP = 2): each copy of a row takes a 32-token slice
//             of every tile with its own running max and sum, so every
//             softmax warp works and each does half of the exponentials; the
//             copies are merged once, each finalising half of the columns.
//             With up to 32 or 65..128 rows (CG = 2) two groups of four
//             softmax warps share the TMEM lanes: group c takes tile 2j + c
//             of score product j. Both take the row max over both tiles (the
//             groups' tile maxima exchanged through shared memory), so they
//             hold the same running max and accumulate into one O; P has two
//             TMEM buffers of its own, so a score product waits only for the
//             softmax to have read the S buffer it overwrites, never for a
//             PV product.
// When the KV range of a (sequence, KV head) is split over a thread-block
// cluster, the CTAs stage their normalised rows in shared memory and merge
// them through distributed shared memory (a cluster barrier, then each CTA
// combines a slice of rows from all peers): the final output, or one partial
// per cluster, leaves the kernel instead of one partial per split.
// The running max is raised lazily: O is rescaled in TMEM only when a row's
// max grows by more than 2^8 (P then stays below 256, exact enough in bf16);
// the final division by the matching sum removes the reference max.
#pragma once
#include "nld_internal.cuh"

namespace nld {
namespace {

constexpr int kProducers = 4;
constexpr int kMmaWarp = 3;
constexpr int kSoftmaxWarp0 = 4;

// MT 128-row M tiles per CTA (MT = 2 for 129..256 packed rows); 4*MT
// softmax warps; TPS 64-token K/V tiles per score product. TPS = 2 (one M
// tile, a split short enough to sit in the ring whole): N = 128 products,
// which the tensor core runs at full rate (N = 64 at about half), and half
// as many steps in the chain S -> softmax -> PV. A long split streams with
// TPS = 1, where a stage frees after each tile and more of the ring stays
// in flight. P lives in TMEM over its consumed S columns, so the ring takes
// what shared memory the Q tiles leave (up to 8 stages): a streaming CTA's
// bandwidth is the bytes it has in flight over the DRAM latency, so every
// stage counts.
//
// CG softmax groups per M tile: with CG = 2 (one M tile of up to 128 rows
// without row copies, paired products) two groups of four warps share the
// TMEM lanes; group c takes tile 2j + c of each product j. Both groups take
// each row's max over both tiles (tile maxima exchanged through shared
// memory every step), so they keep the same running max and
// accumulate into one O (each keeps the sum of its own tiles, added once
// before the epilogue). TMEM: two S buffers, the one O, two P buffers of 64
// columns. Per product the tensor core runs 8 score MMAs of N = 128 and 8
// PV MMAs, each softmax thread exponentiates one 64-column tile, and a score
// product waits only for the softmax warps to have read its S buffer: the
// chain S -> softmax -> PV no longer holds the next score products back.
template <int MT, int TPS, int CG = 1>
struct TcCfg {
  static_assert(TPS == 1 || (TPS == 2 && MT == 1), "paired score products with one M tile");
  static_assert(CG == 1 || (CG == 2 && MT == 1 && TPS == 2), "two softmax groups: one M tile, paired products");
  static constexpr int kTPS = TPS;               // K/V tiles per score product
  static constexpr int kSTok = kTPS * kTileTok;  // tokens (N) of a score product
  static constexpr int kPBufs = 2 * kTPS;        // tiles in flight between the softmax and PV (barrier slots)
  static constexpr int kSmWarps = 4 * MT * CG;   // softmax warps
  static constexpr int kWarps = 5 + kSmWarps;    // 4 producers, 1 MMA, softmax
  static constexpr int kThreads = 32 * kWarps;
  static constexpr uint32_t kTmemCols = 512;     // MT x (S0 | S1), then MT x CG x O
  static_assert(2 * MT * kSTok + MT * CG * 128 <= 512, "TMEM columns");
};

// producer index of a warp, or -1: warps 0-2 and the last warp
template <int MT, int CG>
__device__ __forceinline__ int producer_index(int warp) {
  return warp < 3 ? warp : (warp == 4 + 4 * MT * CG ? 3 : -1);
}
constexpr float kRescaleLog2 = 8.0f;

// Epilogue staging in the freed K/V ring and Q tiles: 128*MT rows of D fp32
// (padded pitch), then 128*MT log2-sum-exp values, then the cluster merge
// weights [rows][8] and merged lse per row.
template <int D>
__host__ __device__ constexpr int merge_pitch() { return D * 4 + 16; }

// K/V ring: the K tiles column-block-major ([column block][stage], so that
// the K tiles of consecutive stages form one operand of 128 rows), then the
// V tiles stage-major ([stage][column block]).
template <int D, int MT, int TPS>
struct TcLayout {
  using Geo = TileGeom<D>;
  static constexpr int kPBufs = TcCfg<MT, TPS>::kPBufs;
  static constexpr int kQBytes = Geo::kColBlocks * 128 * 128;  // one 128-row Q tile, bf16
  // stages: what is left of 227 KB after Q, 512 bytes of barriers and the
  // 1024-byte alignment slack, a multiple of TPS, at most 8 (P lives in TMEM)
  static constexpr int kFitStages = (232448 - 1024 - 512 - 1536 - MT * kQBytes) / Geo::kStageBytes;
  static constexpr int kStages = (kFitStages < 8 ? kFitStages : 8) / TPS * TPS;
  static_assert(kStages >= 2 * TPS, "at least two score products in the ring");
  static constexpr int kVOff = kStages * Geo::kTileBytes;       // V tiles after the K tiles
  static constexpr int kQOff = kStages * Geo::kStageBytes;
  static constexpr int kPOff = kQOff + MT * kQBytes;  // end of the ring and Q tiles
  static constexpr int kBarOff = kPOff;
  // k_full[st], v_full[st], k_empty[st], v_empty[st], s_full[2], s_free[2], p_full[kPBufs], o_done[kPBufs],
  // q_ready, q_full, drain, o_fin, xm_full[2], tmem slot
  static constexpr int kNumBars = 4 * kStages + 4 + 2 * kPBufs + 4 + 2;
  static_assert(kNumBars * 8 + 16 <= 512, "barrier reserve");
  // two softmax groups: each row's score max per group, truncated to 24 bits
  // (high 16 bits [2][group][TMEM lane], then the next 8 bits, same order),
  // exchanged every step (two buffers by step parity)
  static constexpr int kXmOff = kBarOff + 512;
  static constexpr int kXmLoOff = kXmOff + 2 * 2 * 128 * 2;
  static constexpr int kBytes = kXmLoOff + 2 * 2 * 128;
  static_assert(kBytes + 1024 <= 232448, "shared memory per CTA");
  static constexpr int kMergeRows = 128 * MT;
  static constexpr int kLseOff = kMergeRows * merge_pitch<D>();
  static constexpr int kWtsOff = kLseOff + kMergeRows * 4;
  static constexpr int kLseOutOff = kWtsOff + kMergeRows * 8 * 4;
  static_assert(kLseOutOff + kMergeRows * 4 <= kPOff, "epilogue staging overlaps the live buffers");
  // copies of a row (REP > 1) exchange their O column ranges here
  static constexpr int kXchgOff = (kLseOutOff + kMergeRows * 4 + 15) / 16 * 16;
  // output boxes for the tiled stores (128-byte rows, 1024-byte aligned)
  static_assert(D / 64 * kMergeRows * 128 <= kPOff, "output staging");
};

// The sequence of rank blockIdx.z by prefix length (descending, ties by
// index), computed by the whole CTA in `scratch` (2 * B ints of shared
// memory). Out of line, so that kernels that never take it keep their code.
__device__ __noinline__ int sequence_by_length_rank(const AttnArgs& a, int* scratch) {
  int* lens = scratch;
  int* order = scratch + a.B;
  for (int t = threadIdx.x; t < a.B; t += blockDim.x) lens[t] = __ldg(a.prefix_lens + t);
  __syncthreads();
  for (int t = threadIdx.x; t < a.B; t += blockDim.x) {
    const int lt = lens[t];
    int rank = 0;
    for (int u = 0; u < a.B; ++u) {
      const int lu = lens[u];
      rank += (lu > lt || (lu == lt && u < t)) ? 1 : 0;
    }
    order[rank] = t;
  }
  __syncthreads();
  return order[blockIdx.z];
}

template <int D, int MT, int REP, int TPS, bool MASKED, bool ORDERED, int CG>
__global__ void __launch_bounds__(TcCfg<MT, TPS, CG>::kThreads, 1)
    block_attn_tc_kernel(const __grid_constant__ TmaMaps maps, const AttnArgs a) {
  static_assert(REP == 1 || REP == 2, "replication of 1 or 2 (up to 32 rows run on two softmax groups)");
  static_assert(MT == 1 || REP == 1, "replication only with one M tile");
  static_assert(CG == 1 || REP == 1, "softmax groups without row copies");
  using Geo = TileGeom<D>;
  using Cfg = TcCfg<MT, TPS, CG>;
  using Lay = TcLayout<D, MT, TPS>;
  constexpr int kTcStages = Lay::kStages;
  // Ring barriers. With two softmax groups (65..128 rows, a split of its own
  // or a block-slot chunk pair) K and V slots fill and free on their own
  // barriers, so a K slot is refilled as soon as the score product that read
  // it has completed and the K boxes of the early tiles go out first; the
  // kernels with one group (row copies, two M tiles) keep one barrier per
  // stage for K and V together, freed by the PV product. Each scheme
  // measured faster on its own kernels (the split scheme: long prefix +4%,
  // 14B chunk pairs +10% once the score products stopped waiting for the PV
  // products; the joint one: concurrency sweep +6%).
  constexpr bool kSplitKV = CG == 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* q_s = smem + Lay::kQOff;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Lay::kBarOff);
  uint64_t* k_full = bars;                   // K (one-group kernels: K and V) slot of stage st landed
  uint64_t* v_full = bars + kTcStages;       // V slot of stage st landed (split scheme)
  uint64_t* k_empty = bars + 2 * kTcStages;  // the product that read K (one group: the PV product) of stage st completed
  uint64_t* v_empty = bars + 3 * kTcStages;  // the PV product that read V of stage st completed (split scheme)
  uint64_t* s_full = bars + 4 * kTcStages;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* o_done = p_full + Cfg::kPBufs;
  uint64_t* q_ready = o_done + Cfg::kPBufs;
  uint64_t* q_full = q_ready + 1;  // the Q tiles' TMA copies (one M tile)
  uint64_t* drain = q_full + 1;
  // o_fin (two softmax groups): every PV product has completed (committed
  // once, after the last). With one group every softmax warp waits on the
  // last o_done phase.
  uint64_t* o_fin = drain + 1;
  // xm_full[b] (two softmax groups): every softmax warp has written its rows'
  // score maxima of the step with parity b
  uint64_t* xm_full = o_fin + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xm_full + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // Block-slot chunks (a.nh = 2 for 129..256 packed rows): the two CTAs of
  // a (split, KV head, sequence) are adjacent along x and hold block slots
  // [hc*bl_c, (hc+1)*bl_c) of the G heads each, R = G*bl_c rows. A chunk
  // holds 65..128 rows, so only the two-group kernels see nh = 2.
  const int nh = CG == 2 ? a.nh : 1;
  const int split = static_cast<int>(blockIdx.x) / nh, g = blockIdx.y;
  const int slot0 = (static_cast<int>(blockIdx.x) - split * nh) * a.bl_c;  // first block slot of this CTA

  if (threadIdx.x == 0) {
    for (int s = 0; s < kTcStages; ++s) {
      // one expect_tx arrival per producer warp (of the kind, split scheme)
      mbar_init(&k_full[s], kSplitKV ? kProducers / 2 : kProducers);
      mbar_init(&k_empty[s], 1);
      if (kSplitKV) {
        mbar_init(&v_full[s], kProducers / 2);
        mbar_init(&v_empty[s], 1);
      }
    }
    for (int j = 0; j < 2; ++j) {
      mbar_init(&s_full[j], 1);
      mbar_init(&s_free[j], Cfg::kSmWarps);
    }
    for (int j = 0; j < Cfg::kPBufs; ++j) {
      // one group: the four warps of an M tile per tile; two groups: all
      // eight softmax warps per score product (p_full[j % 2])
      mbar_init(&p_full[j], CG == 2 ? Cfg::kSmWarps : 4 * MT);
      mbar_init(&o_done[j], 1);
    }
    mbar_init(q_ready, Cfg::kSmWarps);
    mbar_init(q_full, 1);
    mbar_init(drain, 1);
    if (CG == 2) {
      mbar_init(o_fin, 1);
      mbar_init(&xm_full[0], Cfg::kSmWarps);
      mbar_init(&xm_full[1], Cfg::kSmWarps);
    }
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&maps.k);
    prefetch_tensormap(&maps.v);
    prefetch_tensormap(&maps.o);
    if (MT == 1) prefetch_tensormap(&maps.q);
  }
  if (warp == kMmaWarp) {
    tmem_alloc(tmem_slot, Cfg::kTmemCols);
    tc_fence_before();
  }
  // Without NLD_ATTN_PREFIX_READY nothing global is read before the
  // dependency wait. With it, the page table, the prefix lengths and
  // prefix-only K/V tiles are read first, and only the block slots, Q and the
  // outputs wait (producers: in produce_kv; softmax warps: before Q).
  const bool early = a.prefix_ready != 0;
  grid_launch_dependents();  // dependents launch early; they wait on this grid themselves
  if (!early) grid_dependency_wait();
  // ORDERED (one split per sequence and more (sequence, KV head) units than
  // SMs): CTAs start in z order, so CTA z takes the sequence of rank z by
  // prefix length and the last wave holds the short ones. The ranks are
  // computed in the K/V ring, before any copy into it. A separate
  // instantiation, so the other kernels keep b = blockIdx.z.
  const int b = ORDERED ? sequence_by_length_rank(a, reinterpret_cast<int*>(smem)) : static_cast<int>(blockIdx.z);
  const int t_begin = split * a.chunk;
  // The producers' first page-id loads and the prefix-length load are
  // independent, so they are in flight together.
  PagePrefetch first;
  first.raw = 0;
  if (producer_index<MT, CG>(warp) >= 0) first.load(a, b, t_begin, 0, lane);
  int L = __ldg(a.prefix_lens + b);
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // TMEM columns: S of M tile mt, buffer j at (2*mt + j)*kSTok; then the O
  // accumulators, one per M tile; with two softmax groups one O shared by
  // both groups, then two P buffers of 64 columns (P of score product j in
  // buffer j % 2, tile 2j + h at column h*32).
  constexpr int kTPS = Cfg::kTPS;
  constexpr int kSTok = Cfg::kSTok;
  constexpr int kPBufs = Cfg::kPBufs;
  auto tS = [&](int mt, int j) -> uint32_t { return tmem + static_cast<uint32_t>((2 * mt + j) * kSTok); };
  auto tO = [&](int mt) -> uint32_t { return tmem + static_cast<uint32_t>(2 * MT * kSTok + mt * D); };
  auto tP = [&](int jb) -> uint32_t { return tmem + static_cast<uint32_t>(2 * kSTok + D + jb * kTileTok); };
  static_assert(CG == 1 || 2 * kSTok + D + 2 * kTileTok <= static_cast<int>(Cfg::kTmemCols), "TMEM columns");

  const int lmax = a.max_pages * a.page_size - a.bl;
  if (L < 0 || L > lmax) {
    if (threadIdx.x == 0) atomicOr(a.err, NLD_DEVERR_PREFIX_RANGE);
    L = min(max(L, 0), lmax);
  }
  const int N = L + a.bl;
  const float scl = a.scale_log2;
  const bool diff_mode = a.mode == NLD_MODE_DIFFUSION;
  const int t_end = min(t_begin + a.chunk, N);
  const int ntiles = t_begin < t_end ? (t_end - t_begin + kTileTok - 1) / kTileTok : 0;

  if (ntiles == 0) {
    // This split lies past the sequence: its partials carry no keys.
    if (early) grid_dependency_wait();
    if (a.csize > 1) {
      float* lse_stage = reinterpret_cast<float*>(smem + Lay::kLseOff);
      for (int r = threadIdx.x; r < Lay::kMergeRows; r += blockDim.x) lse_stage[r] = -INFINITY;
    } else {
      for (int r = threadIdx.x; r < a.R; r += blockDim.x) {
        const int i = slot0 + r / a.G, h = g * a.G + (r - (r / a.G) * a.G);
        a.lse_part[((static_cast<size_t>(split) * a.B + b) * a.Hq + h) * a.bl + i] = -INFINITY;
      }
    }
  } else if (producer_index<MT, CG>(warp) >= 0) {
    // ---------------- producers ----------------
    int early_tiles = 0;  // leading tiles made of prefix tokens only
    if (early) {
      while (early_tiles < kTcStages && early_tiles < ntiles &&
             min(t_begin + (early_tiles + 1) * kTileTok, t_end) <= L)
        ++early_tiles;
      if (early_tiles == 0) grid_dependency_wait();
    }
    const int pw = producer_index<MT, CG>(warp);
    const int issued = produce_kv<D, kSplitKV>(a, &maps.k, &maps.v, smem, k_full, v_full, k_empty, v_empty, kTcStages,
                                               g, b, t_begin, t_end, ntiles, lane, pw, kProducers, first, early_tiles);
    if (lane == 0 && issued < ntiles) {
      // Stopped early on a wait timeout: let the copies already issued land
      // before the CTA exits (bounded).
      uint64_t* full = kSplitKV && pw >= kProducers / 2 ? v_full : k_full;
      for (int k = max(0, issued - kTcStages); k < issued; ++k)
        mbar_wait(&full[k % kTcStages], (k / kTcStages) & 1, a.err);
    }
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      if constexpr (MT == 1) {
        // Q by TMA, straight after the dependency wait: per column block one
        // box of the CTA's R rows (G heads x bl slots, in packed row order),
        // written once per copy.
        if (early) grid_dependency_wait();
        mbar_arrive_expect_tx(q_full, static_cast<uint32_t>(REP * (D / 64) * a.R * 128));
#pragma unroll
        for (int q = 0; q < REP; ++q)
#pragma unroll
          for (int cb = 0; cb < D / 64; ++cb)
            tma_load_3d(q_s + cb * (128 * 128) + q * (128 / REP) * 128, &maps.q, q_full, cb * 64, g * a.G,
                        b * a.bl + slot0);
      }
      bool ok = mbar_wait(q_ready, 0, a.err);
      if constexpr (MT == 1) ok = ok && mbar_wait(q_full, 0, a.err);
      tc_fence_after();
      const uint32_t q_addr = smem_u32(q_s);
      const uint32_t idesc_s = umma_idesc_bf16(128, kSTok, false);
      const uint32_t idesc_o = umma_idesc_bf16(128, D, true);
      // Score product j: tiles kTPS*j .. kTPS*j+kTPS-1, whose K tiles sit in
      // consecutive stages (one operand of kSTok rows per column block). If
      // the last product has a single tile, its second half reads a stage
      // no tile of this CTA still needs; those columns are never used.
      auto issue_s = [&](int j) {
        const int st = (j * kTPS) % kTcStages;
        const uint32_t k_addr = smem_u32(smem) + static_cast<uint32_t>(st * Geo::kColBlockBytes);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          const uint32_t d = tS(mt, j & 1);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t koff = (kk & 3) * 32;  // 16 elements along the 128-byte row
            const int cb = kk >> 2;               // 64-dim column block
            const uint64_t ad = sw128_desc(q_addr + mt * Lay::kQBytes + cb * (128 * 128) + koff, 0, 1024);
            const uint64_t bd = sw128_desc(k_addr + cb * kTcStages * Geo::kColBlockBytes + koff, 0, 1024);
            umma_bf16(d, ad, bd, idesc_s, kk > 0 ? 1u : 0u);
          }
        }
        umma_commit(&s_full[j & 1]);
        // Split scheme: the K slots of this product are free once it
        // completes (a last product with one tile frees only that tile's slot).
        if (kSplitKV) {
          umma_commit(&k_empty[st]);
          if (kTPS == 2 && j * kTPS + 1 < ntiles) umma_commit(&k_empty[(st + 1) % kTcStages]);
        }
      };
      // One softmax group: P of tile h of a product starts at S column h*32
      // (one warp reads the whole product's columns before writing).
      constexpr int kPCols = kTileTok / 2;
      auto issue_pv = [&](int k) {
        const int st = k % kTcStages;
        const uint32_t v_addr = smem_u32(smem + Lay::kVOff + st * Geo::kTileBytes);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          // A = P in TMEM (bf16 pairs, 32 columns per 64-token tile, over S
          // columns its tile's softmax has consumed); B = V (MN-major: 64-dim
          // atoms LBO apart, 8-token row groups SBO apart).
          const uint32_t p_tmem = tS(mt, (k / kTPS) & 1) + static_cast<uint32_t>((k % kTPS) * kPCols);
          const uint32_t o_acc = tO(mt);
#pragma unroll
          for (int kt = 0; kt < kTileTok / 16; ++kt) {
            const uint64_t bd = sw128_desc(v_addr + kt * 16 * 128, Geo::kColBlockBytes, 1024);
            umma_bf16_ts(o_acc, p_tmem + kt * 8, bd, idesc_o, (k > 0 || kt > 0) ? 1u : 0u);
          }
        }
        umma_commit(&o_done[k % kPBufs]);
        umma_commit(kSplitKV ? &v_empty[st] : &k_empty[st]);
      };
      // Event-driven issue: score product j needs its K tiles and a free S
      // buffer (the softmax warps have read product j-2), and waits until
      // the PV products of product j-2 are issued; PV_k needs P_k and the V
      // tile of stage k. Whichever
      // is ready goes first, so a late K/V tile never holds back a ready PV.
      // (Letting scores run further ahead measured slower: they queue in
      // front of the PV products on the tensor core.)
      const int nprod = (ntiles + kTPS - 1) / kTPS;
      int next_s = 0, next_pv = 0;
      // The time limit bounds one stall, not the split: it restarts whenever
      // an MMA group is issued.
      uint64_t t_start = global_timer_ns();
      uint32_t spins = 0;
      if constexpr (CG == 2) {
        // Two softmax groups: P has TMEM columns of its own, so score product
        // j waits only for its K tiles and for the softmax warps to have read
        // product j - 2 from the S buffer it overwrites, and runs up to two
        // products ahead of the softmax. The PV products of product j (both
        // tiles into the one O) wait for P_j from all eight softmax warps and,
        // split scheme, for the V tiles. Each tile's PV commits its stage's
        // empty barrier, which the softmax warps also read as "PV of this
        // tile completed".
        auto issue_pv2 = [&](int j) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int k = 2 * j + h;
            if (k >= ntiles) break;
            const int st = k % kTcStages;
            const uint32_t v_addr = smem_u32(smem + Lay::kVOff + st * Geo::kTileBytes);
            const uint32_t p_tmem = tP(j & 1) + static_cast<uint32_t>(h * (kTileTok / 2));
#pragma unroll
            for (int kt = 0; kt < kTileTok / 16; ++kt) {
              const uint64_t bd = sw128_desc(v_addr + kt * 16 * 128, Geo::kColBlockBytes, 1024);
              umma_bf16_ts(tO(0), p_tmem + kt * 8, bd, idesc_o, (k > 0 || kt > 0) ? 1u : 0u);
            }
            umma_commit(kSplitKV ? &v_empty[st] : &k_empty[st]);
          }
          if (j == nprod - 1) umma_commit(o_fin);
        };
        int next_p = 0;
        while (ok && next_p < nprod) {
          bool progressed = false;
          const int t0 = 2 * next_s;
          if (next_s < nprod && mbar_test(&k_full[t0 % kTcStages], (t0 / kTcStages) & 1) &&
              (t0 + 1 >= ntiles || mbar_test(&k_full[(t0 + 1) % kTcStages], ((t0 + 1) / kTcStages) & 1)) &&
              (next_s < 2 || mbar_test(&s_free[next_s & 1], ((next_s - 2) >> 1) & 1))) {
            tc_fence_after();
            issue_s(next_s++);
            progressed = true;
          }
          const int p0 = 2 * next_p;
          if (next_p < next_s && mbar_test(&p_full[next_p & 1], (next_p >> 1) & 1) &&
              (!kSplitKV || (mbar_test(&v_full[p0 % kTcStages], (p0 / kTcStages) & 1) &&
                             (p0 + 1 >= ntiles ||
                              mbar_test(&v_full[(p0 + 1) % kTcStages], ((p0 + 1) / kTcStages) & 1))))) {
            tc_fence_after();
            issue_pv2(next_p++);
            progressed = true;
          }
          if (progressed) {
            if (spins != 0) {
              spins = 0;
              t_start = global_timer_ns();
            }
          } else {
            __nanosleep(20);
            if ((++spins & 255u) == 0 && global_timer_ns() - t_start > kWaitLimitNs) {
              atomicOr(a.err, NLD_DEVERR_WAIT_TIMEOUT);
              ok = false;
            }
          }
        }
      }
      while (CG == 1 && ok && next_pv < ntiles) {
        bool progressed = false;
        const int t0 = next_s * kTPS;  // first tile of the next score product
        if (next_s < nprod && t0 - kTPS <= next_pv &&
            mbar_test(&k_full[t0 % kTcStages], (t0 / kTcStages) & 1) &&
            (kTPS == 1 || t0 + 1 >= ntiles || mbar_test(&k_full[(t0 + 1) % kTcStages], ((t0 + 1) / kTcStages) & 1)) &&
            (next_s < 2 || mbar_test(&s_free[next_s & 1], ((next_s - 2) >> 1) & 1))) {
          tc_fence_after();
          issue_s(next_s++);
          progressed = true;
        }
        if (next_pv < next_s * kTPS && mbar_test(&p_full[next_pv % kPBufs], (next_pv / kPBufs) & 1) &&
            (!kSplitKV || mbar_test(&v_full[next_pv % kTcStages], (next_pv / kTcStages) & 1))) {
          tc_fence_after();
          issue_pv(next_pv++);
          progressed = true;
        }
        if (progressed) {
          if (spins != 0) {
            spins = 0;
            t_start = global_timer_ns();
          }
        } else {
          __nanosleep(20);  // this warp shares an SM sub-partition with a softmax warp
          if ((++spins & 255u) == 0 && global_timer_ns() - t_start > kWaitLimitNs) {
            atomicOr(a.err, NLD_DEVERR_WAIT_TIMEOUT);
            ok = false;
          }
        }
      }
      if (!ok) {
        // Let every MMA already issued finish before TMEM is released (bounded).
        umma_commit(drain);
        mbar_wait(drain, 0, a.err);
      }
    }
    __syncwarp();
  } else {
    // ---------------- softmax warps ----------------
    // Warp `quad` reads TMEM lanes 32*quad..+31. With REP > 1 those lanes hold
    // a copy of row block rq = quad % kRowQuads and the warp takes the token
    // slice cp = quad / kRowQuads (columns c0u .. c0u+kColsU-1) of every step.
    constexpr int kRowQuads = 4 / REP;
    // Softmax steps: one tile, or with paired score products and copies
    // (TPS = 2, REP >= 2) the whole product, so that a step's columns per
    // thread stay at most 64 and its work is one max and one exponential pass.
    constexpr int kU = (kTPS == 2 && REP >= 2) ? 2 : 1;  // tiles per softmax step
    constexpr int kColsU = kU * kTileTok / REP;          // S columns per thread and step
    const int quad = warp & 3;
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int mt = CG == 1 ? wg : 0;                // M tile of this warp
    const int cg = CG == 1 ? 0 : wg;                // softmax group: tile 2j + cg of score product j
    const int part = CG == 1 ? quad / kRowQuads : cg;  // this thread's share of a row's state (copy or group)
    const int rq = quad % kRowQuads;                // row block
    const int cp = quad / kRowQuads;                // token slice
    const int c0u = cp * kColsU;           // first column of this thread's slice of a step
    const int h_own = c0u / kTileTok;      // the step's tile holding the slice
    const int lc0 = c0u % kTileTok;        // first column of the slice within that tile
    const int r_loc = quad * 32 + lane;             // TMEM lane == row of the Q and P tiles
    const int r = mt * 128 + rq * 32 + lane;        // packed query row
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const bool warp_rows = mt * 128 + rq * 32 < a.R;  // warp-uniform: the warp holds a real row
    const bool row_ok = r < a.R;
    const int row_i = slot0 + r / a.G;                    // block slot of this row
    const int row_h = g * a.G + (r - (r / a.G) * a.G);
    const int sm_tid = threadIdx.x - 32 * kSoftmaxWarp0;  // 0 .. 32*kSmWarps-1 across the softmax warps
    const int grp_tid = sm_tid - cg * 128 * MT;           // 0 .. 128*MT-1 within this softmax group
    const int swz = r_loc & 7;                      // 128-byte swizzle phase of this tile row
    uint8_t* q_tile = q_s + mt * Lay::kQBytes;

    // Q rows in shared memory, 128-byte-swizzled K-major (padding rows zero).
    // One M tile: the MMA warp brings Q by TMA and the rows past R are zeroed
    // here, before the dependency wait. Two M tiles: slice 0 of each row loads
    // it here after the wait and writes every copy.
    if (MT == 1 && !row_ok && cg == 0) {
#pragma unroll
      for (int c = 0; c < D / 8; ++c)
        *reinterpret_cast<uint4*>(q_tile + (c >> 3) * (128 * 128) + r_loc * 128 + (((c & 7) ^ swz) << 4)) =
            make_uint4(0, 0, 0, 0);
    }
    if (MT == 2 && early) grid_dependency_wait();
    {
      if (MT == 2 && cp == 0) {
        const uint4* qrow = reinterpret_cast<const uint4*>(
            a.q + ((static_cast<size_t>(b) * a.bl + row_i) * a.Hq + row_h) * D);
        uint4 v[D / 8];
#pragma unroll
        for (int c = 0; c < D / 8; ++c) v[c] = row_ok ? __ldg(qrow + c) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int q = 0; q < REP; ++q) {
          const int rl = r_loc + q * kRowQuads * 32;  // TMEM lane of copy q (same swizzle phase)
#pragma unroll
          for (int c = 0; c < D / 8; ++c)
            *reinterpret_cast<uint4*>(q_tile + (c >> 3) * (128 * 128) + rl * 128 + (((c & 7) ^ swz) << 4)) = v[c];
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_ready);
    }

    if (MT == 1 && early) grid_dependency_wait();  // before the mask table and the outputs

    // The keys this row may see inside [t_begin, t_end) are exactly t < lim
    // (Sec. 2.2: the whole prefix; in the draft pass every block slot, in the
    // verify pass the block slots up to the row's own), so a step's visible
    // columns are a leading run of them, one compare to find; a step whose
    // columns a whole warp sees skips the mask.
    const int lim = diff_mode ? t_end : min(t_end, L + row_i + 1);
    // MASKED (a table mask, e.g. quadratic self-speculation's, Sec. 3): the
    // prefix and the block slots whose bit is set in this row's table entry;
    // per step one 64-bit column mask, tested bit by bit. A separate
    // instantiation, so the two passes above keep their one compare.
    uint32_t rowbits = 0u;
    if constexpr (MASKED) rowbits = row_ok ? __ldg(a.block_mask + row_i) : 0u;
    const int plim = min(t_end, L);  // prefix keys of this split end here
    auto column_mask = [&](int col0) -> uint64_t {  // col0: token of this thread's first column
      const int np = min(max(plim - col0, 0), kColsU);
      uint64_t vis = np >= 64 ? ~0ull : (1ull << np) - 1ull;
      const int off = col0 - L;  // block slot of column 0
      if (off < a.bl && off + kColsU > 0) {
        uint64_t bb = off >= 0 ? static_cast<uint64_t>(rowbits) >> off : static_cast<uint64_t>(rowbits) << -off;
        const int nvalid = min(max(t_end - col0, 0), kColsU);
        bb &= nvalid >= 64 ? ~0ull : (1ull << nvalid) - 1ull;
        vis |= bb;
      }
      return vis;
    };
    // A wait that gives up does so for the whole warp, so that no lane skips
    // a warp-collective TMEM instruction the others execute.
    auto warp_wait = [&](uint64_t* bar, uint32_t parity) {
      return __all_sync(0xffffffffu, mbar_wait(bar, parity, a.err));
    };
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    if constexpr (CG == 2) {
      // Two softmax groups over every score product j: group c takes tile
      // 2j + c. The row max of a step is taken over both tiles of the product
      // (each group's tile max, exchanged through shared memory), so the two
      // groups hold the same running max and accumulate into one shared O;
      // each keeps the sum of its own tiles. P_j goes to P buffer
      // j % 2 once the PV products of product j - 2 (which read that buffer)
      // have completed; every warp waits for that before it hands product j
      // over, so no warp is ever two products ahead on p_full. The empty
      // barrier of a tile's stage (committed after its PV product) tells the
      // softmax warps that PV has completed; a parity wait on it is exact
      // because every earlier phase of that barrier was waited for two steps
      // before.
      const int nprod = (ntiles + 1) / 2;
      uint64_t* pv_done = kSplitKV ? v_empty : k_empty;
      for (int j = 0; j < nprod; ++j) {
        const int k = 2 * j + cg;        // this group's tile
        const bool has = k < ntiles;     // warp-uniform (the last product may hold one tile)
        const int t_own = t_begin + k * kTileTok;
        if (!warp_wait(&s_full[j & 1], (j >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float s[kTileTok];
        constexpr uint64_t kAll = ~0ull;
        auto vis_of = [&](int col0) -> uint64_t {
          if constexpr (MASKED) {
            return column_mask(col0);
          } else {
            const int nv = lim - col0;
            return nv >= 64 ? ~0ull : nv <= 0 ? 0ull : (1ull << nv) - 1ull;
          }
        };
        if (warp_rows && has) tmem_ld64(tS(0, j & 1) + lane_off + static_cast<uint32_t>(cg * kTileTok), s);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[j & 1]);

        // The row max of the product: this group's tile max, truncated to 24
        // bits (toward zero: relative error below 2^-15), exchanged with the
        // other group through shared memory; both groups take the max of the
        // two truncated values, so they agree exactly. The max only offsets
        // the exponent: the largest P is 2^d with d below 2^-15 of the
        // scaled max, which rounds to exactly 1 in bf16 while the scaled max
        // is below ~90, as with the untruncated max.
        uint16_t* xm = reinterpret_cast<uint16_t*>(smem + Lay::kXmOff) + (j & 1) * 256;  // [group][TMEM lane]
        uint8_t* xm_lo = smem + Lay::kXmLoOff + (j & 1) * 256;
        float own = -INFINITY;
        if (warp_rows) {
          if (has) {
            const uint64_t vis = vis_of(t_own);
            if (!__all_sync(0xffffffffu, vis == kAll)) {
#pragma unroll
              for (int e = 0; e < kTileTok; ++e) s[e] = ((vis >> e) & 1ull) ? s[e] : -INFINITY;
            }
            float pm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
            for (int e = 0; e < kTileTok; e += 8) {
#pragma unroll
              for (int q = 0; q < 4; ++q) pm[q] = fmax3(pm[q], s[e + 2 * q], s[e + 2 * q + 1]);
            }
            own = fmax3(pm[0], pm[1], fmaxf(pm[2], pm[3]));
          }
          const uint32_t own_t = __float_as_uint(own) & 0xFFFFFF00u;
          own = __uint_as_float(own_t);
          xm[cg * 128 + r_loc] = static_cast<uint16_t>(own_t >> 16);
          xm_lo[cg * 128 + r_loc] = static_cast<uint8_t>(own_t >> 8);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&xm_full[j & 1]);
        if (!warp_wait(&xm_full[j & 1], (j >> 1) & 1)) {
          ok = false;
          break;
        }
        float alpha = 1.f;
        bool rescale = false;
        if (warp_rows) {
          const float oth = __uint_as_float((static_cast<uint32_t>(xm[(1 - cg) * 128 + r_loc]) << 16) |
                                            (static_cast<uint32_t>(xm_lo[(1 - cg) * 128 + r_loc]) << 8));
          const float mx = fmaxf(own, oth) * scl;  // base-2 units, both tiles
          if (m_run == -INFINITY) {
            m_run = mx;
          } else if (mx > m_run + kRescaleLog2) {
            alpha = ex2(m_run - mx);
            m_run = mx;
            l_run *= alpha;
            rescale = true;
          }
        }
        if (__any_sync(0xffffffffu, rescale)) {
          // The shared O holds the PV products of products < j: wait for the
          // last of them (tile 2j - 1; j >= 1 here), then this group scales
          // its half of O's columns for this warp's rows.
          const int kl = 2 * j - 1;
          if (!warp_wait(&pv_done[kl % kTcStages], (kl / kTcStages) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (lane == 0 && cg == 0) atomicAdd(a.rescales, 1ull);
#pragma unroll 1
          for (int c = 0; c < D / 64; ++c) {
            float o[32];
            const uint32_t ta = tO(0) + lane_off + static_cast<uint32_t>(cg * (D / 2) + c * 32);
            tmem_ld32(ta, o);
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= alpha;
            tmem_st32(ta, o);
          }
        }
        if (j >= 2) {
          // P buffer j % 2 is free once the PV products of product j - 2
          // (last tile 2j - 3) have completed. Every warp waits, with rows
          // or not: a warp that skipped it could run ahead and arrive on
          // p_full[j % 2] for product j + 2 before the others had arrived
          // for product j, releasing PV_j early.
          const int kp = 2 * j - 3;
          if (!warp_wait(&pv_done[kp % kTcStages], (kp / kTcStages) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        if (warp_rows && has) {
          const float nmu = m_run == -INFINITY ? 0.f : -m_run;
          const float2 sc2 = make_float2(scl, scl), nm2 = make_float2(nmu, nmu);
          float2 ls[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
          const uint32_t tp = tP(j & 1) + lane_off + static_cast<uint32_t>(cg * (kTileTok / 2));
#pragma unroll
          for (int c = 0; c < kTileTok / 16; ++c) {
            uint32_t w[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float2 x = fma2(make_float2(s[c * 16 + 2 * e], s[c * 16 + 2 * e + 1]), sc2, nm2);
              const float2 pp = make_float2(ex2(x.x), ex2(x.y));
              ls[e & 1] = add2(ls[e & 1], pp);
              w[e] = pack_bf16(pp.x, pp.y);
            }
            tmem_st_u32<8>(tp + static_cast<uint32_t>(c * 8), w);
          }
          l_run += (ls[0].x + ls[0].y) + (ls[1].x + ls[1].y);
          tmem_wait_st();
        }
        if (has) {
          const int valid = t_end - t_own;
          if (valid < kTileTok && (valid & (kGroupTok - 1))) {
            // V rows past the sequence end inside its last page: zero them
            // (P is 0 there, but 0 * NaN = NaN).
            const int st = k % kTcStages;
            if (!warp_wait(kSplitKV ? &v_full[st] : &k_full[st], (k / kTcStages) & 1)) {
              ok = false;
              break;
            }
            const int r0 = valid, r1 = (valid + kGroupTok - 1) & ~(kGroupTok - 1);
            uint8_t* vt = smem + Lay::kVOff + st * Geo::kTileBytes;
            for (int idx = grp_tid; idx < (r1 - r0) * (D / 8); idx += 128) {
              const int row = r0 + idx / (D / 8), c = idx % (D / 8);
              *reinterpret_cast<uint4*>(vt + kv_swz(row, c)) = make_uint4(0, 0, 0, 0);
            }
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[j & 1]);
      }
    }
    // One softmax group: a step is one tile, or the whole product with row
    // copies and paired products.
    for (int k0 = 0; CG == 1 && k0 < ntiles; k0 += kU) {  // k0: first tile of the step
      const int j = k0 / kTPS, half = k0 % kTPS;  // score product and the step's first 64-token half
      const int step_t0 = t_begin + k0 * kTileTok;
      const int k_own = k0 + h_own;               // the tile holding this thread's columns
      if (half == 0 && !warp_wait(&s_full[j & 1], (j >> 1) & 1)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[kColsU];
      if (warp_rows) {
        const uint32_t ts = tS(mt, j & 1) + lane_off + static_cast<uint32_t>(half * kTileTok + c0u);
        if constexpr (kColsU == 64) {
          tmem_ld64(ts, s);
        } else if constexpr (kColsU == 32) {
          tmem_ld32(ts, s);
        } else {
          tmem_ld16(ts, s);
        }
      }
      tc_fence_before();
      __syncwarp();
      const int k_last = min(k0 + kU - 1, ntiles - 1);  // last tile of the step
      if (lane == 0 && (k_last % kTPS == kTPS - 1 || k_last == ntiles - 1)) mbar_arrive(&s_free[j & 1]);

      float alpha = 1.f;
      bool rescale = false;
      if (warp_rows) {
        // Row max on the raw scores (the scale is positive, so it commutes
        // with the max; it is applied in the exponent below), four partial
        // maxima of three-input max instructions. A step whose columns this
        // warp sees in full (nearly every prefix step) takes no mask.
        uint64_t vis = ~0ull;
        if constexpr (MASKED) {
          vis = column_mask(step_t0 + c0u);
        } else {
          const int nv = lim - (step_t0 + c0u);
          vis = nv >= 64 ? ~0ull : nv <= 0 ? 0ull : (1ull << nv) - 1ull;
        }
        constexpr uint64_t kAll = kColsU >= 64 ? ~0ull : (1ull << kColsU) - 1ull;
        if (!__all_sync(0xffffffffu, (vis & kAll) == kAll)) {
#pragma unroll
          for (int e = 0; e < kColsU; ++e) s[e] = ((vis >> e) & 1ull) ? s[e] : -INFINITY;
        }
        float pm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int e = 0; e < kColsU; e += 8) {
#pragma unroll
          for (int q = 0; q < 4; ++q) pm[q] = fmax3(pm[q], s[e + 2 * q], s[e + 2 * q + 1]);
        }
        const float mx = fmax3(pm[0], pm[1], fmaxf(pm[2], pm[3])) * scl;  // base-2 units
        if (m_run == -INFINITY) {
          m_run = mx;  // nothing accumulated for this row yet
        } else if (mx > m_run + kRescaleLog2) {
          alpha = ex2(m_run - mx);
          m_run = mx;
          l_run *= alpha;
          rescale = true;
        }
      }
      if (__any_sync(0xffffffffu, rescale)) {
        // This warp's O holds the PV of its earlier tiles, the last of them
        // k0 - 1: wait for it, then scale this warp's rows.
        if (!warp_wait(&o_done[(k0 - 1) % kPBufs], ((k0 - 1) / kPBufs) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (lane == 0) atomicAdd(a.rescales, 1ull);
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(tO(mt) + lane_off + c * 32, o);
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] *= alpha;
          tmem_st32(tO(mt) + lane_off + c * 32, o);
        }
      }
      if (warp_rows) {
        // P goes to TMEM over the consumed S columns: tile k of the product
        // takes columns (k % TPS) * 32 .. +31 of its S buffer, bf16 pairs.
        // This thread writes its slice of the tile k_own and zeros over the
        // rest of the step's tiles (other copies' slices).
        const uint32_t tbuf = tS(mt, j & 1) + lane_off;
        constexpr int kPColsS = kTileTok / 2;
        if (k_own < ntiles) {
          // p = 2^(s * scale * log2(e) - m): per pair of elements one paired
          // FMA, two exponentials, one bf16 pack and one paired add.
          const float nmu = m_run == -INFINITY ? 0.f : -m_run;
          const float2 sc2 = make_float2(scl, scl), nm2 = make_float2(nmu, nmu);
          float2 ls[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
          const uint32_t tp = tbuf + static_cast<uint32_t>((k_own % kTPS) * kPColsS);
#pragma unroll
          for (int c = 0; c < kColsU / 16; ++c) {  // 16 columns (8 TMEM columns) per store
            uint32_t w[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float2 x = fma2(make_float2(s[c * 16 + 2 * e], s[c * 16 + 2 * e + 1]), sc2, nm2);
              const float2 pp = make_float2(ex2(x.x), ex2(x.y));
              ls[e & 1] = add2(ls[e & 1], pp);
              w[e] = pack_bf16(pp.x, pp.y);
            }
            tmem_st_u32<8>(tp + static_cast<uint32_t>(lc0 / 2 + c * 8), w);
          }
          l_run += (ls[0].x + ls[0].y) + (ls[1].x + ls[1].y);
          if constexpr (kColsU < kTileTok) {
#pragma unroll
            for (int q = 0; q < kTileTok / kColsU; ++q)
              if (q != lc0 / kColsU) tmem_st_zero<kColsU / 2>(tp + static_cast<uint32_t>(q * (kColsU / 2)));
          }
        }
        if constexpr (kU > 1) {
#pragma unroll
          for (int h = 0; h < kU; ++h)
            if (h != h_own && k0 + h < ntiles)
              tmem_st_zero<32>(tbuf + static_cast<uint32_t>(((k0 + h) % kTPS) * 32));
        }
        tmem_wait_st();
      }
      // Hand the step's tiles to the MMA warp (every softmax warp arrives
      // for every tile; the P columns of other copies' slices are zero).
      bool step_ok = true;
#pragma unroll
      for (int h = 0; h < kU; ++h) {
        const int k = k0 + h;
        if (k >= ntiles) break;
        const int valid = t_end - (t_begin + k * kTileTok);
        if (valid < kTileTok && (valid & (kGroupTok - 1))) {
          // Cache slots past the sequence end inside its last page may hold
          // stale or uninitialised data; P is 0 there but 0 * NaN = NaN, so
          // zero those V rows before the PV MMA reads them.
          const int st = k % kTcStages;
          if (!warp_wait(kSplitKV ? &v_full[st] : &k_full[st], (k / kTcStages) & 1)) {
            step_ok = false;
            break;
          }
          const int r0 = valid, r1 = (valid + kGroupTok - 1) & ~(kGroupTok - 1);
          uint8_t* vt = smem + Lay::kVOff + st * Geo::kTileBytes;
          for (int idx = grp_tid; idx < (r1 - r0) * (D / 8); idx += 128 * MT) {
            const int row = r0 + idx / (D / 8), c = idx % (D / 8);
            *reinterpret_cast<uint4*>(vt + kv_swz(row, c)) = make_uint4(0, 0, 0, 0);
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[k % kPBufs]);
      }
      if (!step_ok) {
        ok = false;
        break;
      }
    }

    // ---------------- epilogue ----------------
    // Every PV has completed once o_fin (one group: the last o_done phase)
    // fires, so the K/V ring is free for staging. Warp-uniform, like every condition around the warp-collective
    // TMEM loads and stores below.
    const bool o_ready = __all_sync(
        0xffffffffu, ok && (CG == 2 ? mbar_wait(o_fin, 0, a.err)
                                    : mbar_wait(&o_done[(ntiles - 1) % kPBufs], ((ntiles - 1) / kPBufs) & 1, a.err)));
    // Copies of a row (REP > 1) hold its O over disjoint token slices, merged
    // by the split-combine rule (Sec. 3 Mode 2, here on one SM). The work is
    // split by columns: copy c finalises output columns [c*kRange,
    // (c+1)*kRange), so it leaves its (max, sum) and its unscaled O over the
    // other copies' ranges in the freed ring and reads theirs over its own.
    // With two softmax groups (CG = 2) the work is split the same way: group
    // c finalises output columns [c*kRange, (c+1)*kRange), reading both
    // groups' O over them from its own TMEM lanes.
    constexpr int kParts = REP * CG;            // states per row: copies or softmax groups
    constexpr int kRange = D / kParts;          // output columns this thread finalises
    // columns per TMEM load: 16, 32 or 64 (32 at most with two groups, whose
    // loads are paired)
    constexpr int kChunk = CG > 1 ? (kRange < 32 ? kRange : 32) : (kRange < 64 ? kRange : 64);
    static_assert(kChunk == 16 || kChunk == 32 || kChunk == 64, "TMEM load width");
    auto ld_chunk = [&](uint32_t taddr, float* o) {
      if constexpr (kChunk == 64) {
        tmem_ld64(taddr, o);
      } else if constexpr (kChunk == 32) {
        tmem_ld32(taddr, o);
      } else {
        tmem_ld16(taddr, o);
      }
    };
    constexpr int kXPitch = kRange * 4 + 16;  // exchange row pitch in bytes (padded: no bank conflicts)
    // copy c's O over copy q's column range, for this thread's row
    auto xchg_row = [&](int c, int q) -> uint8_t* {
      const int slot = c * (REP - 1) + (q < c ? q : q - 1);
      return smem + Lay::kXchgOff + (slot * 32 * kRowQuads + rq * 32 + lane) * kXPitch;
    };
    float wgt[kParts];  // weight of each part's O in this row's output, then with 1/sum folded in
    float m_row = m_run, l_row = l_run;
    wgt[0] = 1.f;
    if (o_ready) tc_fence_after();
    if constexpr (REP > 1) {
      static_assert(Lay::kXchgOff + REP * (REP - 1) * 32 * kRowQuads * kXPitch <= Lay::kPOff, "exchange buffers");
      static_assert(D / 64 * (128 / REP) * 128 <= Lay::kWtsOff, "output staging below the copies' weights");
      float* part_ml = reinterpret_cast<float*>(smem + Lay::kWtsOff);  // [TMEM lane][max, sum]
      part_ml[2 * r_loc] = o_ready ? m_run : -INFINITY;  // a copy cut short by a timeout is dropped
      part_ml[2 * r_loc + 1] = l_run;
      if (warp_rows && o_ready) {
#pragma unroll 1
        for (int q = 0; q < REP; ++q) {
          if (q == cp) continue;
          uint8_t* x = xchg_row(cp, q);
#pragma unroll 1
          for (int cc = 0; cc < kRange / kChunk; ++cc) {
            float o[kChunk];
            ld_chunk(tO(mt) + lane_off + q * kRange + cc * kChunk, o);
#pragma unroll
            for (int q4 = 0; q4 < kChunk / 4; ++q4)
              *reinterpret_cast<float4*>(x + cc * kChunk * 4 + q4 * 16) =
                  make_float4(o[4 * q4], o[4 * q4 + 1], o[4 * q4 + 2], o[4 * q4 + 3]);
          }
        }
      }
      named_bar_sync(2, 128);  // the four softmax warps
      float mc[REP], lc[REP];
      float m = -INFINITY;
#pragma unroll
      for (int c = 0; c < REP; ++c) {
        const int lq = (c * kRowQuads + rq) * 32 + lane;
        mc[c] = part_ml[2 * lq];
        lc[c] = part_ml[2 * lq + 1];
        m = fmaxf(m, mc[c]);
      }
      // A row that saw no key in any slice (possible in the verify pass)
      // keeps m = -inf, sum 0 and weight 0 everywhere.
      float l = 0.f;
#pragma unroll
      for (int c = 0; c < REP; ++c) {
        wgt[c] = mc[c] == -INFINITY ? 0.f : ex2(mc[c] - m);
        l += wgt[c] * lc[c];
      }
      m_row = m;
      l_row = l;
    }
    if constexpr (CG > 1) {
      // The groups' (max, sum) per row, exchanged through the freed ring.
      float* part_ml = reinterpret_cast<float*>(smem + Lay::kWtsOff);  // [group][TMEM lane][max, sum]
      part_ml[2 * (cg * 128 + r_loc)] = o_ready ? m_run : -INFINITY;  // a group cut short is dropped
      part_ml[2 * (cg * 128 + r_loc) + 1] = l_run;
      named_bar_sync(2, 32 * Cfg::kSmWarps);
      float mc[CG], lc[CG];
      float m = -INFINITY;
#pragma unroll
      for (int c = 0; c < CG; ++c) {
        mc[c] = part_ml[2 * (c * 128 + r_loc)];
        lc[c] = part_ml[2 * (c * 128 + r_loc) + 1];
        m = fmaxf(m, mc[c]);
      }
      float l = 0.f;
#pragma unroll
      for (int c = 0; c < CG; ++c) {
        wgt[c] = mc[c] == -INFINITY ? 0.f : ex2(mc[c] - m);
        l += wgt[c] * lc[c];
      }
      m_row = m;
      l_row = l;
    }
    const float inv = l_row > 0.f ? 1.f / l_row : 0.f;
#pragma unroll
    for (int c = 0; c < kParts; ++c) wgt[c] *= inv;
    // Normalised output columns cp*kRange + cc*kChunk .. +kChunk-1 of this
    // thread's row: its own TMEM lane plus the other copies' exchanged ranges.
    // Warp-collective.
    auto final_chunk = [&](int cc, float* o) {
      const int col0 = part * kRange + cc * kChunk;
      if constexpr (CG > 1) {
        // The one O both groups accumulated (same running max), over the
        // sum of both groups' sums.
        ld_chunk(tO(0) + lane_off + col0, o);
#pragma unroll
        for (int j = 0; j < kChunk; ++j) o[j] = l_row > 0.f ? o[j] * inv : 0.f;
        return;
      }
      ld_chunk(tO(mt) + lane_off + col0, o);
      float w_own = wgt[0];
#pragma unroll
      for (int c = 1; c < REP; ++c) w_own = c == cp ? wgt[c] : w_own;  // no dynamic register index
#pragma unroll
      for (int j = 0; j < kChunk; ++j) o[j] *= w_own;
      if constexpr (REP > 1) {
#pragma unroll
        for (int c = 0; c < REP; ++c) {
          if (c == cp || wgt[c] == 0.f) continue;  // a copy without keys never wrote its range
          const uint8_t* x = xchg_row(c, cp) + cc * kChunk * 4;
#pragma unroll
          for (int q4 = 0; q4 < kChunk / 4; ++q4) {
            const float4 v = *reinterpret_cast<const float4*>(x + q4 * 16);
            o[4 * q4] += wgt[c] * v.x;
            o[4 * q4 + 1] += wgt[c] * v.y;
            o[4 * q4 + 2] += wgt[c] * v.z;
            o[4 * q4 + 3] += wgt[c] * v.w;
          }
        }
      }
      if (!(l_row > 0.f)) {
#pragma unroll
        for (int j = 0; j < kChunk; ++j) o[j] = 0.f;  // a row without keys: zeros
      }
    };
    if (a.csize > 1) {
      // Cluster: stage this CTA's normalised rows and their log2-sum-exp in
      // the freed ring for the merge across the cluster (rows without keys,
      // or after a timeout, carry lse = -inf and are skipped by the merge).
      float* lse_stage = reinterpret_cast<float*>(smem + Lay::kLseOff);
      const bool has = o_ready && row_ok && l_row > 0.f;
      if (part == 0) lse_stage[r] = has ? m_row + lg2(l_row) : -INFINITY;
      if (warp_rows && o_ready) {
        uint8_t* my = smem + r * merge_pitch<D>();
#pragma unroll 1
        for (int cc = 0; cc < kRange / kChunk; ++cc) {
          float o[kChunk];
          final_chunk(cc, o);
          uint8_t* dst = my + (part * kRange + cc * kChunk) * 4;
#pragma unroll
          for (int q4 = 0; q4 < kChunk / 4; ++q4)
            *reinterpret_cast<float4*>(dst + q4 * 16) =
                make_float4(o[4 * q4], o[4 * q4 + 1], o[4 * q4 + 2], o[4 * q4 + 3]);
        }
      }
    } else {
      // Each thread stages its columns in 128-byte-swizzled boxes of 128-byte
      // rows in packed row order (block slot major, so that any 8 consecutive
      // lanes hit 8 different bank groups), and one thread stores the boxes
      // with tiled TMA copies: D/64 boxes of 64 bf16 columns per CTA (the
      // output, or the split partials, whose map walks the heads before the
      // block slots).
      const bool split_out = a.o_part != nullptr;
      const int srow = r;  // row within the boxes
      const int box_stride = (a.R * 128 + 1023) & ~1023;
      // kIters rounds (2 with one copy and D = 128, else 1): round cc stages
      // columns [cc*D/kIters, (cc+1)*D/kIters) of every row, and their boxes
      // are stored while the next round is staged.
      constexpr int kIters = kRange / kChunk;
#pragma unroll 1
      for (int cc = 0; cc < kIters; ++cc) {
        if (warp_rows && o_ready) {
          float o[kChunk];
          final_chunk(cc, o);
          const int col0 = part * kRange + cc * kChunk;
          if (row_ok) {
            uint8_t* row = smem + (col0 >> 6) * box_stride + srow * 128;
            const int ch0 = (col0 & 63) >> 3;
#pragma unroll
            for (int c8 = 0; c8 < kChunk / 8; ++c8) {
              const float* v = o + c8 * 8;
              *reinterpret_cast<uint4*>(row + (((ch0 + c8) ^ (srow & 7)) << 4)) =
                  make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]), pack_bf16(v[4], v[5]),
                             pack_bf16(v[6], v[7]));
            }
          }
        }
        // One thread stores the boxes a round completed: with one softmax
        // group round cc staged columns [cc*D/kIters, (cc+1)*D/kIters) of
        // every row; with two groups each round staged a slice of both
        // groups' ranges, so every box is stored after the last round.
        if (CG > 1 && cc + 1 < kIters) continue;
        constexpr int kStoreRounds = CG > 1 ? 1 : kIters;
        const int sr = CG > 1 ? 0 : cc;
        fence_proxy_async_smem();     // the staged boxes, visible to the TMA engine
        named_bar_sync(3, 32 * Cfg::kSmWarps);  // every softmax warp, with rows or not
        if (sm_tid == 0 && o_ready) {
#pragma unroll
          for (int x = sr * (D / 64 / kStoreRounds); x < (sr + 1) * (D / 64 / kStoreRounds); ++x) {
            if (split_out)
              tma_store_4d(&maps.o, smem + x * box_stride, x * 64, g * a.G, slot0, split * a.B + b);
            else
              tma_store_3d(&maps.o, smem + x * box_stride, x * 64, g * a.G, b * a.bl + slot0);
          }
          bulk_commit();
        }
      }
      if (warp_rows && o_ready && row_ok && part == 0) {
        const float lse_v = l_row > 0.f ? (m_row + lg2(l_row)) * kLn2 : -INFINITY;
        if (!split_out) {
          if (a.lse != nullptr) a.lse[(static_cast<size_t>(b) * a.Hq + row_h) * a.bl + row_i] = lse_v;
        } else {
          a.lse_part[((static_cast<size_t>(split) * a.B + b) * a.Hq + row_h) * a.bl + row_i] = lse_v;
        }
      }
      if (sm_tid == 0 && o_ready) bulk_store_wait_read();  // the boxes stay in place until read
    }
    tc_fence_before();
  }

  if (a.csize > 1) {
    // Merge across the cluster (the splits of this sequence and KV head):
    // CTA `rank` combines rows [rank*Rc, (rank+1)*Rc) from every peer's
    // staged rows through distributed shared memory, by the same rule as the
    // split combine, and writes the final output (one cluster per sequence
    // and KV head) or this cluster's partial.
    cluster_sync();
    if (warp >= kSoftmaxWarp0 && warp < kSoftmaxWarp0 + Cfg::kSmWarps) {
      const uint32_t rank = cluster_ctarank();
      const int Rc = (a.R + a.csize - 1) / a.csize;
      const int r0 = static_cast<int>(rank) * Rc;
      const int nrows = max(0, min(a.R, r0 + Rc) - r0);
      const uint32_t stage_u32 = smem_u32(smem);
      const uint32_t lse_u32 = stage_u32 + Lay::kLseOff;
      // this CTA's merge weights, local: [row][peer] and the merged lse per row
      float* wts = reinterpret_cast<float*>(smem + Lay::kWtsOff);
      float* lse_out = reinterpret_cast<float*>(smem + Lay::kLseOutOff);
      const int tid = threadIdx.x - 32 * kSoftmaxWarp0;
      // 1) per-row weights: one thread per row, the peers' lse loads in flight together
      if (tid < nrows) {
        const int r = r0 + tid;
        float lp[8];
        float m = -INFINITY;
#pragma unroll
        for (int p = 0; p < 8; ++p) lp[p] = p < a.csize ? ld_dsmem_f32(dsmem_addr(lse_u32 + r * 4, p)) : -INFINITY;
#pragma unroll
        for (int p = 0; p < 8; ++p) m = fmaxf(m, lp[p]);
        float w[8];
        float wsum = 0.f;
#pragma unroll
        for (int p = 0; p < 8; ++p) {
          w[p] = (m != -INFINITY && lp[p] != -INFINITY) ? ex2(lp[p] - m) : 0.f;
          wsum += w[p];
        }
        const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
#pragma unroll
        for (int p = 0; p < 8; ++p) wts[tid * 8 + p] = w[p] * inv;
        lse_out[tid] = wsum > 0.f ? (m + lg2(wsum)) * kLn2 : -INFINITY;
      }
      named_bar_sync(1, 32 * Cfg::kSmWarps);
      // 2) rows: two (row, 4-dim) items per thread per round, every peer load in flight
      const bool final_out = a.num_partials == 1;
      const int pidx = split / a.csize;
      const int items = nrows * (D / 4);
      for (int base = tid; base < items; base += 2 * 32 * Cfg::kSmWarps) {
        float4 acc[2];
        int ridx[2], d4[2];
        bool live[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int idx = base + u * 32 * Cfg::kSmWarps;
          live[u] = idx < items;
          ridx[u] = live[u] ? idx / (D / 4) : 0;
          d4[u] = idx % (D / 4);
          acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        float4 o[2][8];
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int p = 0; p < 8; ++p)
            if (live[u] && p < a.csize && wts[ridx[u] * 8 + p] > 0.f)  // rows without keys are never read
              o[u][p] = ld_dsmem_f4(dsmem_addr(stage_u32 + (r0 + ridx[u]) * merge_pitch<D>() + d4[u] * 16, p));
            else
              o[u][p] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 2; ++u) {
#pragma unroll
          for (int p = 0; p < 8; ++p) {
            const float w = p < a.csize ? wts[ridx[u] * 8 + p] : 0.f;
            acc[u].x += w * o[u][p].x; acc[u].y += w * o[u][p].y;
            acc[u].z += w * o[u][p].z; acc[u].w += w * o[u][p].w;
          }
          if (!live[u]) continue;
          const int r = r0 + ridx[u];
          const int i = r / a.G, h = g * a.G + (r - i * a.G);
          const float lse_v = lse_out[ridx[u]];
          if (final_out) {
            __nv_bfloat16* orow = a.out + ((static_cast<size_t>(b) * a.bl + i) * a.Hq + h) * D;
            *reinterpret_cast<uint2*>(orow + d4[u] * 4) =
                make_uint2(pack_bf16(acc[u].x, acc[u].y), pack_bf16(acc[u].z, acc[u].w));
            if (d4[u] == 0 && a.lse != nullptr) a.lse[(static_cast<size_t>(b) * a.Hq + h) * a.bl + i] = lse_v;
          } else {
            const size_t prow = ((static_cast<size_t>(pidx) * a.B + b) * a.Hq + h) * a.bl + i;
            if (lse_v != -INFINITY)
              *reinterpret_cast<uint2*>(a.o_part + prow * D + d4[u] * 4) =
                  make_uint2(pack_bf16(acc[u].x, acc[u].y), pack_bf16(acc[u].z, acc[u].w));
            if (d4[u] == 0) a.lse_part[prow] = lse_v;
          }
        }
      }
    }
    cluster_sync();  // peers keep their shared memory until every merge has read it
  }

  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

template <int D, int MT, int REP, int TPS, bool MASKED, bool ORDERED, int CG>
cudaError_t configure_tc(int dev) {
  static int configured[64] = {0};
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!__atomic_load_n(&configured[dev], __ATOMIC_ACQUIRE)) {
    cudaError_t e = cudaFuncSetAttribute(block_attn_tc_kernel<D, MT, REP, TPS, MASKED, ORDERED, CG>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(TcLayout<D, MT, TPS>::kBytes + 1024));
    if (e != cudaSuccess) return e;
    __atomic_store_n(&configured[dev], 1, __ATOMIC_RELEASE);
  }
  return cudaSuccess;
}

template <int D, int MT, int REP, int TPS, bool MASKED, bool ORDERED, int CG>
cudaError_t launch_tc_o(const AttnArgs& a, const TmaMaps& maps, cudaStream_t stream) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if ((e = configure_tc<D, MT, REP, TPS, MASKED, ORDERED, CG>(dev)) != cudaSuccess) return e;
  dim3 grid(a.num_splits * a.nh, a.Hkv, a.B);
  return launch_kernel_cluster(block_attn_tc_kernel<D, MT, REP, TPS, MASKED, ORDERED, CG>, grid,
                               dim3(TcCfg<MT, TPS, CG>::kThreads), TcLayout<D, MT, TPS>::kBytes + 1024, stream,
                               a.csize, maps, a);
}

// The longest-first order only for the unmasked passes (the table-mask
// passes run at the block shapes of one sequence).
template <int D, int MT, int REP, int TPS, bool MASKED, int CG = 1>
cudaError_t launch_tc_t(const AttnArgs& a, const TmaMaps& maps, cudaStream_t stream) {
  if constexpr (!MASKED) {
    if (a.order_by_length) return launch_tc_o<D, MT, REP, TPS, false, true, CG>(a, maps, stream);
  }
  return launch_tc_o<D, MT, REP, TPS, MASKED, false, CG>(a, maps, stream);
}

// Resident clusters of the kernel a plan would launch (one CTA per SM
// either way; row copies and score-product width do not change residency,
// the thread count of two softmax groups does not either, but the query
// uses the instantiation that runs).
template <int D, int MT, int REP, int TPS, int CG>
int max_active_clusters_t(int csize) {
  static int cache[64][4];  // [device][cluster size 2/4/8] + 1 (0 = not queried)
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int slot = csize == 2 ? 0 : csize == 4 ? 1 : csize == 8 ? 2 : 3;
  int v = __atomic_load_n(&cache[dev][slot], __ATOMIC_ACQUIRE);
  if (v) return v - 1;
  if (configure_tc<D, MT, REP, TPS, false, false, CG>(dev) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(csize, 1, 1);
  cfg.blockDim = dim3(TcCfg<MT, TPS, CG>::kThreads);
  cfg.dynamicSmemBytes = TcLayout<D, MT, TPS>::kBytes + 1024;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, block_attn_tc_kernel<D, MT, REP, TPS, false, false, CG>, &cfg) !=
      cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  __atomic_store_n(&cache[dev][slot], n + 1, __ATOMIC_RELEASE);
  return n;
}

// Copies of each Q row in the 128 TMEM lanes of one M tile: 4 for up to 32
// packed rows, 2 for up to 64, else 1 (and 1 with two M tiles).
// Row copies of the one-group kernel: 33..64 rows take two copies; up to
// 32 rows and 65..128 rows run on the two-group kernel (1).
int tc_replication(int rows) { return rows > 32 && rows <= 64 ? 2 : 1; }

template <int D>
int max_active_clusters_d(int csize, int rows) {
  if (rows > 128) return max_active_clusters_t<D, 2, 1, 1, 1>(csize);
  switch (tc_replication(rows)) {
    case 2: return max_active_clusters_t<D, 1, 2, 1, 1>(csize);
    default: return max_active_clusters_t<D, 1, 1, 2, 2>(csize);
  }
}

// One M tile: 33..64 rows copied twice, with paired score products when a
// split fits in the ring whole (it is then latency-bound: fewer, wider steps
// help; the 8B shape's 64 rows measured 7.12 us per launch against 7.32 on
// the two-group kernel) and single tiles when it streams; up to 32 and
// 65..128 rows take paired products and two softmax groups, streaming or
// not (32-row batches measured 50/75/87 -> 55/86/95% of peak at B = 8, 32,
// 128 against four row copies: the score products run ahead of the PV
// products there, and each tile takes 8 MMAs instead of 12).
template <int D, int TPS, bool MASKED>
cudaError_t launch_tc_rep(const AttnArgs& a, const TmaMaps& maps, cudaStream_t stream) {
  switch (tc_replication(a.R)) {
    case 2: return launch_tc_t<D, 1, 2, TPS, MASKED>(a, maps, stream);
    default: return launch_tc_t<D, 1, 1, 2, MASKED, 2>(a, maps, stream);
  }
}

template <int D, bool MASKED>
cudaError_t launch_tc_d(const AttnArgs& a, const TmaMaps& maps, cudaStream_t stream) {
  // Block-slot chunks hold 65..128 rows, which only the two-group kernels
  // take (they read a.nh; the others assume one chunk).
  if (a.nh != 1 && (a.R <= 64 || a.R > 128)) return cudaErrorInvalidValue;
  if (a.R > 128) return launch_tc_t<D, 2, 1, 1, MASKED>(a, maps, stream);
  if (a.chunk <= TcLayout<D, 1, 2>::kStages * kTileTok) return launch_tc_rep<D, 2, MASKED>(a, maps, stream);
  return launch_tc_rep<D, 1, MASKED>(a, maps, stream);
}

}  // namespace
}  // namespace nld
