// Block attention on the tcgen05 tensor cores: the draft and verify passes
// (the kernel and its launch templates are in block_attn_tc.cuh; the
// table-mask instantiations live in block_attn_tc_masked.cu).
#include "block_attn_tc.cuh"

namespace nld {

bool tc_supports(int R, int head_dim) { return R <= 256 && (head_dim == 64 || head_dim == 128); }

int tc_max_active_clusters(int csize, int head_dim, int rows) {
  return head_dim == 128 ? max_active_clusters_d<128>(csize, rows) : max_active_clusters_d<64>(csize, rows);
}

cudaError_t launch_block_attn_tc(const AttnArgs& a, const TmaMaps& maps, int head_dim, cudaStream_t stream) {
  if (a.mode == kModeBlockMask) return launch_block_attn_tc_masked(a, maps, head_dim, stream);
  return head_dim == 128 ? launch_tc_d<128, false>(a, maps, stream) : launch_tc_d<64, false>(a, maps, stream);
}

}  // namespace nld
