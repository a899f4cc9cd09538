// Block attention on the tcgen05 tensor cores with a table mask over the
// block slots (structured masks such as quadratic self-speculation's,
// Sec. 3): the MASKED instantiations of the kernel in block_attn_tc.cuh,
// compiled apart so that the draft and verify kernels keep their code.
#include "block_attn_tc.cuh"

namespace nld {

cudaError_t launch_block_attn_tc_masked(const AttnArgs& a, const TmaMaps& maps, int head_dim, cudaStream_t stream) {
  return head_dim == 128 ? launch_tc_d<128, true>(a, maps, stream) : launch_tc_d<64, true>(a, maps, stream);
}

}  // namespace nld
