// Instantiations of the attention kernels for head_dim 96.
#include "attn_kernel.cuh"

namespace wise {
cudaError_t launch_attn_d96(int block, int mode, const AttnLaunch& L) { return launch_attn_for_dim<96>(block, mode, L); }
}  // namespace wise
