// Instantiations of the attention kernels for head_dim 128.
#include "attn_kernel.cuh"

namespace wise {
cudaError_t launch_attn_d128(int block, int mode, const AttnLaunch& L) { return launch_attn_for_dim<128>(block, mode, L); }
}  // namespace wise
