// Instantiations of the fused round's kernel for Algorithm 1's global step
// (a translation unit of its own so that the families compile in parallel).

#include "dsm_fused.cuh"

namespace dsm {

FusedKernel fused_kernel_sign(const Problem& p, bool adamw) { return fused_kernel_v<kGlobalSign>(p, adamw); }

}  // namespace dsm
