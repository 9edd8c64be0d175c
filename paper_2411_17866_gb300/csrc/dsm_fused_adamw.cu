// Instantiations of the fused round's kernel for the global AdamW step
// (a translation unit of its own so that the families compile in parallel).

#include "dsm_fused.cuh"

namespace dsm {

FusedKernel fused_kernel_adamw(const Problem& p, bool adamw) { return fused_kernel_v<kGlobalAdamW>(p, adamw); }

}  // namespace dsm
