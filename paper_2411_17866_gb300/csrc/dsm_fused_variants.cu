// Instantiations of the fused round's kernel for the SlowMo, signed SlowMo and Lookahead global steps
// (a translation unit of its own so that the families compile in parallel).

#include "dsm_fused.cuh"

namespace dsm {

FusedKernel fused_kernel_variants(const Problem& p, bool adamw) { return fused_kernel_v<kGlobalRuntime>(p, adamw); }

}  // namespace dsm
