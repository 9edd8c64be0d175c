// Host side of the fused round (DSM_FLAG_FUSED_ROUND): which kernel, how much
// shared memory, the launch.  The kernel is in dsm_fused.cuh.

#include "dsm_fused.cuh"

namespace dsm {
namespace {

int fused_global_for(const Problem& p) {
    return p.global_mode == 0 ? kGlobalSign : (p.global_mode == 4 ? kGlobalAdamW : kGlobalRuntime);
}

FusedKernel fused_kernel_for(const Problem& p, bool adamw) {
    switch (fused_global_for(p)) {
        case kGlobalSign: return fused_kernel_sign(p, adamw);
        case kGlobalAdamW: return fused_kernel_adamw(p, adamw);
        default: return fused_kernel_variants(p, adamw);
    }
}

size_t fused_smem_for(const Problem& p, bool adamw) {
    return fused_smem(adamw, p.grad_bf16 != 0, int(p.n), fused_global_for(p));
}

}  // namespace

bool fused_round_available(const Problem& p) {
    // every global step, up to 8 workers (the differences x - x_i of all workers stay in registers)
    return p.global_mode >= 0 && p.global_mode <= 4 && p.n >= 1 && p.n <= kMaxUnrolledWorkers;
}

cudaError_t query_fused_shape(const Problem& p, LaunchShape* out) {
    if (!fused_round_available(p)) return cudaSuccess;
    const FusedKernel fk = fused_kernel_for(p, p.opt_v != nullptr);
    const size_t smem = fused_smem_for(p, p.opt_v != nullptr);
    cudaError_t e = cudaFuncSetAttribute(fk, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) return e;
    out->grid_fused = grid_for(fk, out->sms, smem);
    return cudaSuccess;
}

cudaError_t launch_fused_last_global(const Problem& p, const LaunchShape& ls, const AdamScalars& a,
                                     const SgdmScalars& sa, const GlobalScalars& g, int opts, cudaStream_t s,
                                     uint32_t* grid_used) {
    if (!fused_round_available(p)) return cudaErrorInvalidValue;
    const int grid = clamp_grid(ls.grid_fused, p.num_tiles);
    *grid_used = static_cast<uint32_t>(grid);
    if (grid == 0) return cudaSuccess;
    fused_kernel_for(p, p.opt_v != nullptr)<<<grid, kThreads, fused_smem_for(p, p.opt_v != nullptr), s>>>(
        p, a, sa, g, opts);
    return cudaGetLastError();
}

}  // namespace dsm
