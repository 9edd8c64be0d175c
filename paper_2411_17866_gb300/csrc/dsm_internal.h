// Internal interface between the C-ABI host code (dsm_api.cpp) and the
// CUDA kernels (dsm_kernels.cu).  Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

#include "dsm.h"

namespace dsm {

// Elements of one tile.  A tile lies inside one tensor; a tensor of numel
// elements has ceil(numel / kTile) tiles.  One CTA of kThreads threads
// processes one tile, kElemsPerThread consecutive elements per thread (one
// 16-byte vector of every fp32 stream).
constexpr uint32_t kThreads = 256;
constexpr uint32_t kElemsPerThread = 4;
constexpr uint32_t kTile = kThreads * kElemsPerThread;  // 1024
constexpr uint32_t kMaxWorkers = 64;
constexpr uint32_t kMaxUnrolledWorkers = 8;  // replicas held in registers by the global step

// Per-tensor record in device memory (48 bytes).
struct TensorDesc {
    uint64_t off;          // first element in the packed model
    uint64_t numel;
    float scale;           // s_T
    float scale2;          // fp32(0.1f * s_T)
    float lam_local;       // AdamW decoupled weight decay for this tensor (0 if exempt)
    float lam_global;      // global lambda for this tensor (0 if exempt)
    uint32_t kind;
    uint32_t tile_begin;   // tiles [tile_begin, tile_end) cover this tensor
    uint32_t tile_end;
    uint32_t pad;
};
static_assert(sizeof(TensorDesc) == 48, "TensorDesc layout");

// Per-tile record in device memory (16 bytes).
struct TileDesc {
    uint64_t start;        // first element (logical index)
    uint32_t len;          // 1..kTile
    uint32_t tensor;
};
static_assert(sizeof(TileDesc) == 16, "TileDesc layout");

// Per-tile partial statistics written by the global step (32 bytes).
struct StatPartial {
    double delta_sq;
    double drift;
    uint32_t zero_sign, flips, unanimous, clamped;
};
static_assert(sizeof(StatPartial) == 32, "StatPartial layout");

// Per-tensor statistics (same layout as dsm_tensor_stats).
struct TensorStats {
    double delta_sq;
    double drift;
    unsigned long long zero_sign, flips, unanimous, clamped;
};
static_assert(sizeof(TensorStats) == 48, "TensorStats layout");

// Views of the arena shared by the kernels.
struct Problem {
    const TensorDesc* tensors;
    const TileDesc* tiles;
    uint32_t num_tensors;
    uint32_t num_tiles;
    uint32_t n;
    uint64_t d_stride;     // elements between workers
    float* x;              // [d]
    float* m;              // [d]
    float* gv;             // [d] global AdamW second moment (global mode 4 only)
    int global_mode;
    float* X;              // [n][d_stride] replicas
    float* opt_m;          // [n][d_stride]
    float* opt_v;          // [n][d_stride] (AdamW only)
    void* grad;            // [n][d_stride], fp32 or bf16
    int grad_bf16;
    StatPartial* partials; // [num_tiles]; only each CTA's last tile of a tensor is written
    TensorStats* stats;    // [num_tensors]
};

// Scalars of one AdamW local step (all fp32, computed once on the host).
struct AdamScalars {
    float b1, omb1;        // beta1, 1 - beta1
    float b2, omb2;        // beta2, 1 - beta2
    float bc1, bc2;        // 1 - beta1^j, 1 - beta2^j
    float lr, eps;
};

struct SgdmScalars {
    float mu, lr;
};

struct GlobalScalars {
    float b1, b2;          // global betas (SlowMo: b1 is its beta)
    float c1, c2;          // (1 - beta1)/gamma, (1 - beta2)/gamma
    float eta_gamma;       // eta * gamma
    float inv_gamma;       // 1/gamma (SlowMo, global AdamW)
    float omb1, omb2;      // global AdamW: 1 - beta1, 1 - beta2
    float bc1, bc2;        // global AdamW: 1 - beta1^(t+1), 1 - beta2^(t+1)
    float eps, eta;        // global AdamW epsilon and learning rate
    float B;               // randomized-sign bound
    float n_f;             // n as float (divisor of the average)
    int sign_mode;
    int mode;              // DSM_GLOBAL_*: read by the fused round's kernel for the ablation variants
    uint32_t philox_k0, philox_k1;
    uint64_t philox_q0;    // counter of the layout's first element group: first_element / 4
    int skip_reset;        // K4: leave the replicas' reset to x pending (the next local step starts from x)
};

// SplitMix64 keys of one synthetic-gradient fill.
struct GradKeys {
    uint64_t step;                  // key(seed, 0, step)
    uint64_t worker[kMaxWorkers];   // key(seed, 1, i)
};

// Launch shape: a persistent grid of `blocks` CTAs per kernel.
struct LaunchShape {
    int sms = 0;
    int grid_grad = 0, grid_adamw = 0, grid_sgdm = 0, grid_global = 0, grid_init = 0;
    int grid_fused = 0, grid_adamw_from_x = 0, grid_sgdm_from_x = 0;
};

// Launchers (dsm_kernels.cu, dsm_local.cu, dsm_fused.cu).  Each returns the cudaError_t of its launch.
cudaError_t query_launch_shape(const Problem& p, LaunchShape* out);
cudaError_t query_local_shape(const Problem& p, LaunchShape* out);  // the local steps' grids (dsm_local.cu)
cudaError_t launch_init(const Problem& p, const LaunchShape& ls, uint64_t seed_key_init, int from_hash,
                        cudaStream_t s);
cudaError_t launch_grad_fill(const Problem& p, const LaunchShape& ls, const GradKeys& k, cudaStream_t s);
// from_x: every worker starts from the global x (the replicas' reset is pending).
// zero_state: every worker's base-optimizer state is zero (its reset is pending); none is read.
cudaError_t launch_local_adamw(const Problem& p, const LaunchShape& ls, const AdamScalars& a, bool from_x,
                               bool zero_state, cudaStream_t s);
cudaError_t launch_local_sgdm(const Problem& p, const LaunchShape& ls, const SgdmScalars& a, bool from_x,
                              bool zero_state, cudaStream_t s);
// The fused round's last local step + sign-momentum global step (n <= 8).
// Options of the fused kernel (bits of its `opts` argument).
constexpr int kFusedFromX = 1;      // the replicas' reset is pending: every worker starts from x
constexpr int kFusedZeroState = 2;  // the base-optimizer states are zero: none is read
constexpr int kFusedDropState = 4;  // the new base-optimizer states are not written (the round resets them)
bool fused_round_available(const Problem& p);
cudaError_t query_fused_shape(const Problem& p, LaunchShape* out);  // sets grid_fused (out->sms must be set)
// The global-step launchers write per-tile statistics partials and set *grid to the number of CTAs
// they launched; launch_stats reduces those partials per tensor and needs that grid.
cudaError_t launch_fused_last_global(const Problem& p, const LaunchShape& ls, const AdamScalars& a,
                                     const SgdmScalars& sa, const GlobalScalars& g, int opts, cudaStream_t s,
                                     uint32_t* grid);
cudaError_t launch_global(const Problem& p, const LaunchShape& ls, const GlobalScalars& g, cudaStream_t s,
                          uint32_t* grid);
cudaError_t launch_stats(const Problem& p, uint32_t producer_grid, cudaStream_t s);

// Sets the calling thread's message returned by dsm_last_error() (dsm_api.cpp).
void set_last_error_message(const char* msg);

// The checks every entry point applies to a tensor list (dsm_api.cpp): at least one tensor, kinds
// known, grad_scale finite, reserved 0, sizes within 2^40 elements, at least one element, and
// first_element a multiple of 4 below 2^60.
// Sets *d and *tiles (tiles of kTile elements) and returns DSM_OK, or fails like every call.
int check_tensor_list(const dsm_layout* layout, uint64_t* d, uint64_t* tiles);

}  // namespace dsm
