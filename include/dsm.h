/*
 * dsm.h -- C ABI of the GB300 library for one global round of distributed
 * sign momentum with local steps (arXiv 2411.17866, Algorithm 1).
 *
 * The problem (Sec. 1, Eq. (dist-opt)): n workers minimise the average of
 * their local losses over a shared model x in R^d.  One global round
 * (Algorithm 1) runs tau local base-optimizer steps on every worker's copy
 * of the model, Eq. (local-steps), then averages the copies (the
 * all-reduce), forms the sign-momentum update Eqs. (ut-update) and
 * (model-update), updates the global momentum, Eq. (mom-update), and
 * resets every worker copy to the new global model.
 *
 * Here the n workers are simulated as n replicas held in one GPU's memory;
 * the all-reduce is an on-device reduction over the replicas.
 *
 * Memory and ownership
 *   - The caller allocates one device buffer (the "arena", at least
 *     dsm_state_bytes() bytes, 256-byte aligned) and keeps it alive until
 *     dsm_destroy().  Every state of the method lives in it: global model x,
 *     global momentum m, n worker replicas, n base-optimizer states, n
 *     gradient buffers, the tile table and the statistics scratch.
 *   - The library allocates no device memory.  It owns only the handle's
 *     host-side metadata.
 *   - Streams belong to the caller.  A stream argument is a cudaStream_t
 *     passed as void*; NULL means the legacy default stream.
 *
 * Asynchrony
 *   Every call that takes a stream only enqueues work on it, except where
 *   its comment says it synchronises.  Calls on one handle must be issued in
 *   the order of Algorithm 1 (the handle enforces it, see DSM_ESTATE).
 *
 * Errors
 *   Every int-returning call returns DSM_OK (0) or a negative DSM_E* code
 *   and never aborts the process; dsm_last_error() gives a message for the
 *   calling thread's last failure.  A call that fails argument or order
 *   checks (DSM_EINVAL, DSM_ERANGE, DSM_ESTATE, ...) changes nothing.  After
 *   DSM_ECUDA from a call that enqueues work, the device state is whatever
 *   the failed CUDA call left: restore a checkpoint or create a new handle.
 *
 * Thread safety: a handle is not thread-safe; distinct handles are
 * independent.
 */
#ifndef DSM_H
#define DSM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes ---------------------------------------------------- */
#define DSM_OK      0
#define DSM_EINVAL (-1)  /* bad argument (null pointer, n = 0, tau = 0, beta outside its range, ...) */
#define DSM_ENOMEM (-2)  /* arena smaller than dsm_state_bytes() */
#define DSM_EALIGN (-3)  /* arena not 256-byte aligned, or not device memory */
#define DSM_ESTATE (-4)  /* call out of Algorithm 1's order (see dsm_local_step / dsm_global_step) */
#define DSM_ECUDA  (-5)  /* a CUDA call or kernel launch failed; dsm_last_error() has its message */
#define DSM_ERANGE (-6)  /* element range outside the model, worker index >= n, or a size beyond a limit */

/* ---- enumerations ---------------------------------------------------- */
/* Tensor kinds: only the initialisation depends on them (weights draw a
 * hash value, LayerNorm weights start at 1, biases at 0). */
#define DSM_KIND_WEIGHT 0
#define DSM_KIND_BIAS   1
#define DSM_KIND_LN_W   2
#define DSM_KIND_LN_B   3

/* Base optimizer of the local steps, Eq. (local-steps) (Appendix A). */
#define DSM_BASE_ADAMW 0  /* Algorithm "AdamW" */
#define DSM_BASE_SGDM  1  /* Algorithm "Polyak" (heavy ball); mu = 0 is plain SGD, Eq. (base-sgd) */

/* Sign operator of the global step. */
#define DSM_SIGN        0  /* deterministic sign, Eq. (model-update); sign(0) = 0 */
#define DSM_RSIGN_ZERO  1  /* randomized sign, Eq. (rand-sign-2): sign(v) w.p. |v|/B, else 0 */
#define DSM_RSIGN_PM    2  /* randomized sign, Eq. (rand-sign-1): sign(v) w.p. 1/2+|v|/(2B), else -sign(v) */

/* Gradient storage type. */
#define DSM_F32  0
#define DSM_BF16 1

/* Global step.  Algorithm 1 (the default) or a variant of the ablations
 * (Sec. 5), all with the same all-reduce average and reset:
 *   SIGN_MOMENTUM  Eqs. (ut-update), (model-update), (mom-update)
 *   SLOWMO         Appendix A, Algorithm "SlowMo": u <- b1 u + (1/gamma) Delta (kept in m),
 *                  x' = x - eta gamma u (eta plays the role of SlowMo's alpha)
 *   SIGNED_SLOWMO  Sec. 5: u = b1 m + ((1-b1)/gamma) sign(Delta), x' = x - eta gamma u,
 *                  m' = b2 m + ((1-b2)/gamma) Delta
 *   LOOKAHEAD      Sec. 5: Algorithm 1 with x' = x - eta gamma u
 *   ADAMW          Appendix, Algorithm "global AdamW": g = Delta/gamma, AdamW moments m, v with
 *                  bias corrections 1 - b^(t+1), x' = x - eta (mhat/(sqrt(vhat)+g_eps) + lambda x)
 * The randomized sign modes apply to SIGN_MOMENTUM only. */
#define DSM_GLOBAL_SIGN_MOMENTUM 0
#define DSM_GLOBAL_SLOWMO        1
#define DSM_GLOBAL_SIGNED_SLOWMO 2
#define DSM_GLOBAL_LOOKAHEAD     3
#define DSM_GLOBAL_ADAMW         4

/* Fused round.  Same results, fewer bytes: the round's last local step
 * runs inside dsm_global_step (dsm_local_step for k = tau-1 only records
 * it), so its new replicas never go to memory, and the reset of the replicas
 * is lazy: the next round's first local step starts every worker from x
 * instead of reading n copies of it.  Applies to every global step; with
 * more than 8 workers only the reset is deferred (the last local step runs
 * on its own: the differences of all workers no longer fit in registers).
 * Reading a replica while
 * the reset is pending returns x; reading or writing worker state, or
 * writing gradients through dsm_fill_synthetic_grads/dsm_load_grads, while
 * the last local step is pending first runs that step unfused.  Gradients
 * written through dsm_grad_ptr must not change between the last
 * dsm_local_step and dsm_global_step. */
#define DSM_FLAG_FUSED_ROUND 1u

/* Restart the base optimizer every round.  Algorithm 1 synchronises only
 * the model (its last step) and leaves open what becomes of each worker's
 * base-optimizer state; by default that state (AdamW moments, SGD-momentum
 * buffer) persists across rounds and AdamW counts j = t*tau + k + 1.  With
 * this flag every round instead starts each worker's base optimizer afresh,
 * as if a new optimizer were built at each synchronisation: its state is
 * zero at the round's first local step and AdamW counts j = k + 1.  Reading
 * DSM_BUF_OPT_M / DSM_BUF_OPT_V between rounds returns zeros.  The zeroing
 * is lazy: the round's first local step reads no state, and the fused
 * round's last local step writes none (the next round would discard it). */
#define DSM_FLAG_RESET_LOCAL_STATE 2u

/* Buffers for dsm_read_params / dsm_write_params. */
#define DSM_BUF_X        0  /* global model x_{t,0} (fp32, d) */
#define DSM_BUF_M        1  /* global momentum m_t (fp32, d) */
#define DSM_BUF_REPLICA  2  /* worker replica x^{(i)} (fp32, d) */
#define DSM_BUF_OPT_M    3  /* worker AdamW first moment, or SGD-momentum buffer (fp32, d) */
#define DSM_BUF_OPT_V    4  /* worker AdamW second moment (fp32, d); AdamW only */
#define DSM_BUF_GRAD     5  /* worker gradient buffer (fp32 or bf16 per grad_dtype, d) */
#define DSM_BUF_GLOBAL_V 6  /* global AdamW second moment (fp32, d); DSM_GLOBAL_ADAMW only */

typedef void* dsm_stream_t;  /* a cudaStream_t */

/* One parameter tensor.  Tensors are packed in order into one flat model
 * of d = sum(numel) elements; element e of the model is the "logical
 * index" used by the synthetic generators and by dsm_read_params. */
typedef struct {
    uint64_t numel;       /* elements (0 allowed) */
    float grad_scale;     /* s_T of the synthetic gradient generator */
    uint32_t kind;        /* DSM_KIND_* */
    uint32_t wd;          /* nonzero: decoupled weight decay applies (local and global) */
    uint32_t reserved;    /* must be 0 */
} dsm_tensor;

/* A parameter layout: the tensor list, packed in order.  first_element is
 * the logical index of the layout's first element within a larger model of
 * which this layout is a contiguous part (0 for a whole model): a parameter
 * shard of a model split over processes or GPUs (every step of Algorithm 1
 * is elementwise, so a shard needs no communication).  The synthetic
 * generators and the randomized sign's Philox counter then take element e
 * of this layout as element first_element + e of the larger model, so the
 * shards together compute exactly what one process computes on the whole
 * model.  Must be a multiple of 4 and below 2^60 (DSM_EINVAL otherwise). */
typedef struct {
    const dsm_tensor* tensors;  /* host array of count entries */
    uint32_t count;
    uint64_t first_element;
} dsm_layout;

/* Hyper-parameters.  Float fields are used as the fp32 values given. */
typedef struct {
    int32_t base;        /* DSM_BASE_* */
    float lr;            /* gamma: local learning rate, also gamma_t of the global step; > 0 */
    float b1, b2;        /* AdamW betas, in [0, 1) */
    float eps;           /* AdamW epsilon, > 0 (the paper uses 1e-8) */
    float wd;            /* AdamW decoupled weight decay, >= 0 */
    float mu;            /* SGD-momentum coefficient, in [0, 1) */
    float g_b1, g_b2;    /* global beta1, beta2 of Eqs. (ut-update), (mom-update), in [0, 1] ([0, 1) for ADAMW) */
    float g_eta;         /* global learning rate eta of Eq. (model-update), >= 0 */
    float g_wd;          /* global decoupled weight decay lambda, >= 0 */
    int32_t sign_mode;   /* DSM_SIGN | DSM_RSIGN_ZERO | DSM_RSIGN_PM */
    float rsign_B;       /* bound B of Eqs. (rand-sign-1/2); > 0 when randomized */
    int32_t grad_dtype;  /* DSM_F32 | DSM_BF16 */
    uint32_t flags;      /* DSM_FLAG_* bits; others must be 0 */
    uint64_t seed;       /* seed of the synthetic generators and of the Philox key */
    int32_t global_mode; /* DSM_GLOBAL_* */
    float g_eps;         /* epsilon of the global AdamW step, > 0 when global_mode is DSM_GLOBAL_ADAMW */
} dsm_hparams;

/* Statistics of one global step for one tensor (Algorithm 1's quantities):
 *   delta_sq  = sum_e Delta_e^2, Delta = (1/n) sum_i (x - x_i)      (pseudo-gradient norm, times gamma^2)
 *   drift     = sum_e sum_i ((x_e - x_{i,e}) - Delta_e)^2           (spread of the workers around their mean)
 *   zero_sign = #{e : applied sign = 0}  (for the unsigned variants: sign(u) = 0; signed SlowMo: sign(Delta) = 0)
 *   flips     = #{e : sign(u_e) != sign(Delta_e)}                    (momentum overrides the round's direction;
 *               u is the new momentum for SlowMo and the new first moment for global AdamW)
 *   unanimous = #{e : sign(x_e - x_{i,e}) = sign(Delta_e) for every worker i}
 *   clamped   = #{e : |u_e| > B} in the randomized modes, else 0
 * Per element the terms are fp32 values; they are summed with compensated
 * (TwoSum) fp32 arithmetic per thread and warp and in fp64 beyond, so a
 * tensor's sums are within (n + 2) * 2^-24 relative of the exact sums of
 * the element terms; counts are exact. */
typedef struct {
    double delta_sq;
    double drift;
    uint64_t zero_sign;
    uint64_t flips;
    uint64_t unanimous;
    uint64_t clamped;
} dsm_tensor_stats;

/* Read-only description of a handle. */
typedef struct {
    uint64_t d;            /* model size */
    uint64_t d_stride;     /* elements between consecutive workers in the replica/state/gradient buffers */
    uint32_t n, tau;
    uint32_t num_tensors, num_tiles;
    uint64_t round;        /* t: completed global steps */
    uint32_t local_steps;  /* k: local steps done in the current round (0..tau) */
    float gamma;           /* gamma_t of the current round */
} dsm_info;

typedef struct dsm_handle dsm_handle;

/* Bytes of device memory the arena must hold for the state of Algorithm 1
 * (x_{t,0}, m_t, n replicas x^{(i)}, n base-optimizer states, n gradient
 * buffers, tables and statistics) for this layout, n and hparams; 0 if the
 * arguments are invalid (dsm_last_error() says why).  Host only: touches no
 * GPU.  Errors are those of dsm_create's argument checks. */
size_t dsm_state_bytes(const dsm_layout* layout, uint32_t n, const dsm_hparams* hp);

/* Create a handle over the caller's arena and initialise the state of
 * Algorithm 1's first line: x_{0,0} from x0 (d fp32 values, host or device
 * memory per x0_is_device) or, when x0 is NULL, from the hash
 * initialisation (weights 0.02*(2u-1), LayerNorm weights 1, biases 0);
 * m_0 = 0; every replica = x_{0,0}; base-optimizer states = 0.
 * n in [1, 64], tau >= 1.  Enqueues the initialisation on stream and
 * returns without waiting for it.  On failure *out is set to NULL. */
int dsm_create(const dsm_layout* layout, uint32_t n, uint32_t tau, const dsm_hparams* hp,
               void* dev_arena, size_t arena_bytes, const float* x0, int x0_is_device,
               dsm_stream_t stream, dsm_handle** out);

/* Set gamma_t for the current round: the local steps use it as their
 * learning rate and the global step scales by it (Algorithm 1).  Only
 * between rounds (no local step done yet in this round), else DSM_ESTATE;
 * gamma must be > 0 and finite. */
int dsm_set_gamma(dsm_handle* h, float gamma);

/* Fill every worker's gradient buffer with the synthetic gradient of local
 * step index `step` (conventionally t*tau + k):
 *   g_i[e] = s_T*(u(seed,0,step,e) - 1/2) + fp32(0.1f*s_T)*(u(seed,1,i,e) - 1/2)
 * with u the top 24 bits of a SplitMix64 output scaled by 2^-24, rounded to
 * bf16 (nearest even) when grad_dtype is DSM_BF16.  Stands in for the
 * backward pass.  Worker i draws with index first_worker + i (0 unless
 * dsm_set_first_worker set it).  Asynchronous. */
int dsm_fill_synthetic_grads(dsm_handle* h, uint64_t step, dsm_stream_t stream);

/* Place the handle's n workers at positions first_worker .. first_worker+n-1
 * of a larger set of Algorithm 1's workers: a process that holds one
 * contiguous group of the workers of a worker-sharded deployment (the
 * paper's workers are devices, Sec. 5).  Worker i then draws the synthetic
 * gradient of worker first_worker + i in dsm_fill_synthetic_grads; nothing
 * else depends on it.  Any time; takes effect at the next fill.  DSM_EINVAL
 * for a NULL handle, DSM_ERANGE if first_worker + n exceeds 2^32. */
int dsm_set_first_worker(dsm_handle* h, uint32_t first_worker);

/* Device pointer to worker `worker`'s gradient buffer, for a caller that
 * writes the update directions' inputs itself (the stochastic gradients
 * grad f_i(x^{(i)}, xi^{(i)}) of Eq. (base-sgd)).  The buffer holds d
 * elements of the gradient type; consecutive workers are d_stride elements
 * apart (dsm_get_info).  The pointer stays valid, and owned by the arena,
 * until dsm_destroy.  DSM_EINVAL for NULL arguments, DSM_ERANGE for
 * worker >= n. */
int dsm_grad_ptr(dsm_handle* h, uint32_t worker, void** dev_ptr);

/* Device address of worker `worker`'s current model x^{(i)} (d fp32 values,
 * the caller must not write through it), the point at which Eq. (base-sgd)
 * evaluates that worker's stochastic gradient: a framework runs its forward
 * and backward pass over views of this memory, then writes the gradients
 * through dsm_grad_ptr.  While the replicas' reset is pending (fused round)
 * the address is that of x itself; if the round's last local step is
 * pending, the call first runs it on stream.  The address and its contents
 * stay valid until the next call that changes the state (a local or global
 * step, a write of worker state).  DSM_EINVAL for NULL arguments, DSM_ERANGE
 * for worker >= n, DSM_ECUDA if the pending step fails to launch. */
int dsm_replica_ptr(dsm_handle* h, uint32_t worker, dsm_stream_t stream, const float** dev_ptr);

/* Copy all workers' gradients (the grad f_i of Eq. (base-sgd)) from src, a
 * dense [n][d] array of the gradient type in host (src_is_device = 0;
 * pinned memory makes it asynchronous) or device memory, into the gradient
 * buffers.  src stays the caller's.  DSM_EINVAL for NULL arguments,
 * DSM_ECUDA if the copy fails to enqueue. */
int dsm_load_grads(dsm_handle* h, const void* src, int src_is_device, dsm_stream_t stream);

/* Local step k of the current round on every worker, Eq. (local-steps):
 * the base optimizer's update of each replica from its gradient buffer.
 * AdamW's bias corrections use step count j = t*tau + k + 1 (the
 * base-optimizer states persist across rounds; only the model is
 * synchronised), or j = k + 1 with DSM_FLAG_RESET_LOCAL_STATE.  DSM_ESTATE
 * if tau local steps were already done in this round.  Asynchronous. */
int dsm_local_step(dsm_handle* h, dsm_stream_t stream);

/* Local step k of the current round, Eq. (local-steps), with the gradients
 * of every worker (the grad f_i of Eq. (base-sgd)) taken from host memory,
 * and their transfer overlapped with the update.  src is a dense [n][d]
 * array of the gradient type in host memory, the caller's; pinned memory
 * makes the copies asynchronous (pageable memory works, without overlap).
 * The model is cut into chunks of whole tiles (about 64 MB of gradients
 * each, at most 64): for every chunk the call enqueues the copy of its n
 * gradient slices on copy_stream and, on stream, the local step on that
 * chunk once its copy has landed, so that the copy of one chunk runs while
 * the previous chunk is updated.  The copies start after everything
 * enqueued on stream before the call; work enqueued on stream after the
 * call follows every copy and every update.  copy_stream may equal stream
 * (no overlap).  Same results, bit for bit, as dsm_load_grads followed by
 * dsm_local_step; with the fused round's last step the copies are enqueued
 * and the update is left to dsm_global_step, as for dsm_local_step.  The
 * first call creates the handle's chunk events (cudaEventCreate); the
 * environment variable DSM_HOST_GRAD_CHUNK_BYTES, read then, sets another
 * chunk size.  src must stay unchanged until the copies have completed (until
 * stream reaches work enqueued after the call).
 * DSM_EINVAL for NULL handle or src, DSM_ESTATE as for dsm_local_step,
 * DSM_ECUDA if an event, copy or launch fails to enqueue (the step is then
 * not counted, and the gradients and states are undefined). */
int dsm_local_step_host_grads(dsm_handle* h, const void* src, dsm_stream_t stream, dsm_stream_t copy_stream);

/* Global step of Algorithm 1 after the round's tau local steps (else
 * DSM_ESTATE): Delta = (1/n) sum_{i=0..n-1} (x - x_i) (summed in worker
 * order), u = b1 m + ((1-b1)/gamma) Delta, x' = x - eta gamma (S(u) + lambda x),
 * m' = b2 m + ((1-b2)/gamma) Delta, every replica <- x', with S the sign
 * or the randomized sign (Philox4x32-10, key (seed mod 2^32, t), counter
 * floor(e/4), word e mod 4).  Also computes the per-tensor statistics.
 * If stats is non-NULL (host memory, stats_count >= number of tensors) it
 * copies them there and synchronises the stream; else it is asynchronous. */
int dsm_global_step(dsm_handle* h, dsm_stream_t stream, dsm_tensor_stats* stats, uint32_t stats_count);

/* Device pointer to the per-tensor statistics of the last global step
 * (num_tensors dsm_tensor_stats in the arena; see that struct for the
 * quantities of Algorithm 1 they measure), valid once that step has run on
 * the stream and until the next one.  DSM_EINVAL for NULL arguments. */
int dsm_stats_ptr(dsm_handle* h, const dsm_tensor_stats** dev_ptr);

/* Copy elements [offset, offset+count) of a buffer of Algorithm 1's state
 * (DSM_BUF_*: x_{t,0}, m_t, x^{(i)}, the base optimizer's state, gradients)
 * of worker `worker` (ignored for X, M and GLOBAL_V) to dst (host or device
 * memory, the caller's).  Elements are fp32 except DSM_BUF_GRAD, which has
 * the gradient type.  With a host dst the call synchronises the stream
 * before returning.  DSM_EINVAL for an unknown or absent buffer,
 * DSM_ERANGE for worker >= n or a range outside [0, d). */
int dsm_read_params(dsm_handle* h, int which, uint32_t worker, void* dst, uint64_t offset,
                    uint64_t count, int dst_is_device, dsm_stream_t stream);

/* The reverse of dsm_read_params (checkpoint restore, or a caller-set
 * state of Algorithm 1).  With a host src the call synchronises the
 * stream.  Same errors as dsm_read_params. */
int dsm_write_params(dsm_handle* h, int which, uint32_t worker, const void* src, uint64_t offset,
                     uint64_t count, int src_is_device, dsm_stream_t stream);

/* The paper's learning-rate schedule (Sec. 5, implementations): linear
 * warm-up to `peak` over `warmup_steps` local steps (step s < warmup_steps
 * gives peak*(s+1)/warmup_steps), then a cosine decay to final_ratio*peak at
 * `total_steps` (final_ratio*peak + (peak - final_ratio*peak)*(1 + cos(pi*r))/2
 * with r = (s - warmup_steps)/(total_steps - warmup_steps)), constant after.
 * Algorithm 1 keeps gamma_t fixed within a round: pass step = t*tau and give
 * the result to dsm_set_gamma.  Computed in double, returned as fp32 in
 * *gamma.  DSM_EINVAL if peak <= 0, final_ratio outside [0, 1],
 * warmup_steps > total_steps or total_steps = 0. */
int dsm_cosine_gamma(float peak, float final_ratio, uint64_t warmup_steps, uint64_t total_steps, uint64_t step,
                     float* gamma);

/* Set the round counter t of Algorithm 1 (checkpoint restore): it keys the
 * randomized sign and fixes the AdamW step counts j = t*tau + k + 1 (j = k + 1
 * with DSM_FLAG_RESET_LOCAL_STATE) and the global AdamW count t + 1.  Only
 * between rounds, else DSM_ESTATE. */
int dsm_set_round(dsm_handle* h, uint64_t round);

/* End round t of Algorithm 1 with a global model computed elsewhere.  In a
 * worker-sharded deployment the processes that own the model's parameter
 * ranges compute x_{t+1,0} = x_{t,0} - eta*gamma_t*(S(u_{t+1}) + lambda*x_{t,0})
 * (Eq. (model-update)) and the global momentum, from every worker's model,
 * so the handles that hold the workers do not run dsm_global_step: each
 * ends its round with this call instead.  Needs all tau local steps of the
 * round (DSM_ESTATE otherwise); a last local step deferred by
 * DSM_FLAG_FUSED_ROUND runs first, so that the workers' base-optimizer
 * states are complete.  Then x <- x_next (d fp32 values, in host or device
 * memory, x_is_device), every worker restarts from x (Algorithm 1's
 * synchronisation; the next local step reads x, as after a fused round),
 * t <- t + 1 (the randomized sign's key and the global AdamW count advance
 * as after dsm_global_step) and, with DSM_FLAG_RESET_LOCAL_STATE, the
 * base optimizer restarts.  The handle's own m (and global v) are left as
 * they are.  With host memory the call synchronises the stream.
 * DSM_EINVAL for NULL arguments. */
int dsm_end_round(dsm_handle* h, const float* x_next, int x_is_device, dsm_stream_t stream);

/* Describe the handle (sizes, t and k of Algorithm 1, gamma_t) into *out.
 * Host only.  DSM_EINVAL for NULL arguments. */
int dsm_get_info(const dsm_handle* h, dsm_info* out);

/* Memory-safety check (no counterpart in the paper): every buffer of the
 * arena is followed by a 256-byte guard region filled with 0xA5 at create;
 * a write past the end of any buffer changes it.  Synchronises the stream
 * and sets *bad_regions to the number of guard regions that changed. */
int dsm_check_guards(dsm_handle* h, dsm_stream_t stream, uint32_t* bad_regions);

/* Release the handle's host metadata; the arena stays the caller's and may
 * be freed once the stream's work on it is complete.  NULL is accepted.
 * Infrastructure: no counterpart in the paper. */
int dsm_destroy(dsm_handle* h);

/* Message for the calling thread's last failed call ("" if none); the
 * string is the library's and stays valid until that thread's next failing
 * call.  Infrastructure: no counterpart in the paper. */
const char* dsm_last_error(void);

/* ---- global step without any device allocation ----------------------- */
/* The paper has no counterpart to this entry point; it exists for callers
 * that cannot allocate device memory themselves: code that lives inside a
 * host framework which owns all of HBM through its own pool allocator and
 * forbids outside allocations, or latency-critical loops in which a
 * cudaMalloc/cudaFree (which may block or synchronise the device) is not
 * acceptable.  Such a caller has its model, momentum and replicas in
 * buffers it already owns, but no arena for dsm_create().
 *
 * dsm_global_step_noalloc() runs the same global step as dsm_global_step()
 * (same kernels, bit-identical results) directly on the caller's buffers.
 * Its tile table and per-tile statistics live in one scratch array inside
 * the library, a static device array of DSM_NOALLOC_SCRATCH_BYTES bytes that
 * every GPU which loads the library holds until the process exits.  Nothing
 * is allocated: no cudaMalloc, no cudaFree, no allocating library routine.
 *
 * Limits: at most DSM_NOALLOC_MAX_TENSORS tensors and DSM_NOALLOC_MAX_TILES
 * tiles of 1024 elements (a one-tensor model of up to 2^29 elements); larger
 * layouts return DSM_ERANGE.
 *
 * Arguments: layout, n (1..64) and hp as for dsm_create (the tensor list
 * passes the same checks; of hp only the global fields and the seed are
 * used; global_mode is Algorithm 1's DSM_GLOBAL_SIGN_MOMENTUM or one of the
 * variants that keep only x and m, DSM_GLOBAL_SLOWMO, _SIGNED_SLOWMO and
 * _LOOKAHEAD, with m holding their momentum; DSM_GLOBAL_ADAMW, which also
 * needs a second moment, returns DSM_EINVAL here, and so does a randomized
 * sign_mode with a variant); gamma the round's gamma_t (> 0); round the
 * round index t (it keys the randomized sign); x and m the global model and
 * momentum (d fp32 each); replicas the n worker models (fp32, worker i at
 * replicas + i*replica_stride, replica_stride >= d and a multiple of 8);
 * x, m and replicas 16-byte aligned, and device memory of the current
 * device (checked: DSM_EINVAL otherwise).  x, m and the replicas are
 * updated in place.  stats: NULL, or num_tensors entries in device memory
 * of the current device (stats_is_device = 1) or in host memory (0; the
 * call then copies them there and synchronises the stream).
 *
 * Every call looks up the scratch array's device address on the current
 * device (cudaGetSymbolAddress: a lookup, no allocation).  The first call
 * on a device may load the library's device code there; make that first
 * call before any stream capture.  All calls share the one scratch array
 * and leave their contents in it; nothing in it needs to start at zero,
 * because every call rewrites the parts it reads.  Calls whose work
 * overlaps on the GPU (on different streams, or from different threads, on
 * the same device) race on the scratch array: order them on one stream or
 * serialise them.  The layout's tensor list is copied from host memory to
 * the device on the stream; from pageable host memory that copy has
 * consumed the list when the call returns, from pinned memory the list must
 * stay unchanged until the stream reaches it. */
#define DSM_NOALLOC_MAX_TENSORS 4096u
#define DSM_NOALLOC_MAX_TILES   524288u
#define DSM_NOALLOC_SCRATCH_BYTES 25657344u
int dsm_global_step_noalloc(const dsm_layout* layout, uint32_t n, const dsm_hparams* hp, float gamma,
                            uint64_t round, float* x, float* m, float* replicas, uint64_t replica_stride,
                            dsm_tensor_stats* stats, int stats_is_device, dsm_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* DSM_H */
