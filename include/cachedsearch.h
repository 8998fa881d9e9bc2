/*
 * cachedsearch.h — C ABI of the GB300 (sm_103a) cached-search denoising step.
 *
 * Method: CachedSearch (arxiv 2607.23159).  N search candidates of a flow-matching
 * video DiT are advanced one Euler step at a time (Sec. 2, Eq. euler).  For each
 * candidate the adaptive transformation-vector cache (Sec. 3.1: Eq. delta, Eq. skip,
 * Eq. indicator) decides whether the transformer runs; skipped candidates are
 * compacted out of the transformer batch.  Candidates are scored and the best kept
 * (Algorithm 1).
 *
 * Conventions shared by every call
 *  - Pointers named *_dev are device pointers; ownership stays with the caller
 *    unless stated.  Latent tensors are float32, candidate-major [N][D] with
 *    D = C*F*H*W in (c, f, h, w) row-major order.
 *  - Every call is asynchronous on the given stream unless it says it synchronises;
 *    nothing is thrown across the ABI.  Each returns a cs_status; on failure
 *    cs_last_error() gives a message for the calling thread.
 *  - Kernels wait on nothing without a time limit: a wait that runs out records
 *    CS_ERR_TIMEOUT in the device error word (read by cs_device_error()).
 */
#ifndef CACHEDSEARCH_H
#define CACHEDSEARCH_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  CS_OK = 0,
  CS_ERR_ARG = 1,         /* bad pointer, size or configuration                         */
  CS_ERR_CUDA = 2,        /* a CUDA runtime/driver call failed (message has the reason)  */
  CS_ERR_NONFINITE = 3,   /* a norm in the drift indicator was NaN/Inf or ||x_ref|| = 0   */
  CS_ERR_TIMEOUT = 4,     /* a bounded device-side wait ran out                          */
  CS_ERR_NOMEM = 5,       /* device allocation failed                                    */
  CS_ERR_UNSUPPORTED = 6, /* shape outside what the kernels implement                    */
  CS_ERR_BOUNDS = 7       /* index-checking build only (cs_build_flags() bit 0): a device
                             index read from memory was out of range; the access was
                             skipped and the error recorded in the device error word    */
} cs_status;

/* Shape of the DiT velocity model v_theta(x, t, c) (Sec. 2) and of its latent. */
typedef struct {
  int C, F, H, W;   /* latent channels, frames, height, width (H, W even)               */
  int d;            /* model width                                                      */
  int heads;        /* attention heads; head dim d/heads must be 32 or 128              */
  int ffn;          /* FFN hidden width                                                 */
  int blocks;       /* transformer blocks                                               */
  int f_dim;        /* timestep sinusoid features (even)                                */
  int d_text;       /* raw text-embedding width                                         */
  int Lt;           /* text tokens                                                      */
  int max_batch;    /* most candidates one cs_search_step / cs_dit_forward call takes   */
} cs_model_config;

typedef struct cs_model cs_model;

/* Message for the last failing call on this thread ("" if none). Never NULL. */
const char* cs_last_error(void);

/* Library version string. */
const char* cs_version(void);

/* Build options: bit 0 set when the library was compiled with CS_DEBUG_CHECKS (built by
 * `python -m paper_2607_23159_gb300.build --debug` as lib/libcachedsearch_debug.so).
 * That build checks every index the kernels read from device memory (the compaction list
 * of computing candidates, the guidance K/V set of an item) before using it, records
 * CS_ERR_BOUNDS in the device error word on a violation and skips the access; results are
 * otherwise bit-identical to the normal build.  It stands in for a device memory checker. */
int cs_build_flags(void);

/* Number of float32 parameters of a model of this shape (the length of the flat
 * buffer cs_load_weights takes).  Layout, in order, Linear weights stored [out][in]
 * (y = x W^T + b):
 *   patch_w[d][4C] patch_b[d]  time_w1[d][f_dim] time_b1[d]  time_w2[d][d] time_b2[d]
 *   mod_w[6d][d] mod_b[6d]  text_w1[d][d_text] text_b1[d]  text_w2[d][d] text_b2[d]
 *   head_mod_w[2d][d] head_mod_b[2d]  head_w[4C][d] head_b[4C]
 *   then per block: mod_off[6][d]  qkv_w[3d][d] qkv_b[3d]  o_w[d][d] o_b[d]
 *   cq_w[d][d] cq_b[d]  ckv_w[2d][d] ckv_b[2d]  co_w[d][d] co_b[d]
 *   ff1_w[ffn][d] ff1_b[ffn]  ff2_w[d][ffn] ff2_b[d]
 * Returns 0 for an invalid configuration. */
size_t cs_param_count(const cs_model_config* cfg);

/* Create a model: validates the shape, allocates device weights and the workspace
 * for cfg->max_batch candidates on the current device.  The library owns both;
 * free them with cs_destroy_model.  Errors: CS_ERR_ARG (shape), CS_ERR_UNSUPPORTED,
 * CS_ERR_NOMEM. */
cs_status cs_init_model(const cs_model_config* cfg, cs_model** out);
cs_status cs_destroy_model(cs_model* model);

/* Load all parameters from a flat float32 buffer in the cs_param_count layout (host
 * memory if params_on_device == 0, else device memory).  GEMM weights are stored as
 * bf16 (round to nearest even), biases and the small conditioning MLPs as float32.
 * Synchronises the stream. */
cs_status cs_load_weights(cs_model* model, const float* params, size_t count, int params_on_device,
                          cudaStream_t stream);

/* Number of tensors in the parameter layout above (16 + 15 per block). */
int cs_param_tensor_count(const cs_model_config* cfg);

/* Load one tensor of the layout (index in layout order) from float32 data of exactly its
 * size, host (params_on_device == 0) or device memory; lets a caller stream a large model
 * tensor by tensor instead of building the whole flat buffer.  Synchronises the stream. */
cs_status cs_load_param(cs_model* model, int index, const float* data, size_t count, int params_on_device,
                        cudaStream_t stream);

/* Project the prompt's text context once per search: ctx_dev [Lt][d_text] float32
 * (device).  Computes text = W2 GELU(W1 ctx + b1) + b2 and each block's
 * cross-attention K/V, cached in the model for every later step (the prompt is shared
 * by all candidates, Algorithm 1). */
cs_status cs_set_text_context(cs_model* model, const float* ctx_dev, cudaStream_t stream);

/* Classifier-free guidance (Eq. cfg): the unconditional ("empty prompt") text context
 * ctx_dev [Lt][d_text], projected like cs_set_text_context into a second K/V set per
 * block.  Needed by cs_search_step_cfg. */
cs_status cs_set_null_text_context(cs_model* model, const float* ctx_dev, cudaStream_t stream);

/* Velocity of a compacted subset: for j < n_c, v_dev[idx[j]] = v_theta(x_dev[idx[j]], t, c)
 * (Sec. 2).  idx_dev: int32 [n_c] candidate indices (device); n_c <= max_batch.  Rows of
 * v_dev not named in idx are left untouched. */
cs_status cs_dit_forward(cs_model* model, const float* x_dev, const int32_t* idx_dev, int n_c, float t,
                         float* v_dev, cudaStream_t stream);

/* Bytes of scratch cs_cache_decide / cs_cache_apply / cs_score need for N candidates
 * of D elements. */
size_t cs_cache_workspace_bytes(int N, long long D);

/* Cache rule, part 1 (Sec. 3.1, Eq. indicator).  For every candidate i at step k
 * (1-based) of T:
 *   forced_i = (k <= K_w) || (k > T - K_c) || !has_ref[i]
 *   if !forced_i: a_i += ||x_i - x_ref_i||_F / ||x_ref_i||_F
 *   compute_i = forced_i || tau <= 0 || a_i > tau     (tau <= 0 is "off": always compute)
 *   force_compute (nullable, device u8 [N]) replaces compute_i after the accumulation.
 *   computed candidates get a_i = 0 and has_ref_i = 1.
 * Outputs: skip_mask_dev[i] = 1 if candidate i skips; compute_idx_dev [N] the indices
 * of computing candidates in increasing order; n_compute_dev [1] their count.
 * workspace_dev: cs_cache_workspace_bytes(N, D) bytes of device scratch.
 * err_dev (nullable, device int): receives CS_ERR_NONFINITE when a norm is not finite
 * or ||x_ref|| = 0 (that candidate is then computed), CS_ERR_ARG when force_compute
 * asks an empty cache to skip. */
cs_status cs_cache_decide(const float* x_dev, const float* x_ref_dev, float* accum_dev, uint8_t* has_ref_dev,
                          int N, long long D, int step_k, int T, float tau, int K_w, int K_c,
                          const uint8_t* force_compute_dev, uint8_t* skip_mask_dev, int32_t* compute_idx_dev,
                          int32_t* n_compute_dev, void* workspace_dev, int* err_dev, cudaStream_t stream);

/* Allocation-free form of cs_cache_decide, for callers that cannot allocate device
 * memory: a serving runtime whose memory pool owns the whole device after start-up, or
 * host code that must not let an allocation synchronise the device mid-step.  It takes
 * no workspace; the partial sums live in a fixed array compiled into the library (one
 * per GPU that loads it, kept until the process exits, 256 KB).  The paper has no
 * counterpart: this is a deployment convenience of this library.
 *   Limits: N <= CS_NOALLOC_MAX_N candidates and D <= CS_NOALLOC_MAX_CHUNKS * 8192
 *   elements per candidate; larger sizes return CS_ERR_ARG with a message, nothing runs.
 *   The first call on a device looks up the array's device address (cudaGetSymbolAddress)
 *   with that device current; make that first call before any stream capture.  The
 *   address is kept for the life of the process: after cudaDeviceReset on that device
 *   it would be stale, so a process that resets a device must not call this again.
 *   All calls on a device share the array: calls that overlap on the GPU (other streams
 *   or threads) race and must be serialised by the caller.  Each call writes every
 *   partial it reads, so nothing from a previous call needs clearing.
 * Arguments, results and errors are those of cs_cache_decide. */
#define CS_NOALLOC_MAX_N 64
#define CS_NOALLOC_MAX_CHUNKS 512
cs_status cs_cache_decide_noalloc(const float* x_dev, const float* x_ref_dev, float* accum_dev,
                                  uint8_t* has_ref_dev, int N, long long D, int step_k, int T, float tau,
                                  int K_w, int K_c, const uint8_t* force_compute_dev, uint8_t* skip_mask_dev,
                                  int32_t* compute_idx_dev, int32_t* n_compute_dev, int* err_dev,
                                  cudaStream_t stream);

/* Cache rule, part 2, fused with the Euler update (Eq. delta, Eq. skip, Eq. euler),
 * h = t_next - t_cur:
 *   skipped:  x += h (x + Delta)
 *   computed: Delta = v - x;  x_ref = x;  x += h v       (v_dev [N][D], rows of computed candidates)
 * If target_dev (device [D]) is given, scores_dev[i] = -||x0_i - target||_2 with the x0
 * estimate x0_i = x_next_i - t_next * v_used_i (x_next itself on the last step). */
cs_status cs_cache_apply(float* x_dev, float* x_ref_dev, float* delta_dev, const float* v_dev,
                         const uint8_t* skip_mask_dev, int N, long long D, float t_cur, float t_next,
                         const float* target_dev, float* scores_dev, void* workspace_dev, cudaStream_t stream);

/* Guided forms (Eq. cfg with per-branch cache state, Sec. 3.1): each candidate i has two
 * cache states, row i (conditional branch) and row N + i (unconditional branch), that
 * share its latent x_i and decide independently.  x_ref, delta: [2N][D]; accum, has_ref,
 * force_compute, skip_mask: [2N]; compute_idx: [2N] state rows; workspace:
 * cs_cache_workspace_bytes(2N, D).  The apply step combines the two branch velocities
 * (computed v_b, or x + Delta_b when skipped) as v_u + w (v_c - v_u) and takes the Euler
 * step with it; scores use that combined velocity in the x0 estimate. */
cs_status cs_cache_decide_cfg(const float* x_dev, const float* x_ref_dev, float* accum_dev, uint8_t* has_ref_dev,
                              int N, long long D, int step_k, int T, float tau, int K_w, int K_c,
                              const uint8_t* force_compute_dev, uint8_t* skip_mask_dev, int32_t* compute_idx_dev,
                              int32_t* n_compute_dev, void* workspace_dev, int* err_dev, cudaStream_t stream);
cs_status cs_cache_apply_cfg(float* x_dev, float* x_ref_dev, float* delta_dev, const float* v_dev,
                             const uint8_t* skip_mask_dev, int N, long long D, float t_cur, float t_next, float w,
                             const float* target_dev, float* scores_dev, void* workspace_dev, cudaStream_t stream);

/* One guided denoising step of N candidates: both branches' decisions, one DiT forward
 * of all computing branch items (conditional items use the prompt's K/V, unconditional
 * items the null context's), then the guided update.  2N <= max_batch.  Same state
 * conventions as the guided forms above; *n_computed counts branch items. */
cs_status cs_search_step_cfg(cs_model* model, float* x_dev, float* x_ref_dev, float* delta_dev, float* accum_dev,
                             uint8_t* has_ref_dev, int N, int step_k, int T, float t_cur, float t_next, float tau,
                             int K_w, int K_c, float guidance, const uint8_t* force_compute_dev,
                             uint8_t* skip_mask_dev, const float* target_dev, float* scores_dev, int* n_computed,
                             cudaStream_t stream);

/* Single-pass form used by cs_search_step.  cs_cache_decide_skip takes the decision of
 * every candidate (as cs_cache_decide, with the same arithmetic and results) and applies
 * Eq. skip + Eq. euler to the skipped ones (writing their score partials if target_dev
 * is given), so that a skipped candidate's x_ref and Delta are read once, x read while
 * still in L2 and written once.  Two launches and no grid-wide wait: the drift pass,
 * in which the CTA that arrives last on one counter takes every decision, then the skip
 * update, scheduled by programmatic dependent launch while the first drains.  Needs
 * D % 8 == 0, 32-byte aligned tensors and cs_cache_workspace_bytes(N, D) of workspace
 * (its arrival counter is cleared by the call).  cs_cache_apply_computed then updates
 * only the computed candidates (Eq. delta + Eq. euler, v_dev from the DiT) and, with
 * target_dev, finalises the scores of all candidates. */
cs_status cs_cache_decide_skip(float* x_dev, const float* x_ref_dev, const float* delta_dev, float* accum_dev,
                               uint8_t* has_ref_dev, int N, long long D, int step_k, int T, float t_cur,
                               float t_next, float tau, int K_w, int K_c, const uint8_t* force_compute_dev,
                               uint8_t* skip_mask_dev, int32_t* compute_idx_dev, int32_t* n_compute_dev,
                               const float* target_dev, void* workspace_dev, int* err_dev, cudaStream_t stream);
cs_status cs_cache_apply_computed(float* x_dev, float* x_ref_dev, float* delta_dev, const float* v_dev,
                                  const uint8_t* skip_mask_dev, int N, long long D, float t_cur, float t_next,
                                  const float* target_dev, float* scores_dev, void* workspace_dev,
                                  cudaStream_t stream);

/* The computed candidates' update taken directly from the DiT head's output in token
 * layout (the unpatchify scatter fused with Eq. delta and Eq. euler), so that the
 * velocity is never written to memory as a latent.  For j < n_c, candidate i = idx[j]
 * and latent element (c, f, h, w) of a [C][F][H][W] latent:
 *   v = hout[(j*L + l)*4C + 4c + 2(h%2) + (w%2)],  l = (f*(H/2) + h/2)*(W/2) + w/2,
 *   Delta_i = v - x_i;  x_ref_i = x_i;  x_i += (t_next - t_cur) v;
 *   accum[i] = 0, has_ref[i] = 1, skip_mask[i] = 0.
 * hout_dev: float32 [n_c * L][4C] (the head Linear's output rows of the compacted batch).
 * Needs even H, W % 4 == 0 and 16-byte aligned tensors.  With target_dev, the computed
 * candidates' score partials go to tile_partials_dev (float32 [N][F*H/2]) and
 * scores_dev[i] = -||x0_i - target||_2 is finalised for all N candidates, the skipped
 * ones from the partials cs_cache_decide_skip left in workspace_dev (same target). */
cs_status cs_cache_apply_tokens(float* x_dev, float* x_ref_dev, float* delta_dev, float* accum_dev,
                                uint8_t* has_ref_dev, uint8_t* skip_mask_dev, const float* hout_dev,
                                const int32_t* compute_idx_dev, int n_c, int N, int C, int F, int H, int W,
                                float t_cur, float t_next, const float* target_dev, float* scores_dev,
                                void* workspace_dev, float* tile_partials_dev, int* err_dev, cudaStream_t stream);

/* Carried form of the two calls above (Sec. 3.1, Eq. indicator, Eq. skip, Eq. euler), the
 * one cs_search_step runs.  The drift of step k needs ||x - x_ref|| and ||x_ref|| of the
 * latent a candidate holds at step k, which the update of step k - 1 writes: these calls
 * make every update also leave those two squared norms for the next step (the "carried"
 * drift), so that a step takes its decisions without reading x or x_ref and its skip
 * update is the only pass over a skipped candidate's state (read x, Delta, x_ref; write
 * x).  Results are those of cs_cache_decide_skip + cs_cache_apply_tokens except for the
 * order in which the drift's sums are added (float32, fixed per candidate).
 *   has_ref = 3 (bit 1 set) marks a candidate whose carried sums belong to its current
 *   x and x_ref; the carrying calls leave 3, every other call leaves 1 (or 0).  A caller
 *   that changes x or x_ref of a candidate between two steps in any other way must clear
 *   bit 1 of its has_ref (has_ref &= 1).
 *   step_ws_dev: cs_cache_step_bytes(N, C, F, H, W) bytes of device memory, zero-filled
 *   before its first use and then kept with the state (it holds the carried sums per
 *   candidate row, by the parity of step_k); every call leaves its counters at zero.
 *   Use one step_ws with one N and latent shape.
 *   carried = 1: on a free step the decisions use the sums the previous step (step_k - 1)
 *   left.  If a cached candidate has none (has_ref == 1), the call changes nothing and
 *   writes *n_compute_dev = -1: call again with carried = 0.  carried = 0: a drift pass
 *   reads x and x_ref (as cs_cache_decide_skip), then the skip update runs.  Inside the
 *   warm-up / cool-down window no drift is needed and `carried` does not matter.
 *   Either way the skipped candidates leave their sums for step_k + 1 (has_ref = 3), and
 *   cs_cache_apply_tokens_carry does the same for the computed ones.
 * Latent shape and alignment as cs_cache_apply_tokens; N <= 4096.  Errors as
 * cs_cache_decide_skip. */
size_t cs_cache_step_bytes(int N, int C, int F, int H, int W);
cs_status cs_cache_decide_skip_carry(float* x_dev, const float* x_ref_dev, const float* delta_dev,
                                     float* accum_dev, uint8_t* has_ref_dev, int N, int C, int F, int H, int W,
                                     int step_k, int T, float t_cur, float t_next, float tau, int K_w, int K_c,
                                     const uint8_t* force_compute_dev, uint8_t* skip_mask_dev,
                                     int32_t* compute_idx_dev, int32_t* n_compute_dev, const float* target_dev,
                                     int carried, void* step_ws_dev, int* err_dev, cudaStream_t stream);
cs_status cs_cache_apply_tokens_carry(float* x_dev, float* x_ref_dev, float* delta_dev, float* accum_dev,
                                      uint8_t* has_ref_dev, uint8_t* skip_mask_dev, const float* hout_dev,
                                      const int32_t* compute_idx_dev, int n_c, int N, int C, int F, int H, int W,
                                      int step_k, float t_cur, float t_next, const float* target_dev,
                                      float* scores_dev, void* step_ws_dev, int* err_dev, cudaStream_t stream);

/* One denoising step of N candidates (the unit of work of the search):
 * cs_cache_decide_skip, then the DiT forward (as cs_dit_forward) on the computing
 * subset, then the computed candidates' update from the head's token output
 * (cs_cache_apply_tokens; latents with W % 4 != 0 take the velocity scatter and
 * cs_cache_apply_computed instead).
 * State buffers (x, x_ref, delta: [N][D]; accum: [N]; has_ref: [N]) are caller-owned
 * device memory and are updated in place; a fresh search starts with has_ref = 0.
 * With the token-layout update, the step takes the carried form
 * (cs_cache_decide_skip_carry, cs_cache_apply_tokens_carry) with the model's own step
 * workspace: a step uses the drift sums the previous call left when that call was step
 * k - 1 on the same state buffers and N, and otherwise (or when a candidate's has_ref is
 * 1) runs the drift pass; writes to x or x_ref between steps other than through these
 * calls must clear bit 1 of the candidate's has_ref, as described there.
 * Synchronises once to read the number of computing candidates; that count is returned
 * in *n_computed (host, nullable).  A warm-up or cool-down step without a forced mask
 * computes every candidate (Sec. 3.1): it takes no decision pass and does not
 * synchronise, so a device error recorded during it is returned by the next call that
 * synchronises (a free step, cs_search_step_host or cs_device_error). */
cs_status cs_search_step(cs_model* model, float* x_dev, float* x_ref_dev, float* delta_dev, float* accum_dev,
                         uint8_t* has_ref_dev, int N, int step_k, int T, float t_cur, float t_next, float tau,
                         int K_w, int K_c, const uint8_t* force_compute_dev, uint8_t* skip_mask_dev,
                         const float* target_dev, float* scores_dev, int* n_computed, cudaStream_t stream);

/* The same step with the latents in HOST memory (x_host [N][D], in/out) and the skip
 * mask returned to HOST memory (skip_mask_host [N]); the cache state stays on the
 * device.  Copies in, steps, copies out, and synchronises. */
cs_status cs_search_step_host(cs_model* model, float* x_host, float* x_ref_dev, float* delta_dev,
                              float* accum_dev, uint8_t* has_ref_dev, int N, int step_k, int T, float t_cur,
                              float t_next, float tau, int K_w, int K_c, uint8_t* skip_mask_host,
                              int* n_computed, cudaStream_t stream);

/* scores_dev[i] = -||x_i - target||_2: the stand-in for the verifier score that Algorithm 1
 * assigns to each explored candidate. */
cs_status cs_score(const float* x_dev, const float* target_dev, int N, long long D, float* scores_dev,
                   void* workspace_dev, cudaStream_t stream);

/* Indices of the k largest scores in descending order (Algorithm 1, argmax when k = 1);
 * equal scores keep the lower index first; NaN ranks below every number.  N <= 4096. */
cs_status cs_select_topk(const float* scores_dev, int N, int k, int32_t* idx_dev, cudaStream_t stream);

/* Beam refill: destination slot s = p*(1+children) + j takes the full state of
 * candidate survivors[p] (x, x_ref, delta, accum, has_ref as 0 or 1: a carried drift
 * belongs to the source row and is not copied); for j > 0 (a child) it adds
 * sigma * noise[p*children + j - 1] to x.  src and dst buffers must not overlap.
 * survivors_dev: int32 [keep]; noise_dev: [keep*children][D]. */
cs_status cs_beam_refill(const float* src_x, const float* src_x_ref, const float* src_delta,
                         const float* src_accum, const uint8_t* src_has_ref, float* dst_x, float* dst_x_ref,
                         float* dst_delta, float* dst_accum, uint8_t* dst_has_ref, const int32_t* survivors_dev,
                         int keep, int children, float sigma, const float* noise_dev, long long D,
                         cudaStream_t stream);

/* First error recorded by the model's kernels since the last call (0 = none); clears
 * it.  Synchronises the stream. */
cs_status cs_device_error(cs_model* model, int* code, cudaStream_t stream);

/* Per-kernel-class timing: when enabled, the model brackets every launch of the
 * class with CUDA events on its stream.  Classes: 0 self-attention, 1 cross-attention,
 * 2 GEMM, 3 cache decide+apply, 4 other.  cs_kernel_stats synchronises and returns
 * the launches, summed milliseconds and algorithmic work (FLOPs for 0-2, bytes for 3)
 * since the last reset. */
cs_status cs_set_profiling(cs_model* model, int enable);
cs_status cs_kernel_stats(cs_model* model, int kernel_class, long long* launches, double* total_ms,
                          double* work);
cs_status cs_reset_kernel_stats(cs_model* model);

/* Kernel launches this library has issued in this process (all entry points). */
long long cs_launch_count(void);

/* Self-test of the failure path (the paper has no counterpart).  Launches one kernel
 * whose thread waits on an mbarrier that nothing arrives on, with the bounded wait every
 * kernel of this library uses: after CS_WAIT_TIMEOUT_NS (2 s) of GPU time the wait gives
 * up, CS_ERR_TIMEOUT is written to *err_dev (device int, first error wins: clear it
 * first) and the kernel returns, so the CUDA context stays usable.  Returns CS_OK once
 * the launch is queued on `stream`, CS_ERR_ARG for a null err_dev. */
cs_status cs_selftest_bounded_wait(int* err_dev, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* CACHEDSEARCH_H */
