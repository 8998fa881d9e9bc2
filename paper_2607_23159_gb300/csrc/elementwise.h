// Internal interfaces between the library's translation units.
#pragma once
#include <cstdint>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "../../include/cachedsearch.h"

namespace cs {

struct CondWeights {
  int d, f_dim, blocks;
  const __nv_bfloat16 *time_w1, *time_w2, *mod_w, *head_mod_w;
  const float *time_b1, *time_b2, *mod_b, *head_mod_b;
  const float* const* mod_offs;   // device array of `blocks` pointers to [6][d]
};

// scratch: f_dim + 9 d floats; mods: [blocks][6][d]; hmod: [2][d] (shift, scale)
cs_status timestep_conditioning(const CondWeights& w, float t, float* scratch, float* mods, float* hmod,
                                cudaStream_t s);
cs_status layernorm_modulate(const float* x, const float* shift, const float* scale, __nv_bfloat16* out, int M, int d,
                             cudaStream_t s);
// tokens of latent rows idx[j] % x_rows (x_rows: rows of x; a cache state index may
// exceed it when several states share a latent, as the two guidance branches do);
// idx_limit: valid state indices are [0, idx_limit) (checked in CS_DEBUG_CHECKS builds)
cs_status patchify(const float* x, const int32_t* idx, int n_c, int x_rows, int C, int F, int H, int W, int Kp,
                   __nv_bfloat16* tok, long long idx_limit, int* err, cudaStream_t s);
// self/cross attention; with kv_sets > 1 batch item j uses shared K/V set item_idx[j] / x_rows
cs_status attention_run(const void* q, const void* k, const void* vt, void* o, int B, int heads, int Lq, int Lk,
                        int hd, int Lkv_stride, int kv_shared, int kv_sets, const int32_t* item_idx, int x_rows,
                        int* err, cudaStream_t stream);
cs_status unpatchify(const float* hout, const int32_t* idx, int n_c, int C, int F, int H, int W, float* v,
                     long long idx_limit, int* err, cudaStream_t s);
cs_status to_bf16_pad(const float* src, long long rows, int cols, int ld, __nv_bfloat16* dst, cudaStream_t s);

// cache.cu: the single-pass decide + skip and its small scratch (counter: the arrival
// counter, zero on entry and left zero; sidx: N + 1 ints, the skipped candidates and their
// count; both nullptr for the pair inside the workspace, cleared by the call), and the
// computed update from the head's token output (spart: the skipped candidates' score
// partials; tpart [N][F*H/2]).
struct StepScratch {
  unsigned* counter = nullptr;
  int32_t* sidx = nullptr;
};
cs_status decide_skip_run(float* x, const float* x_ref, const float* delta, float* accum, uint8_t* has_ref, int N,
                          long long D, int step_k, int T, float t_cur, float t_next, float tau, int K_w, int K_c,
                          const uint8_t* force, uint8_t* skip_mask, int32_t* idx, int32_t* n_compute,
                          const float* target, void* workspace, StepScratch sc, int* err, cudaStream_t stream);
cs_status apply_tokens_run(float* x, float* x_ref, float* delta, float* accum, uint8_t* has_ref, uint8_t* skip_mask,
                           const float* hout, const int32_t* idx, int n_c, int N, int C, int F, int H, int W,
                           float t_cur, float t_next, const float* target, float* scores, const float* spart,
                           float* tpart, long long idx_limit, int* err, cudaStream_t stream);
bool apply_tokens_supported(int C, int F, int H, int W);

// The carried form of the step's cache work (the drift of the next step left by each
// update): a step workspace of carry_state_bytes(cap, D, ntiles) bytes, zero-filled once,
// holding `cap` candidate slots (ntiles = F*H/2).  carry_decide_skip_run takes the
// decisions from the carried drift when `carried` (or inside the window, where none is
// needed), else from a drift pass; it reports *n_compute = -1 and changes nothing when a
// cached candidate carries no drift.  carry_apply_tokens_run is apply_tokens_run that
// also leaves the computed candidates' drift for step_k + 1.
struct CarryState {
  void* base;
  int cap;
  long long D;
  int ntiles;
};
size_t carry_state_bytes(int cap, long long D, int ntiles);
cs_status carry_decide_skip_run(float* x, const float* x_ref, const float* delta, float* accum, uint8_t* has_ref,
                                int N, int step_k, int T, float t_cur, float t_next, float tau, int K_w, int K_c,
                                const uint8_t* force, uint8_t* skip_mask, int32_t* idx, int32_t* n_compute,
                                const float* target, bool carried, const CarryState& cs, int* err,
                                cudaStream_t stream);
cs_status carry_apply_tokens_run(float* x, float* x_ref, float* delta, float* accum, uint8_t* has_ref,
                                 uint8_t* skip_mask, const float* hout, const int32_t* idx, int n_c, int N, int C,
                                 int F, int H, int W, int step_k, float t_cur, float t_next, const float* target,
                                 float* scores, const CarryState& cs, long long idx_limit, int* err,
                                 cudaStream_t stream);
cs_status load_cache_kernels();

}  // namespace cs
