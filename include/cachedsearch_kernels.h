/*
 * cachedsearch_kernels.h — C ABI of the individual sm_103a kernels that make up the
 * DiT velocity model v_theta(x, t, c) (Sec. 2) inside cs_dit_forward.  Exposed for
 * callers that drive the blocks themselves and for parity tests.
 *
 * All pointers are device pointers owned by the caller; all calls are asynchronous on
 * the given stream.  bf16 tensors are __nv_bfloat16 passed as void*.  err_dev
 * (nullable, device int) receives CS_ERR_TIMEOUT if a bounded wait inside a kernel
 * runs out.
 */
#ifndef CACHEDSEARCH_KERNELS_H
#define CACHEDSEARCH_KERNELS_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime.h>

#include "cachedsearch.h"

#ifdef __cplusplus
extern "C" {
#endif

/* GEMM epilogues (acc = A B^T in float32, then + bias[n] if bias is given). */
typedef enum {
  CS_EPI_F32 = 0,        /* out_f32[m][n]  = acc                                              */
  CS_EPI_BF16 = 1,       /* out_bf16[m][n] = bf16(acc)                                         */
  CS_EPI_GELU_BF16 = 2,  /* out_bf16[m][n] = bf16(GELU_tanh(acc))                              */
  CS_EPI_RESID_F32 = 3,  /* out_f32[m][n] += gate[n] * acc   (gate NULL: += acc); residual add */
  CS_EPI_QKV = 4         /* scatter into per-head Q, K and transposed V (cs_gemm_qkv)          */
} cs_epilogue;

/* C = A B^T on the tcgen05 tensor cores: A bf16 [M][K] row-major (K contiguous), B bf16
 * [N][K] row-major (a Linear weight [out][in]), float32 accumulation in TMEM, fused
 * epilogue `epi` writing out [M][ldo].  Requirements: K % 64 == 0, ldo >= N, A and B
 * 16-byte aligned.  The K loop runs in the same order for every output tile, and the
 * tile shape depends only on N, so a row's result does not depend on M. */
cs_status cs_gemm_bf16(const void* A_dev, const void* B_dev, int M, int N, int K, int epi,
                       const float* bias_dev, const float* gate_dev, void* out_dev, int ldo, int* err_dev,
                       cudaStream_t stream);

/* Same GEMM with the attention-layout epilogue.  Row m = j*L + l is token l of batch
 * item j; column n = w*d + head*hd + e is element e of head `head` of projection
 * w in [0, N/d) ('which' = which_base + w: 0 = Q, 1 = K, 2 = V).  Writes
 *   Q/K: q_dev/k_dev [j*heads + head][l][hd_s]  (hd_s = max(hd, 64); columns >= hd untouched)
 *   V:   vt_dev      [j*heads + head][e][Lv]    (transposed; Lv >= L, Lv % 8 == 0)
 * hd must be 32 or 128 and d = heads * hd. */
cs_status cs_gemm_qkv(const void* A_dev, const void* B_dev, int M, int N, int K, const float* bias_dev, int L,
                      int d, int heads, int which_base, void* q_dev, void* k_dev, void* vt_dev, int Lv,
                      int* err_dev, cudaStream_t stream);

/* Flash attention on the tcgen05 tensor cores, one (batch item, head) per grid row:
 *   O[j][l][head*hd + e] = sum_m softmax_m(Q[bh][l] . K[bkv][m] / sqrt(hd)) V[bkv][m][e]
 * with bh = j*heads + head and bkv = kv_shared ? head : bh (cross-attention shares one
 * K/V set among all batch items).  q_dev [B*heads][Lq][hd_s], k_dev [Bkv][Lk][hd_s],
 * vt_dev [Bkv][hd][Lkv_stride] (V transposed), all bf16 with hd_s = max(hd, 64) and
 * columns >= hd of Q and K equal to zero; o_dev bf16 [B][Lq][heads*hd].
 * hd in {32, 128}; Lq, Lk >= 1; Lkv_stride >= Lk, % 8 == 0. */
cs_status cs_attention(const void* q_dev, const void* k_dev, const void* vt_dev, void* o_dev, int B, int heads,
                       int Lq, int Lk, int hd, int Lkv_stride, int kv_shared, int* err_dev, cudaStream_t stream);

/* adaLN-modulated LayerNorm (no affine, eps 1e-6) of float32 rows, bf16 out:
 *   out[m][c] = bf16( (x[m][c] - mean_m) / sqrt(var_m + eps) * (1 + scale[c]) + shift[c] )
 * shift/scale [d] float32, either NULL for a plain LayerNorm. */
cs_status cs_layernorm_modulate(const float* x_dev, const float* shift_dev, const float* scale_dev,
                                void* out_dev, int M, int d, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* CACHEDSEARCH_KERNELS_H */
