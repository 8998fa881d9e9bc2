// Memory-bound pieces of the DiT forward around the tensor-core kernels:
// adaLN-modulated LayerNorm, patchify gather / unpatchify scatter of the computing
// candidates (the compaction of Sec. 3.1's skipped candidates out of the batch),
// the timestep conditioning (sinusoid + small MLPs as GEMVs), and weight conversion.
#include <cuda_bf16.h>

#include "common.cuh"
#include "elementwise.h"
#include "ptx.cuh"

namespace cs {

// ------------------------------------------------------------- LayerNorm ----
// One warp per row; mean, then the centred second moment, then the normalised,
// modulated bf16 row (three passes over a row that stays in L1).
__global__ void __launch_bounds__(256) ln_modulate_kernel(const float* __restrict__ x,
                                                          const float* __restrict__ shift,
                                                          const float* __restrict__ scale,
                                                          __nv_bfloat16* __restrict__ out, int M, int d) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= M) return;
  const float4* row = reinterpret_cast<const float4*>(x + (long long)warp * d);
  const int n4 = d >> 2;
  float s = 0.f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = row[i];
    s += (v.x + v.y) + (v.z + v.w);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  const float mean = s / (float)d;
  float q = 0.f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = row[i];
    const float a = v.x - mean, b = v.y - mean, c = v.z - mean, e = v.w - mean;
    q += (a * a + b * b) + (c * c + e * e);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  const float rstd = rsqrtf(q / (float)d + 1e-6f);
  uint2* orow = reinterpret_cast<uint2*>(out + (long long)warp * d);
  for (int i = lane; i < n4; i += 32) {
    const float4 v = row[i];
    float y0 = (v.x - mean) * rstd, y1 = (v.y - mean) * rstd, y2 = (v.z - mean) * rstd, y3 = (v.w - mean) * rstd;
    if (scale) {
      const float4 sc = __ldg(reinterpret_cast<const float4*>(scale) + i);
      y0 *= 1.f + sc.x; y1 *= 1.f + sc.y; y2 *= 1.f + sc.z; y3 *= 1.f + sc.w;
    }
    if (shift) {
      const float4 sh = __ldg(reinterpret_cast<const float4*>(shift) + i);
      y0 += sh.x; y1 += sh.y; y2 += sh.z; y3 += sh.w;
    }
    orow[i] = make_uint2(pack_bf16x2(y0, y1), pack_bf16x2(y2, y3));
  }
}

cs_status layernorm_modulate(const float* x, const float* shift, const float* scale, __nv_bfloat16* out, int M, int d,
                             cudaStream_t s) {
  if (M <= 0 || d <= 0 || (d % 4) != 0) {
    set_error("layernorm: need M > 0 and d %% 4 == 0");
    return CS_ERR_ARG;
  }
  const int blocks = (int)(((long long)M * 32 + 255) / 256);
  ln_modulate_kernel<<<blocks, 256, 0, s>>>(x, shift, scale, out, M, d);
  CS_LAUNCHED();
  return CS_OK;
}

// ------------------------------------------------------- patchify / scatter ----
// tokens[j*L + l][k]: for k < 4C, element (c, f, 2hh+ph, 2ww+pw) of candidate idx[j]
// with k = 4c + 2ph + pw and l = (f*(H/2) + hh)*(W/2) + ww; columns 4C..Kp-1 are 0.
__global__ void patchify_kernel(const float* __restrict__ x, const int32_t* __restrict__ idx, int n_c, int x_rows,
                                int C, int F, int H, int W, int Kp, __nv_bfloat16* __restrict__ tok,
                                long long idx_limit, int* err) {
  const int L = F * (H / 2) * (W / 2);
  const long long total = (long long)n_c * L * Kp;
  const long long D = (long long)C * F * H * W;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const int k = (int)(t % Kp);
    const long long row = t / Kp;
    const int l = (int)(row % L), j = (int)(row / L);
    float v = 0.f;
    if (k < 4 * C && index_ok(idx[j], idx_limit, err)) {
      const int c = k >> 2, ph = (k >> 1) & 1, pw = k & 1;
      const int ww = l % (W / 2), hh = (l / (W / 2)) % (H / 2), f = l / ((W / 2) * (H / 2));
      v = x[(long long)(idx[j] % x_rows) * D + (((long long)c * F + f) * H + (2 * hh + ph)) * W + (2 * ww + pw)];
    }
    tok[t] = __float2bfloat16_rn(v);
  }
}

// v[idx[j]][c][f][h][w] = hout[(j*L + l)*P + 4c + 2(h%2) + (w%2)]
__global__ void unpatchify_kernel(const float* __restrict__ hout, const int32_t* __restrict__ idx, int n_c, int C,
                                  int F, int H, int W, float* __restrict__ v, long long idx_limit, int* err) {
  const int L = F * (H / 2) * (W / 2), P = 4 * C;
  const long long D = (long long)C * F * H * W;
  const long long total = (long long)n_c * D;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long e = t % D;
    const int j = (int)(t / D);
    const int w = (int)(e % W), h = (int)((e / W) % H), f = (int)((e / ((long long)W * H)) % F);
    const int c = (int)(e / ((long long)W * H * F));
    const int l = (f * (H / 2) + h / 2) * (W / 2) + w / 2;
    if (index_ok(idx[j], idx_limit, err))
      v[(long long)idx[j] * D + e] = hout[((long long)j * L + l) * P + 4 * c + 2 * (h & 1) + (w & 1)];
  }
}

cs_status patchify(const float* x, const int32_t* idx, int n_c, int x_rows, int C, int F, int H, int W, int Kp,
                   __nv_bfloat16* tok, long long idx_limit, int* err, cudaStream_t s) {
  const long long total = (long long)n_c * F * (H / 2) * (W / 2) * Kp;
  const int blocks = (int)((total + 255) / 256 < 65535 * 16 ? (total + 255) / 256 : 65535 * 16);
  patchify_kernel<<<blocks, 256, 0, s>>>(x, idx, n_c, x_rows, C, F, H, W, Kp, tok, idx_limit, err);
  CS_LAUNCHED();
  return CS_OK;
}

cs_status unpatchify(const float* hout, const int32_t* idx, int n_c, int C, int F, int H, int W, float* v,
                     long long idx_limit, int* err, cudaStream_t s) {
  const long long total = (long long)n_c * C * F * H * W;
  const int blocks = (int)((total + 255) / 256 < 65535 * 16 ? (total + 255) / 256 : 65535 * 16);
  unpatchify_kernel<<<blocks, 256, 0, s>>>(hout, idx, n_c, C, F, H, W, v, idx_limit, err);
  CS_LAUNCHED();
  return CS_OK;
}

// ----------------------------------------------------------- conditioning ----
// [cos(1000 t f_j), sin(1000 t f_j)], f_j = exp(-ln(1e4) j / half), in double.
__global__ void sinusoid_kernel(float t, int f_dim, float* __restrict__ out) {
  const int half = f_dim / 2;
  for (int j = threadIdx.x; j < half; j += blockDim.x) {
    const double fr = exp(-log(10000.0) * (double)j / (double)half);
    const double a = 1000.0 * (double)t * fr;
    out[j] = (float)cos(a);
    out[half + j] = (float)sin(a);
  }
}

__device__ __forceinline__ float silu(float x) { return x / (1.f + expf(-x)); }

// out[o] = act(sum_i W[o][i] in[i] + b[o]) (+ add[o]); one warp per output row.
// act: 0 none, 1 SiLU.  W is bf16 [rows][cols].
__global__ void gemv_kernel(const __nv_bfloat16* __restrict__ W, const float* __restrict__ b,
                            const float* __restrict__ in, int rows, int cols, int act, float* __restrict__ out) {
  const int o = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (o >= rows) return;
  const __nv_bfloat16* w = W + (long long)o * cols;
  float s = 0.f;
  for (int i = lane; i < cols; i += 32) s += __bfloat162float(w[i]) * in[i];
#pragma unroll
  for (int k = 16; k > 0; k >>= 1) s += __shfl_xor_sync(0xffffffffu, s, k);
  if (lane == 0) {
    s += b ? b[o] : 0.f;
    out[o] = act == 1 ? silu(s) : s;
  }
}

__global__ void silu_kernel(const float* __restrict__ in, int n, float* __restrict__ out) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) out[i] = silu(in[i]);
}

// mods[b][r][c] = shared[r*d + c] + off_b[r][c] for every block b
__global__ void block_mods_kernel(const float* __restrict__ shared, const float* const* __restrict__ offs, int blocks,
                                  int n6d, float* __restrict__ mods) {
  const long long total = (long long)blocks * n6d;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const int b = (int)(t / n6d), i = (int)(t % n6d);
    mods[t] = shared[i] + offs[b][i];
  }
}

cs_status timestep_conditioning(const CondWeights& w, float t, float* scratch, float* mods, float* hmod,
                                cudaStream_t s) {
  const int d = w.d;
  float* sinus = scratch;            // [f_dim]
  float* h1 = sinus + w.f_dim;       // [d]
  float* e = h1 + d;                 // [d]
  float* se = e + d;                 // [d]
  float* shared = se + d;            // [6d]
  sinusoid_kernel<<<1, 128, 0, s>>>(t, w.f_dim, sinus);
  CS_LAUNCHED();
  auto gemv = [&](const __nv_bfloat16* W, const float* b, const float* in, int rows, int cols, int act,
                  float* out) -> cs_status {
    gemv_kernel<<<(rows * 32 + 255) / 256, 256, 0, s>>>(W, b, in, rows, cols, act, out);
    CS_LAUNCHED();
    return CS_OK;
  };
  CS_TRY(gemv(w.time_w1, w.time_b1, sinus, d, w.f_dim, 1, h1));
  CS_TRY(gemv(w.time_w2, w.time_b2, h1, d, d, 0, e));
  silu_kernel<<<(d + 255) / 256, 256, 0, s>>>(e, d, se);
  CS_LAUNCHED();
  CS_TRY(gemv(w.mod_w, w.mod_b, se, 6 * d, d, 0, shared));
  CS_TRY(gemv(w.head_mod_w, w.head_mod_b, se, 2 * d, d, 0, hmod));
  block_mods_kernel<<<(w.blocks * 6 * d + 255) / 256, 256, 0, s>>>(shared, w.mod_offs, w.blocks, 6 * d, mods);
  CS_LAUNCHED();
  return CS_OK;
}

// ------------------------------------------------------------- conversion ----
// dst[r][c] (row stride ld) = bf16(src[r][c]) for c < cols, 0 for cols <= c < ld
__global__ void to_bf16_pad_kernel(const float* __restrict__ src, long long rows, int cols, int ld,
                                   __nv_bfloat16* __restrict__ dst) {
  const long long total = rows * ld;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long r = t / ld;
    const int c = (int)(t % ld);
    dst[t] = __float2bfloat16_rn(c < cols ? src[r * cols + c] : 0.f);
  }
}

cs_status to_bf16_pad(const float* src, long long rows, int cols, int ld, __nv_bfloat16* dst, cudaStream_t s) {
  const long long total = rows * ld;
  const int blocks = (int)((total + 255) / 256 < 65535 * 16 ? (total + 255) / 256 : 65535 * 16);
  to_bf16_pad_kernel<<<blocks, 256, 0, s>>>(src, rows, cols, ld, dst);
  CS_LAUNCHED();
  return CS_OK;
}

}  // namespace cs

extern "C" cs_status cs_layernorm_modulate(const float* x, const float* shift, const float* scale, void* out, int M,
                                           int d, cudaStream_t stream) {
  CS_REQUIRE(x && out, "cs_layernorm_modulate: null pointer");
  return cs::layernorm_modulate(x, shift, scale, static_cast<__nv_bfloat16*>(out), M, d, stream);
}
