// Bandwidth-bound kernels of the cache rule, the Euler update, scoring and selection.
//
//  decide   Sec. 3.1 Eq. indicator: per-candidate ||x - x_ref||^2 and ||x_ref||^2 as
//           fixed-order partial sums (128-bit loads, warp-shuffle trees), then one
//           block turns them into a += drift, the skip decision and the compaction list.
//  apply    Eq. delta / Eq. skip fused with Eq. euler (and, optionally, the x0-estimate
//           score) in one pass over the candidate's latent.
//  carry    the form cs_search_step runs: every update also leaves the next step's two
//           drift sums (the values are in its registers), so a step decides from them
//           without reading x or x_ref, and the skipped candidates' update (fed by TMA
//           bulk copies) is the one pass over their state.
//  score    -||x - y*||_2 (the verifier stand-in of Algorithm 1).
//  topk     rank-by-counting selection, deterministic tie-break.
//  refill   beam refill (state copy of survivors + seeded perturbation of children).
//
// Every reduction's order depends only on D (never on N or on which candidates are
// present), so a candidate's numbers are the same whatever batch it is in.
#include <cmath>
#include <cstdint>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "elementwise.h"
#include "ptx.cuh"

namespace cs {

constexpr int kCacheThreads = 256;
constexpr int kCacheWarps = kCacheThreads / 32;
constexpr long long kChunkElems = 8192;    // elements of one candidate per CTA (multiple of 4*256)

__host__ __device__ inline int cache_chunks(long long D) {
  long long c = (D + kChunkElems - 1) / kChunkElems;
  return (int)(c < 1 ? 1 : c);
}

// Block-wide sum of two values in a fixed order (warp shuffle tree, then warp 0).
template <int NV>
__device__ __forceinline__ void block_sum(float (&v)[NV], float (*red)[32]) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int q = 0; q < NV; ++q) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v[q] += __shfl_xor_sync(0xffffffffu, v[q], o);
  }
  if (lane == 0) {
#pragma unroll
    for (int q = 0; q < NV; ++q) red[q][warp] = v[q];
  }
  block_sync();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
#pragma unroll
    for (int q = 0; q < NV; ++q) {
      float s = lane < nw ? red[q][lane] : 0.f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      v[q] = s;
    }
  }
}

// 256-bit global loads with an L2 eviction-priority hint: data read again soon (x, re-read
// by the update after the decision) is kept, data used once is dropped first.
struct F8 {
  float v[8];
};
#define CS_LD8(QUAL)                                                                                      \
  asm volatile("ld.global.L1::no_allocate.L2::" QUAL ".v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];" \
               : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]),      \
                 "=r"(u[7])                                                                               \
               : "l"(p))
__device__ __forceinline__ F8 ld8_keep(const float* p) {
  uint32_t u[8];
  CS_LD8("evict_last");
  F8 r;
#pragma unroll
  for (int j = 0; j < 8; ++j) r.v[j] = __uint_as_float(u[j]);
  return r;
}
__device__ __forceinline__ F8 ld8_once(const float* p) {
  uint32_t u[8];
  CS_LD8("evict_first");
  F8 r;
#pragma unroll
  for (int j = 0; j < 8; ++j) r.v[j] = __uint_as_float(u[j]);
  return r;
}
#undef CS_LD8

__host__ __device__ __forceinline__ bool window_forced(int k, int T, int K_w, int K_c) {
  return k <= K_w || k > T - K_c;
}

// ------------------------------------------------------------------ decide ----
__global__ void __launch_bounds__(kCacheThreads) drift_partials_kernel(
    const float* __restrict__ x, const float* __restrict__ xr, const uint8_t* __restrict__ has_ref, long long D,
    int window_forced_step, int x_rows, float* __restrict__ partials) {
  const int i = blockIdx.y, c = blockIdx.x, nch = gridDim.x;
  __shared__ float red[2][32];
  if (window_forced_step || !has_ref[i]) return;   // forced step: no drift is evaluated
  const long long lo = (long long)c * kChunkElems;
  const long long hi = min(D, lo + kChunkElems);
  const float* xi = x + (long long)(i % x_rows) * D;   // cache state i reads latent row i % x_rows
  const float* ri = xr + (long long)i * D;
  float v[2] = {0.f, 0.f};
  const bool vec = ((D & 7) == 0) && ((reinterpret_cast<uintptr_t>(x) & 31) == 0) &&
                   ((reinterpret_cast<uintptr_t>(xr) & 31) == 0);
  if (vec) {
    const int n8 = (int)((hi - lo) >> 3);
#pragma unroll 4
    for (int e = threadIdx.x; e < n8; e += kCacheThreads) {
      const F8 a = ld8_keep(xi + lo + 8 * e), b = ld8_once(ri + lo + 8 * e);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float dd = a.v[j] - b.v[j];
        v[0] += dd * dd;
        v[1] += b.v[j] * b.v[j];
      }
    }
  } else {
    for (long long e = lo + threadIdx.x; e < hi; e += kCacheThreads) {
      const float a = xi[e], b = ri[e];
      v[0] += (a - b) * (a - b);
      v[1] += b * b;
    }
  }
  block_sum<2>(v, red);
  if (threadIdx.x == 0) {
    partials[((long long)i * nch + c) * 2 + 0] = v[0];
    partials[((long long)i * nch + c) * 2 + 1] = v[1];
  }
}

// Fixed-order sum of one candidate's chunk partials by one warp: lane l takes chunks
// l, l+32, ... in order, then a fixed shuffle tree (the order depends only on nch).
__device__ __forceinline__ double warp_sum_partials(const float* __restrict__ p, int nch, int stride, int lane) {
  double s = 0.0;
  for (int c = lane; c < nch; c += 32) s += (double)p[(long long)c * stride];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  return s;
}

// The drift's sums in the same order, in fp32: fp64 arithmetic on GB300 runs at a small
// fraction of the fp32 rate, and its latency (~5 us per decision, measured) sat on the
// critical path of the fused step.  256 chunk partials summed in fp32 add a relative
// error of order 1e-6, far inside the 1e-3 near-tie zone of the decision.
__device__ __forceinline__ float warp_sum_partials_f32(const float* __restrict__ p, int nch, int stride, int lane) {
  float s = 0.f;
  for (int c = lane; c < nch; c += 32) s += p[(long long)c * stride];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  return s;
}

// Relative drift of Eq. indicator from the two sums.
__device__ __forceinline__ float drift_of(float num, float den) { return sqrtf(num) / sqrtf(den); }

// One warp per candidate: drift from the partials, accumulate, decide; then thread 0
// writes the ordered compaction list.
__global__ void decide_finalize_kernel(const float* __restrict__ partials, int nch, float* __restrict__ accum,
                                       uint8_t* __restrict__ has_ref, int N, int window_forced_step, float tau,
                                       const uint8_t* __restrict__ force, uint8_t* __restrict__ skip_mask,
                                       int32_t* __restrict__ idx, int32_t* __restrict__ n_compute, int* err,
                                       int32_t* __restrict__ sidx = nullptr) {
  extern __shared__ uint8_t flags[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int i = warp; i < N; i += nw) {
    const bool had = has_ref[i] != 0;
    const bool free_step = !window_forced_step && had;
    float num = 0.f, den = 0.f;
    if (free_step) {
      num = warp_sum_partials_f32(partials + (long long)i * nch * 2 + 0, nch, 2, lane);
      den = warp_sum_partials_f32(partials + (long long)i * nch * 2 + 1, nch, 2, lane);
    }
    if (lane == 0) {
      bool compute;
      float a = accum[i];
      if (!free_step) {
        compute = true;
      } else {
        const float drift = drift_of(num, den);
        if (!isfinite(drift)) {
          record_error(err, CS_ERR_NONFINITE);
          compute = true;
        } else {
          a = a + drift;
          compute = (tau <= 0.f) || (a > tau);
        }
      }
      if (force) {
        const bool f = force[i] != 0;
        if (!f && !had) {
          record_error(err, CS_ERR_ARG);
        } else {
          compute = f;
        }
      }
      if (compute) {
        a = 0.f;
        has_ref[i] = 1;
      }
      accum[i] = a;
      skip_mask[i] = compute ? 0 : 1;
      flags[i] = compute ? 1 : 0;
    }
  }
  block_sync();
  if (threadIdx.x == 0) {
    int n = 0, ns = 0;
    for (int i = 0; i < N; ++i) {
      if (flags[i]) idx[n++] = i;
      else if (sidx) sidx[ns++] = i;
    }
    *n_compute = n;
    if (sidx) sidx[N] = ns;   // optional list of skipped candidates, its count after it
  }
}

// ------------------------------------------------------------------- apply ----
template <bool kScore>
__global__ void __launch_bounds__(kCacheThreads) apply_kernel(float* __restrict__ x, float* __restrict__ xr,
                                                              float* __restrict__ delta,
                                                              const float* __restrict__ v,
                                                              const uint8_t* __restrict__ skip, long long D,
                                                              float h, float t_next,
                                                              const float* __restrict__ target,
                                                              float* __restrict__ partials) {
  const int i = blockIdx.y, c = blockIdx.x, nch = gridDim.x;
  __shared__ float red[1][32];
  const long long lo = (long long)c * kChunkElems;
  const long long hi = min(D, lo + kChunkElems);
  const long long base = (long long)i * D;
  const bool skipped = skip[i] != 0;
  float acc[1] = {0.f};
  const bool vec = ((D & 3) == 0) && ((reinterpret_cast<uintptr_t>(x) & 15) == 0) &&
                   ((reinterpret_cast<uintptr_t>(xr) & 15) == 0) &&
                   ((reinterpret_cast<uintptr_t>(delta) & 15) == 0) &&
                   ((reinterpret_cast<uintptr_t>(v) & 15) == 0) &&
                   (!kScore || (reinterpret_cast<uintptr_t>(target) & 15) == 0);
  if (vec) {
    float4* x4 = reinterpret_cast<float4*>(x + base + lo);
    float4* r4 = reinterpret_cast<float4*>(xr + base + lo);
    float4* d4 = reinterpret_cast<float4*>(delta + base + lo);
    const float4* v4 = reinterpret_cast<const float4*>(v + base + lo);
    const float4* y4 = reinterpret_cast<const float4*>(target + lo);
    const int n4 = (int)((hi - lo) >> 2);
#pragma unroll 4
    for (int e = threadIdx.x; e < n4; e += kCacheThreads) {
      const float4 xv = __ldcs(x4 + e);
      float4 vu, xn;
      if (skipped) {   // Eq. skip: v_hat = x + Delta
        const float4 dv = __ldcs(d4 + e);
        vu = make_float4(xv.x + dv.x, xv.y + dv.y, xv.z + dv.z, xv.w + dv.w);
      } else {         // Eq. delta: Delta = v - x, x_ref = x
        vu = __ldcs(v4 + e);
        __stcs(d4 + e, make_float4(vu.x - xv.x, vu.y - xv.y, vu.z - xv.z, vu.w - xv.w));
        __stcs(r4 + e, xv);
      }
      xn = make_float4(xv.x + h * vu.x, xv.y + h * vu.y, xv.z + h * vu.z, xv.w + h * vu.w);   // Eq. euler
      __stcs(x4 + e, xn);
      if (kScore) {
        const float4 y = __ldg(y4 + e);
        const float e0 = xn.x - t_next * vu.x - y.x, e1 = xn.y - t_next * vu.y - y.y;
        const float e2 = xn.z - t_next * vu.z - y.z, e3 = xn.w - t_next * vu.w - y.w;
        acc[0] += e0 * e0 + e1 * e1 + e2 * e2 + e3 * e3;
      }
    }
  } else {
    for (long long e = lo + threadIdx.x; e < hi; e += kCacheThreads) {
      const float xv = x[base + e];
      float vu;
      if (skipped) {
        vu = xv + delta[base + e];
      } else {
        vu = v[base + e];
        delta[base + e] = vu - xv;
        xr[base + e] = xv;
      }
      const float xn = xv + h * vu;
      x[base + e] = xn;
      if (kScore) {
        const float d0 = xn - t_next * vu - target[e];
        acc[0] += d0 * d0;
      }
    }
  }
  if (kScore) {
    block_sum<1>(acc, red);
    if (threadIdx.x == 0) partials[(long long)i * nch + c] = acc[0];
  }
}

// Guided update (Eq. cfg with per-branch cache state): state rows i (conditional) and
// N + i (unconditional) belong to latent row i; each branch's velocity is its DiT output
// (computed: Delta_b = v_b - x, x_ref_b = x) or x + Delta_b (skipped); the Euler step uses
// v_u + w (v_c - v_u).
template <bool kScore>
__global__ void __launch_bounds__(kCacheThreads) apply_cfg_kernel(
    float* __restrict__ x, float* __restrict__ xr, float* __restrict__ delta, const float* __restrict__ v,
    const uint8_t* __restrict__ skip, int N, long long D, float h, float t_next, float w,
    const float* __restrict__ target, float* __restrict__ partials) {
  const int i = blockIdx.y, c = blockIdx.x, nch = gridDim.x;
  __shared__ float red[1][32];
  const long long lo = (long long)c * kChunkElems;
  const long long hi = min(D, lo + kChunkElems);
  const long long xo = (long long)i * D, co = (long long)i * D, uo = (long long)(N + i) * D;
  const bool sk_c = skip[i] != 0, sk_u = skip[N + i] != 0;
  float acc[1] = {0.f};
  for (long long e = lo + threadIdx.x; e < hi; e += kCacheThreads) {
    const float xv = x[xo + e];
    float vc, vu;
    if (sk_c) {
      vc = xv + delta[co + e];
    } else {
      vc = v[co + e];
      delta[co + e] = vc - xv;
      xr[co + e] = xv;
    }
    if (sk_u) {
      vu = xv + delta[uo + e];
    } else {
      vu = v[uo + e];
      delta[uo + e] = vu - xv;
      xr[uo + e] = xv;
    }
    const float vg = vu + w * (vc - vu);
    const float xn = xv + h * vg;
    x[xo + e] = xn;
    if (kScore) {
      const float d0 = xn - t_next * vg - target[e];
      acc[0] += d0 * d0;
    }
  }
  if (kScore) {
    block_sum<1>(acc, red);
    if (threadIdx.x == 0) partials[(long long)i * nch + c] = acc[0];
  }
}

// ------------------------------------------------------------------- score ----
__global__ void __launch_bounds__(kCacheThreads) sqdist_partials_kernel(const float* __restrict__ x,
                                                                        const float* __restrict__ y, long long D,
                                                                        float* __restrict__ partials) {
  const int i = blockIdx.y, c = blockIdx.x, nch = gridDim.x;
  __shared__ float red[1][32];
  const long long lo = (long long)c * kChunkElems;
  const long long hi = min(D, lo + kChunkElems);
  const float* xi = x + (long long)i * D;
  float acc[1] = {0.f};
  const bool vec = ((D & 3) == 0) && ((reinterpret_cast<uintptr_t>(x) & 15) == 0) &&
                   ((reinterpret_cast<uintptr_t>(y) & 15) == 0);
  if (vec) {
    const float4* x4 = reinterpret_cast<const float4*>(xi + lo);
    const float4* y4 = reinterpret_cast<const float4*>(y + lo);
    const int n4 = (int)((hi - lo) >> 2);
    for (int e = threadIdx.x; e < n4; e += kCacheThreads) {
      const float4 a = __ldcs(x4 + e), b = __ldg(y4 + e);
      const float d0 = a.x - b.x, d1 = a.y - b.y, d2 = a.z - b.z, d3 = a.w - b.w;
      acc[0] += d0 * d0 + d1 * d1 + d2 * d2 + d3 * d3;
    }
  } else {
    for (long long e = lo + threadIdx.x; e < hi; e += kCacheThreads) {
      const float d0 = xi[e] - y[e];
      acc[0] += d0 * d0;
    }
  }
  block_sum<1>(acc, red);
  if (threadIdx.x == 0) partials[(long long)i * nch + c] = acc[0];
}

__global__ void score_finalize_kernel(const float* __restrict__ partials, int nch, int N,
                                      float* __restrict__ scores) {
  const int lane = threadIdx.x & 31;
  const int w0 = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, nw = (gridDim.x * blockDim.x) >> 5;
  for (int i = w0; i < N; i += nw) {
    const double s = warp_sum_partials(partials + (long long)i * nch, nch, 1, lane);
    if (lane == 0) scores[i] = (float)(-sqrt(s));
  }
}

// ------------------------------------------------- single-pass decide + skip ----
// Used by cs_search_step.  Two launches, no grid-wide barrier:
//  drift_decide  every CTA takes a contiguous range of (candidate, chunk) items and
//                writes their drift partials (x read with an L2 evict-last hint, so the
//                skip update finds it in L2), then counts itself in on one arrival
//                counter.  The CTA that arrives last takes every decision (one warp per
//                candidate, the same fixed-order sum of the same partials as the two-pass
//                form, so the same bits), writes the lists of computing and skipped
//                candidates and leaves the counter at zero.
//  skip_update   launched with programmatic stream serialisation: its CTAs are
//                scheduled while the first kernel drains and wait (griddepcontrol.wait)
//                for its completion, then spread the skipped candidates' chunks over
//                the grid and apply Eq. skip + Eq. euler.
// No CTA ever waits for another CTA, so neither kernel needs co-resident CTAs.

__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait_primary() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// The decision of one candidate from its chunk partials (one warp; lane 0 writes the
// state, the skip mask and dec[i] = 1 when it computes).  Identical arithmetic to
// decide_finalize_kernel.
__device__ __forceinline__ void decide_one(int i, const float* __restrict__ partials, int nch, bool free_step,
                                           float a_before, bool had, float tau, const uint8_t* __restrict__ force,
                                           float* __restrict__ accum, uint8_t* __restrict__ has_ref,
                                           uint8_t* __restrict__ skip_mask, uint8_t* __restrict__ dec, int* err,
                                           int lane) {
  float num = 0.f, den = 0.f;
  if (free_step) {
    // partials written by other CTAs: read through L2 (never from this SM's L1).  Lane l
    // adds chunks l, l + 32, ... in order, as warp_sum_partials_f32 does (adding the 0 of
    // a missing chunk changes nothing), but with every load issued before the first add.
    const float2* pp = reinterpret_cast<const float2*>(partials) + (long long)i * nch;
    float s0 = 0.f, s1 = 0.f;
    if (nch <= 32 * 16) {
      float2 v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) v[u] = lane + 32 * u < nch ? __ldcg(pp + lane + 32 * u) : make_float2(0.f, 0.f);
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        s0 += v[u].x;
        s1 += v[u].y;
      }
    } else {
      for (int c = lane; c < nch; c += 32) {
        const float2 v = __ldcg(pp + c);
        s0 += v.x;
        s1 += v.y;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      s0 += __shfl_xor_sync(0xffffffffu, s0, o);
      s1 += __shfl_xor_sync(0xffffffffu, s1, o);
    }
    num = s0;
    den = s1;
  }
  if (lane == 0) {
    bool compute = true;
    float a = a_before;
    if (free_step) {
      const float drift = drift_of(num, den);
      if (!isfinite(drift)) {
        record_error(err, CS_ERR_NONFINITE);
      } else {
        a = a + drift;
        compute = (tau <= 0.f) || (a > tau);
      }
    }
    if (force) {
      const bool f = force[i] != 0;
      if (!f && !had) {
        record_error(err, CS_ERR_ARG);
      } else {
        compute = f;
      }
    }
    accum[i] = compute ? 0.f : a;
    skip_mask[i] = compute ? 0 : 1;
    if (compute) has_ref[i] = 1;
    dec[i] = compute ? 1 : 0;
  }
}

__global__ void __launch_bounds__(kCacheThreads) drift_decide_kernel(
    const float* __restrict__ x, const float* __restrict__ xr, float* __restrict__ accum,
    uint8_t* __restrict__ has_ref, int N, long long D, int nch, float tau, const uint8_t* __restrict__ force,
    uint8_t* __restrict__ skip_mask, int32_t* __restrict__ idx, int32_t* __restrict__ n_compute,
    int32_t* __restrict__ sidx, float* __restrict__ partials, unsigned* __restrict__ counter, int* err) {
  __shared__ float red[2][32];
  __shared__ int s_last;
  extern __shared__ uint8_t flags[];            // [N] decisions (1 = compute), in the deciding CTA
  pdl_launch_dependents();   // the skip-update grid may be scheduled as soon as every CTA runs
  const int items = N * nch;
  const int per = (items + gridDim.x - 1) / gridDim.x;
  const int active = (items + per - 1) / per;   // CTAs that own items (the others return)
  const int it0 = blockIdx.x * per, it1 = min(items, it0 + per);
  if (it0 >= it1) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = kCacheThreads / 32;
  for (int item = it0; item < it1; ++item) {
    const int i = item / nch, c = item % nch;
    // has_ref is rewritten only by the deciding CTA, after every CTA has arrived
    if (!has_ref[i]) continue;                  // uniform over the CTA
    const long long clo = (long long)c * kChunkElems, chi = min(D, clo + kChunkElems);
    const float* xi = x + (long long)i * D + clo;
    const float* ri = xr + (long long)i * D + clo;
    const int n8 = (int)((chi - clo) >> 3);
    float v[2] = {0.f, 0.f};
    if (n8 == 4 * kCacheThreads) {
      // a full chunk: all eight 32-byte loads of the thread issued before the first use
      // (the compiler left only part of them in flight, which cost ~4 us at N = 4)
      F8 a[4], b[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        a[u] = ld8_keep(xi + 8 * (threadIdx.x + u * kCacheThreads));
        b[u] = ld8_once(ri + 8 * (threadIdx.x + u * kCacheThreads));
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float dd = a[u].v[j] - b[u].v[j];
          v[0] += dd * dd;
          v[1] += b[u].v[j] * b[u].v[j];
        }
    } else {
      for (int e = threadIdx.x; e < n8; e += kCacheThreads) {
        const F8 a = ld8_keep(xi + 8 * e), b = ld8_once(ri + 8 * e);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float dd = a.v[j] - b.v[j];
          v[0] += dd * dd;
          v[1] += b.v[j] * b.v[j];
        }
      }
    }
    block_sum<2>(v, red);
    if (threadIdx.x == 0) {
      partials[((long long)i * nch + c) * 2 + 0] = v[0];
      partials[((long long)i * nch + c) * 2 + 1] = v[1];
    }
    block_sync();
  }
  // arrival: the CTA that arrives last takes every decision
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(counter, 1u) == (unsigned)(active - 1);
  }
  block_sync();
  if (!s_last) return;
  __threadfence();
  for (int i = warp; i < N; i += nw) {
    const bool had = has_ref[i] != 0;
    decide_one(i, partials, nch, had, accum[i], had, tau, force, accum, has_ref, skip_mask, flags, err, lane);
  }
  block_sync();
  // compaction lists (computing candidates in idx, skipped ones in sidx, count after them)
  if (warp == 0) {
    int nc = 0, ns = 0;
    for (int base = 0; base < N; base += 32) {
      const int k = base + lane;
      const bool valid = k < N;
      const bool comp = valid && flags[k];
      const unsigned bc = __ballot_sync(0xffffffffu, comp), bs = __ballot_sync(0xffffffffu, valid && !comp);
      const unsigned below = (1u << lane) - 1u;
      if (comp) idx[nc + __popc(bc & below)] = k;
      if (valid && !comp) sidx[ns + __popc(bs & below)] = k;
      nc += __popc(bc);
      ns += __popc(bs);
    }
    if (lane == 0) {
      *n_compute = nc;
      sidx[N] = ns;
      *counter = 0u;                            // ready for the next call
    }
  }
}

// Skipped candidates: x += h (x + Delta).  The (skipped candidate, chunk) items, taken
// from the list the deciding CTA wrote (sidx[0..n), n = sidx[N]), are spread evenly over
// the grid, the last ones first (the latents the drift pass read last are the likeliest
// to be still in L2).
template <bool kScore>
__global__ void __launch_bounds__(kCacheThreads, 4) skip_update_kernel(
    float* __restrict__ x, const float* __restrict__ delta, const int32_t* sidx, int N, long long D,
    int nch, float h, float t_next, const float* __restrict__ target, float* __restrict__ spart) {
  __shared__ float red[1][32];
  // the decisions (and every write of the first kernel) are visible after the wait; the
  // list is read through L2 (a read-only cached load could be placed before the wait)
  pdl_wait_primary();
  const int items = __ldcg(sidx + N) * nch;
  const int per = (items + gridDim.x - 1) / gridDim.x;
  const int it1 = items - blockIdx.x * per, it0 = max(0, it1 - per);
  for (int item = it1 - 1; item >= it0; --item) {
    const int i = __ldcg(sidx + item / nch), c = item % nch;
    const long long lo = (long long)c * kChunkElems, hi = min(D, lo + kChunkElems);
    float* xi = x + (long long)i * D + lo;
    const float* di = delta + (long long)i * D + lo;
    const float* yi = kScore ? target + lo : nullptr;
    const int n8 = (int)((hi - lo) >> 3);
    float acc[1] = {0.f};
    if (!kScore && n8 == 4 * kCacheThreads) {   // a full chunk: all eight 32-byte loads in flight
      F8 xa[4], da[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        xa[u] = ld8_once(xi + 8 * (threadIdx.x + u * kCacheThreads));
        da[u] = ld8_once(di + 8 * (threadIdx.x + u * kCacheThreads));
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        float xn[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) xn[j] = xa[u].v[j] + h * (xa[u].v[j] + da[u].v[j]);   // Eq. skip + Eq. euler
        float4* o4 = reinterpret_cast<float4*>(xi + 8 * (threadIdx.x + u * kCacheThreads));
        __stcs(o4, make_float4(xn[0], xn[1], xn[2], xn[3]));
        __stcs(o4 + 1, make_float4(xn[4], xn[5], xn[6], xn[7]));
      }
      continue;
    }
#pragma unroll 4
    for (int e = threadIdx.x; e < n8; e += kCacheThreads) {   // a chunk's four rounds of loads all in flight
      const F8 xv = ld8_once(xi + 8 * e), dv = ld8_once(di + 8 * e);
      float xn[8], vu[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        vu[j] = xv.v[j] + dv.v[j];              // Eq. skip
        xn[j] = xv.v[j] + h * vu[j];            // Eq. euler
      }
      float4* o4 = reinterpret_cast<float4*>(xi + 8 * e);
      __stcs(o4, make_float4(xn[0], xn[1], xn[2], xn[3]));
      __stcs(o4 + 1, make_float4(xn[4], xn[5], xn[6], xn[7]));
      if (kScore) {
        const F8 y = ld8_once(yi + 8 * e);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float d0 = xn[j] - t_next * vu[j] - y.v[j];
          acc[0] += d0 * d0;
        }
      }
    }
    if (kScore) {
      block_sum<1>(acc, red);
      if (threadIdx.x == 0) spart[(long long)i * nch + c] = acc[0];
      block_sync();
    }
  }
}

// ---------------------------------------------------------- carried drift ----
// The drift of Eq. indicator at step k needs ||x - x_ref|| and ||x_ref|| of the latent a
// candidate holds at step k.  That latent is written by the update of step k - 1, which
// has x_next and the x_ref it leaves in registers at that moment, so the update kernels
// also leave the two squared norms, per candidate, for the next step: the drift is
// carried.  A step whose cached candidates all carry one takes its decisions without
// reading x or x_ref, and its skip update is the one pass over a skipped candidate's
// state: read x, Delta and x_ref, write x, and leave the sums for step k + 1.
// has_ref = 3 (bit 1 set) marks a candidate whose carried sums belong to its current x
// and x_ref; every other writer of the state leaves has_ref = 1.
//
// The partial pairs of a candidate (one per 4096-element unit of a skipped candidate, one
// per token row of a computed one) are summed once every pair is stored, in a fixed order
// that does not depend on which CTA sums them, so the carried value depends on the
// candidate alone.
struct CarryOut {
  float2* part;        // [cap][P] partial pairs of the candidate's units or token rows
  int P;
  float2* drift_out;   // [cap] (sum (x_next - x_ref)^2, sum x_ref^2) for the next step
};

__device__ __forceinline__ void carry_finalize(const CarryOut& c, int i, int n, float (*red)[32]) {
  __threadfence();
  float v[2] = {0.f, 0.f};
  const float2* p = c.part + (long long)i * c.P;
  for (int q = threadIdx.x; q < n; q += kCacheThreads) {
    const float2 a = __ldcg(p + q);
    v[0] += a.x;
    v[1] += a.y;
  }
  block_sum<2>(v, red);
  if (threadIdx.x == 0) c.drift_out[i] = make_float2(v[0], v[1]);
  block_sync();
}

// Decision flags of the carried form (per candidate, in shared memory).
constexpr uint8_t kFlCompute = 1, kFlNonFinite = 2, kFlArg = 4, kFlBad = 8;

// The decision of candidate i from the drift carried into this step (Sec. 3.1): free step
// with a cached reference: a += drift, compute iff tau <= 0 or a > tau; inside the window
// or with an empty cache: compute, no drift; then the forced mask.  kFlBad: a cached
// candidate without a carried drift on a free step.  Every caller gets the same bits.
__device__ __forceinline__ uint8_t decide_carried(int i, int wf, float tau, const uint8_t* __restrict__ has_ref,
                                                  const float* __restrict__ accum, const float2* __restrict__ drift_in,
                                                  const uint8_t* __restrict__ force, float& a) {
  // every input loaded before the first use (one round trip, not one per branch)
  const uint8_t hr = has_ref[i];
  const float a0 = accum[i];
  const float2 s2 = drift_in[i];
  const uint8_t fi = force ? force[i] : 0;
  const bool had = hr != 0;
  bool compute = true;
  uint8_t fl = 0;
  a = a0;
  if (!wf && had) {
    if (!(hr & 2)) {
      fl |= kFlBad;
    } else {
      const float drift = drift_of(s2.x, s2.y);
      if (!isfinite(drift)) {
        fl |= kFlNonFinite;
      } else {
        a = a + drift;
        compute = (tau <= 0.f) || (a > tau);
      }
    }
  }
  if (force) {
    const bool f = fi != 0;
    if (!f && !had) fl |= kFlArg;
    else compute = f;
  }
  if (compute) a = 0.f;
  return fl | (compute ? kFlCompute : 0);
}

// TMA ring of the skip update: a unit is 4096 elements of one candidate; one stage holds a
// unit of x, Delta and x_ref (48 KB); four stages keep 192 KB per SM in flight whatever
// the registers of the consuming threads.
constexpr int kUnitElems = 4096;
constexpr int kSkipStages = 4;
constexpr int kSkipStageFloats = 3 * kUnitElems;
constexpr size_t kSkipRingBytes = (size_t)kSkipStages * kSkipStageFloats * sizeof(float);
constexpr int kSkipThreads = kCacheThreads + 32;   // eight consumer warps and one producer warp
constexpr int kClaim = 2;                          // units a producer claims at a time

__host__ __device__ inline int carry_units(long long D) {
  long long u = (D + kUnitElems - 1) / kUnitElems;
  return (int)(u < 1 ? 1 : u);
}

__host__ inline size_t carry_skip_smem(int N) {
  return kSkipRingBytes + (size_t)(3 * N + 15) / 16 * 16;   // + skipped list (16-bit) and flags
}

// Fixed-order sum of a candidate's n partial pairs by one warp (lane l adds l, l + 32, ...,
// then the shuffle tree): the carried value does not depend on which CTA sums it.
__device__ __forceinline__ void carry_finalize_warp(const CarryOut& c, int i, int n, int lane) {
  __threadfence();
  const float2* pp = c.part + (long long)i * c.P;
  float s0 = 0.f, s1 = 0.f;
  constexpr int kU = 16;                 // loads in flight per lane before the adds
  for (int base = 0; base < n; base += 32 * kU) {
    float2 v[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int q = base + lane + 32 * u;
      v[u] = q < n ? __ldcg(pp + q) : make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {       // the same order as one pair at a time (adding 0 changes nothing)
      s0 += v[u].x;
      s1 += v[u].y;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s0 += __shfl_xor_sync(0xffffffffu, s0, o);
    s1 += __shfl_xor_sync(0xffffffffu, s1, o);
  }
  if (lane == 0) c.drift_out[i] = make_float2(s0, s1);
}

// The skip update of cs_search_step with the carried drift, one CTA per SM, warp
// specialised.  Per skipped candidate and unit: x_next = x + h (x + Delta) (Eq. skip +
// Eq. euler), written back, and the unit's partial pair of the next step's drift,
// (x_next - x_ref)^2 and x_ref^2 (thread sums over the unit's float4s, warp trees, then
// the eight warps in order); with a target, the unit's score partial.
//  producer warp  claims units from a counter shared by the grid (a full ring at kernel
//                 start, while the decisions are taken, then two at a time, one claim
//                 ahead), so that CTAs that are served faster take more units;
//                 keeps the four-stage ring full (cp.async.bulk of x, Delta and x_ref, one
//                 mbarrier per stage, a sentinel when the units run out); when the
//                 consumers release a stage it adds the unit's eight warp pairs in order
//                 and stores them.
//  consumer warps wait for a stage, update the unit, leave their warp sums and release it.
// Every wait is bounded.  Every CTA counts itself in on one arrival counter; the CTA that
// arrives last (every unit pair is stored by then) resets it and the claim counter, and
// its warps sum each skipped candidate's unit pairs in order into carry.drift_out:
//  kDecide  every CTA takes the same decisions from the same inputs (decide_carried) and
//           so knows the skipped list; the CTA that arrives last (after every CTA has read
//           the state) also writes accum, has_ref (3 for skipped candidates), the skip
//           mask and the list of computing candidates.  A free step on
//           which a cached candidate carries no drift changes nothing and reports
//           *n_compute = -1: the caller then runs the drift pass.
//  !kDecide the decisions and the skipped list come from drift_decide_kernel (launched
//           before this one with programmatic stream serialisation); the last CTA sets the
//           skipped candidates' has_ref to 3.
template <bool kScore, bool kDecide>
__global__ void __launch_bounds__(kSkipThreads, 1) carry_skip_kernel(
    float* __restrict__ x, const float* __restrict__ xr, const float* __restrict__ delta, float* __restrict__ accum,
    uint8_t* __restrict__ has_ref, int N, long long D, int nun, int wf, float tau, const uint8_t* __restrict__ force,
    uint8_t* __restrict__ skip_mask, int32_t* __restrict__ idx, int32_t* __restrict__ n_compute,
    const int32_t* sidx_in, const float2* __restrict__ drift_in, CarryOut carry, unsigned* __restrict__ counter,
    unsigned* __restrict__ claim, float h, float t_next, const float* __restrict__ target, float* __restrict__ spart,
    int* err) {
  constexpr int NV = kScore ? 3 : 2;
  constexpr int S = kSkipStages;
  extern __shared__ __align__(128) uint8_t smem[];
  float* ring = reinterpret_cast<float*>(smem);
  uint16_t* s_list = reinterpret_cast<uint16_t*>(smem + kSkipRingBytes);
  uint8_t* s_flag = reinterpret_cast<uint8_t*>(s_list + N);
  __shared__ uint64_t full[S], empty[S];
  __shared__ int s_item[S];
  __shared__ float red[S][NV][kCacheWarps];
  __shared__ int s_ns, s_bad, s_last, s_abort;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool producer = warp == kCacheWarps;
  // the producer's first claims (a full ring, then the next claim) go out now, so that their
  // round trips overlap the decisions; claims past the last item become sentinels
  unsigned first_claim = 0, next_claim = 0;
  if (producer && lane == 0) {
    first_claim = atomicAdd(claim, (unsigned)S);
    next_claim = atomicAdd(claim, (unsigned)kClaim);
  }
  if (threadIdx.x == 0) {
    for (int q = 0; q < S; ++q) {
      mbar_init(&full[q], 1);
      mbar_init(&empty[q], kCacheWarps);
    }
    fence_mbar_init();
    s_bad = 0;
    s_abort = 0;
  }
  block_sync();
  int ns;
  if (kDecide) {
    for (int i = threadIdx.x; i < N; i += kSkipThreads) {
      float a;
      const uint8_t fl = decide_carried(i, wf, tau, has_ref, accum, drift_in, force, a);
      s_flag[i] = fl;
      if (fl & kFlBad) s_bad = 1;
    }
    block_sync();
    if (warp == 0) {
      int n = 0;
      for (int base = 0; base < N; base += 32) {
        const int k = base + lane;
        const bool sk = k < N && !(s_flag[k] & kFlCompute);
        const unsigned b = __ballot_sync(0xffffffffu, sk);
        if (sk) s_list[n + __popc(b & ((1u << lane) - 1u))] = (uint16_t)k;
        n += __popc(b);
      }
      if (lane == 0) s_ns = s_bad ? 0 : n;
    }
    block_sync();
    ns = s_ns;
  } else {
    // the decisions (and every write of the drift pass) are visible after the wait; read
    // them through L2 (a read-only cached load could be placed before the wait)
    pdl_wait_primary();
    ns = __ldcg(sidx_in + N);
    for (int q = threadIdx.x; q < ns; q += kSkipThreads) {
      const int i = __ldcg(sidx_in + q);
      s_list[q] = (uint16_t)(index_ok(i, N, err) ? i : 0);   // checked in CS_DEBUG_CHECKS builds
    }
    block_sync();
  }
  const int items = ns * nun;
  volatile int* abort = &s_abort;
  if (producer) {
    // ---- producer warp: lane 0 claims and issues, the whole warp finalizes candidates
    int cur = (int)first_claim, left = S, n_real = 0;
    bool exhausted = false;
    auto fill = [&](int j) {                       // lane 0: use j of stage j % S
      const int st = j % S;
      if (left == 0) {
        cur = (int)next_claim;
        left = kClaim;
        next_claim = atomicAdd(claim, (unsigned)kClaim);   // needed one claim later
      }
      const int it = cur;
      ++cur;
      --left;
      if (it >= items) {
        s_item[st] = -1;
        mbar_arrive(&full[st]);
        exhausted = true;
        return;
      }
      const int sq = it / nun, u = it - sq * nun, i = s_list[sq];
      const long long lo = (long long)u * kUnitElems;
      const uint32_t bytes = (uint32_t)(min((long long)kUnitElems, D - lo) * sizeof(float));
      float* dst = ring + (size_t)st * kSkipStageFloats;
      s_item[st] = it;
      mbar_arrive_expect_tx(&full[st], 3 * bytes);
      bulk_load_1d(dst, x + (long long)i * D + lo, bytes, &full[st]);
      bulk_load_1d(dst + kUnitElems, delta + (long long)i * D + lo, bytes, &full[st]);
      bulk_load_1d(dst + 2 * kUnitElems, xr + (long long)i * D + lo, bytes, &full[st]);
      ++n_real;
    };
    if (lane == 0 && items > 0)
      for (int j = 0; j < S && !exhausted; ++j) fill(j);
    n_real = __shfl_sync(0xffffffffu, n_real, 0);
    int j_released = 0;                            // uses whose copies have landed and been consumed
    for (int j = 0; j < n_real; ++j) {
      const int st = j % S;
      if (!mbar_wait(&empty[st], (uint32_t)(j / S) & 1u, abort, err)) break;   // the consumers are done with use j
      j_released = j + 1;
      if (lane == 0) {
        const int it = s_item[st], sq = it / nun, u = it - sq * nun, i = s_list[sq];
        float p[NV];
#pragma unroll
        for (int q = 0; q < NV; ++q) {
          p[q] = 0.f;
#pragma unroll
          for (int w = 0; w < kCacheWarps; ++w) p[q] += red[st][q][w];
        }
        carry.part[(long long)i * carry.P + u] = make_float2(p[0], p[1]);
        if (kScore) spart[(long long)i * nun + u] = p[NV - 1];
        if (!exhausted) fill(j + S);
      }
      n_real = __shfl_sync(0xffffffffu, n_real, 0);
    }
    if (*abort && lane == 0) {
      // a wait ran out: let the copies still outstanding (uses not yet released) land
      // before the CTA's memory goes
      for (int j = j_released; j < n_real; ++j) mbar_wait_teardown(&full[j % S], (uint32_t)(j / S) & 1u);
    }
    if (lane == 0) {
      // the claims made ahead must be performed before this CTA arrives (the last CTA to
      // arrive resets the counter): wait for their values
      if ((int)(first_claim | next_claim) < 0) record_error(err, CS_ERR_ARG);
      __threadfence();
    }
  } else if (items > 0) {
    // ---- consumer warps
    for (int j = 0;; ++j) {
      const int st = j % S;
      if (!mbar_wait(&full[st], (uint32_t)(j / S) & 1u, abort, err)) break;
      const int it = s_item[st];
      if (it < 0) break;
      const int sq = it / nun, u = it - sq * nun, i = s_list[sq];
      const float* sb = ring + (size_t)st * kSkipStageFloats;
      const float4* sx = reinterpret_cast<const float4*>(sb);
      const float4* sd = reinterpret_cast<const float4*>(sb + kUnitElems);
      const float4* sr = reinterpret_cast<const float4*>(sb + 2 * kUnitElems);
      const long long lo = (long long)u * kUnitElems;
      const int n4 = (int)(min((long long)kUnitElems, D - lo) >> 2);
      float4* xo = reinterpret_cast<float4*>(x + (long long)i * D + lo);
      const float4* y4 = kScore ? reinterpret_cast<const float4*>(target + lo) : nullptr;
      float acc[NV];
#pragma unroll
      for (int q = 0; q < NV; ++q) acc[q] = 0.f;
#pragma unroll 4
      for (int q = threadIdx.x; q < n4; q += kCacheThreads) {
        const float4 xv = sx[q], dv = sd[q], rv = sr[q];
        const float4 vu = make_float4(xv.x + dv.x, xv.y + dv.y, xv.z + dv.z, xv.w + dv.w);            // Eq. skip
        const float4 xn = make_float4(xv.x + h * vu.x, xv.y + h * vu.y, xv.z + h * vu.z, xv.w + h * vu.w);  // Eq. euler
        __stcs(xo + q, xn);
        const float d0 = xn.x - rv.x, d1 = xn.y - rv.y, d2 = xn.z - rv.z, d3 = xn.w - rv.w;
        acc[0] += d0 * d0 + d1 * d1 + d2 * d2 + d3 * d3;
        acc[1] += rv.x * rv.x + rv.y * rv.y + rv.z * rv.z + rv.w * rv.w;
        if (kScore) {
          const float4 y = __ldg(y4 + q);
          const float e0 = xn.x - t_next * vu.x - y.x, e1 = xn.y - t_next * vu.y - y.y;
          const float e2 = xn.z - t_next * vu.z - y.z, e3 = xn.w - t_next * vu.w - y.w;
          acc[2] += e0 * e0 + e1 * e1 + e2 * e2 + e3 * e3;
        }
      }
#pragma unroll
      for (int q = 0; q < NV; ++q) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[q] += __shfl_xor_sync(0xffffffffu, acc[q], o);
      }
      if (lane == 0) {
#pragma unroll
        for (int q = 0; q < NV; ++q) red[st][q][warp] = acc[q];
        mbar_arrive(&empty[st]);
      }
      __syncwarp();
    }
  }
  block_sync();
  // arrival: the CTA that arrives last (every CTA has read the state and claimed its last
  // unit by then) resets both counters and, deciding, writes the state
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(counter, 1u) == gridDim.x - 1;
  }
  block_sync();
  if (!s_last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    *claim = 0u;
    *counter = 0u;
  }
  if (s_bad) {
    if (threadIdx.x == 0) *n_compute = -1;
    return;
  }
  // every unit pair is stored: one warp per skipped candidate sums them in order
  for (int q = warp; q < ns; q += kSkipThreads / 32) {
    carry_finalize_warp(carry, s_list[q], nun, lane);
    if (!kDecide && lane == 0) has_ref[s_list[q]] = 3;
  }
  if constexpr (kDecide) {   // the state writes of the deciding form
    for (int i = threadIdx.x; i < N; i += kSkipThreads) {
      float a;
      const uint8_t fl = decide_carried(i, wf, tau, has_ref, accum, drift_in, force, a);
      const bool compute = fl & kFlCompute;
      if (fl & kFlNonFinite) record_error(err, CS_ERR_NONFINITE);
      if (fl & kFlArg) record_error(err, CS_ERR_ARG);
      s_flag[i] = fl;
      accum[i] = a;
      skip_mask[i] = compute ? 0 : 1;
      has_ref[i] = compute ? 1 : 3;
    }
    block_sync();
    if (warp == 0) {
      int nc = 0;
      for (int base = 0; base < N; base += 32) {
        const int k = base + lane;
        const bool comp = k < N && (s_flag[k] & kFlCompute);
        const unsigned b = __ballot_sync(0xffffffffu, comp);
        if (comp) idx[nc + __popc(b & ((1u << lane) - 1u))] = k;
        nc += __popc(b);
      }
      if (lane == 0) *n_compute = nc;
    }
  }
}

// A step inside the warm-up or cool-down window without a forced mask: every candidate
// computes and no drift is evaluated (Sec. 3.1), so the decision needs no pass over the
// latents and no grid-wide launch.
__global__ void decide_all_compute_kernel(float* __restrict__ accum, uint8_t* __restrict__ has_ref, int N,
                                          uint8_t* __restrict__ skip_mask, int32_t* __restrict__ idx,
                                          int32_t* __restrict__ n_compute) {
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    accum[i] = 0.f;
    has_ref[i] = 1;
    skip_mask[i] = 0;
    idx[i] = i;
  }
  if (threadIdx.x == 0) *n_compute = N;
}

// The update of computed candidates only (skipped ones were updated by decide_skip).
template <bool kScore>
__global__ void __launch_bounds__(kCacheThreads) apply_computed_kernel(
    float* __restrict__ x, float* __restrict__ xr, float* __restrict__ delta, const float* __restrict__ v,
    const uint8_t* __restrict__ skip, long long D, float h, float t_next, const float* __restrict__ target,
    float* __restrict__ spart) {
  const int i = blockIdx.y, c = blockIdx.x, nch = gridDim.x;
  if (skip[i]) return;
  __shared__ float red[1][32];
  const long long lo = (long long)c * kChunkElems, hi = min(D, lo + kChunkElems);
  const long long base = (long long)i * D;
  float4* x4 = reinterpret_cast<float4*>(x + base + lo);
  float4* r4 = reinterpret_cast<float4*>(xr + base + lo);
  float4* d4 = reinterpret_cast<float4*>(delta + base + lo);
  const float4* v4 = reinterpret_cast<const float4*>(v + base + lo);
  const float4* y4 = kScore ? reinterpret_cast<const float4*>(target + lo) : nullptr;
  const int n4 = (int)((hi - lo) >> 2);
  float acc[1] = {0.f};
#pragma unroll 4
  for (int e = threadIdx.x; e < n4; e += kCacheThreads) {
    const float4 xv = __ldcs(x4 + e), vu = __ldcs(v4 + e);
    __stcs(d4 + e, make_float4(vu.x - xv.x, vu.y - xv.y, vu.z - xv.z, vu.w - xv.w));
    __stcs(r4 + e, xv);
    const float4 xn = make_float4(xv.x + h * vu.x, xv.y + h * vu.y, xv.z + h * vu.z, xv.w + h * vu.w);
    __stcs(x4 + e, xn);
    if (kScore) {
      const float4 y = __ldg(y4 + e);
      const float e0 = xn.x - t_next * vu.x - y.x, e1 = xn.y - t_next * vu.y - y.y;
      const float e2 = xn.z - t_next * vu.z - y.z, e3 = xn.w - t_next * vu.w - y.w;
      acc[0] += e0 * e0 + e1 * e1 + e2 * e2 + e3 * e3;
    }
  }
  if (kScore) {
    block_sum<1>(acc, red);
    if (threadIdx.x == 0) spart[(long long)i * nch + c] = acc[0];
  }
}

// ------------------------------------------------ computed update from tokens ----
// The update of computed candidates straight from the DiT head's token-layout output, so
// that the velocity never makes a round trip through HBM: the unpatchify scatter fused
// with Eq. delta and Eq. euler.  For candidate i = idx[j] and latent element (c, f, h, w):
//   v = hout[(j L + l) P + 4c + 2 (h & 1) + (w & 1)],  l = (f H/2 + h/2) W/2 + w/2,
//   Delta = v - x,  x_ref = x,  x += (t_next - t_cur) v,  accum = 0, has_ref = 1, skip = 0.
// One CTA per (token row (f, h/2), computed candidate): the row's W/2 tokens x P features
// (contiguous in hout) are staged in shared memory as one float4 per (w/4, c, h&1) that
// holds v at w..w+3, so hout and the four state tensors all move in 16-byte accesses; a
// thread issues all its loads of a phase before it uses the first.
// The score partial of a tile is a fixed-order block sum (independent of the batch).
// With kCarry the CTA also leaves the row's pair of the next step's drift terms
// (x_next - x_ref_new = x_next - x, and x_ref_new = x, both in registers here) for
// carry_rows_finalize_kernel, and has_ref = 3.
constexpr int kVelUnroll = 4;   // float4 loads in flight per thread and phase (rows up to 1024 of them)

template <bool kScore, bool kCarry>
__global__ void __launch_bounds__(kCacheThreads) velocity_update_kernel(
    const float* __restrict__ hout, const int32_t* __restrict__ idx, int C, int F, int H, int W,
    float* __restrict__ x, float* __restrict__ xr, float* __restrict__ delta, float* __restrict__ accum,
    uint8_t* __restrict__ has_ref, uint8_t* __restrict__ skip_mask, float h, float t_next,
    const float* __restrict__ target, float* __restrict__ tpart, CarryOut carry, long long idx_limit, int* err) {
  constexpr int NV = kCarry ? 3 : 1;              // score, then the carried pair
  extern __shared__ float4 s_v[];                 // [W/4][2C + 1]: the +1 staggers the banks
  __shared__ float red[3][32];
  if (kCarry) pdl_launch_dependents();            // the finalize may be scheduled while this drains
  const int H2 = H / 2, W2 = W / 2, W4 = W / 4, S = 2 * C + 1;
  const int row = blockIdx.x, j = blockIdx.y;     // row = f * H/2 + h/2
  const int f = row / H2, hh = row % H2;
  const int i = idx[j];
  if (!index_ok(i, idx_limit, err)) return;      // uniform over the CTA
  const long long D = (long long)C * F * H * W;
  const long long L = (long long)F * H2 * W2;
  const float4* src = reinterpret_cast<const float4*>(hout + ((long long)j * L + (long long)row * W2) * (4 * C));
  auto stage = [&](int q, float4 a) {             // features 4c..4c+3 of token T: (ph, pw) = 00 01 10 11
    const int T = q / C, c = q % C;
    float2* d = reinterpret_cast<float2*>(&s_v[(T >> 1) * S + 2 * c]) + (T & 1);
    d[0] = make_float2(a.x, a.y);                 // h even: w = 2T, 2T + 1
    d[2] = make_float2(a.z, a.w);                 // h odd
  };
  const int nq = W2 * C;
  {
    float4 a[kVelUnroll];
#pragma unroll
    for (int u = 0; u < kVelUnroll; ++u) {
      const int q = threadIdx.x + u * kCacheThreads;
      if (q < nq) a[u] = __ldcs(src + q);
    }
#pragma unroll
    for (int u = 0; u < kVelUnroll; ++u) {
      const int q = threadIdx.x + u * kCacheThreads;
      if (q < nq) stage(q, a[u]);
    }
    for (int q = threadIdx.x + kVelUnroll * kCacheThreads; q < nq; q += kCacheThreads) stage(q, __ldcs(src + q));
  }
  block_sync();
  float* xi = x + (long long)i * D;
  float* ri = xr + (long long)i * D;
  float* di = delta + (long long)i * D;
  float acc[NV];
#pragma unroll
  for (int q = 0; q < NV; ++q) acc[q] = 0.f;
  // element offset of update item q inside the candidate's latent (D < 2^31 elements)
  auto offset = [&](int q) {
    const int w4 = q % W4, cp = q / W4;           // cp = 2c + (h & 1)
    return (((cp >> 1) * F + f) * H + 2 * hh + (cp & 1)) * W + 4 * w4;
  };
  auto update = [&](int q, int e, float4 xv) {
    const float4 vu = s_v[(q % W4) * S + q / W4];
    __stcs(reinterpret_cast<float4*>(di + e), make_float4(vu.x - xv.x, vu.y - xv.y, vu.z - xv.z, vu.w - xv.w));
    __stcs(reinterpret_cast<float4*>(ri + e), xv);
    const float4 xn = make_float4(xv.x + h * vu.x, xv.y + h * vu.y, xv.z + h * vu.z, xv.w + h * vu.w);
    __stcs(reinterpret_cast<float4*>(xi + e), xn);
    if (kScore) {
      const float4 y = __ldg(reinterpret_cast<const float4*>(target + e));
      const float e0 = xn.x - t_next * vu.x - y.x, e1 = xn.y - t_next * vu.y - y.y;
      const float e2 = xn.z - t_next * vu.z - y.z, e3 = xn.w - t_next * vu.w - y.w;
      acc[0] += e0 * e0 + e1 * e1 + e2 * e2 + e3 * e3;
    }
    if (kCarry) {   // the next step's drift terms: x_next - x_ref_new (as stored), x_ref_new
      const float d0 = xn.x - xv.x, d1 = xn.y - xv.y, d2 = xn.z - xv.z, d3 = xn.w - xv.w;
      acc[NV - 2] += d0 * d0 + d1 * d1 + d2 * d2 + d3 * d3;
      acc[NV - 1] += xv.x * xv.x + xv.y * xv.y + xv.z * xv.z + xv.w * xv.w;
    }
  };
  const int nu = 2 * C * W4;
  {
    float4 xv[kVelUnroll];
#pragma unroll
    for (int u = 0; u < kVelUnroll; ++u) {
      const int q = threadIdx.x + u * kCacheThreads;
      if (q < nu) xv[u] = __ldcs(reinterpret_cast<const float4*>(xi + offset(q)));
    }
#pragma unroll
    for (int u = 0; u < kVelUnroll; ++u) {
      const int q = threadIdx.x + u * kCacheThreads;
      if (q < nu) update(q, offset(q), xv[u]);
    }
    for (int q = threadIdx.x + kVelUnroll * kCacheThreads; q < nu; q += kCacheThreads)
      update(q, offset(q), __ldcs(reinterpret_cast<const float4*>(xi + offset(q))));
  }
  if (kScore || kCarry) {
    block_sum<NV>(acc, red);
    if (threadIdx.x == 0) {
      if (kScore) tpart[(long long)i * gridDim.x + row] = acc[0];
      if (kCarry) carry.part[(long long)i * carry.P + row] = make_float2(acc[NV - 2], acc[NV - 1]);
    }
  }
  if (row == 0 && threadIdx.x == 0) {
    accum[i] = 0.f;
    has_ref[i] = kCarry ? 3 : 1;
    skip_mask[i] = 0;
  }
}

// The computed candidates' carried drift: one CTA per computed candidate sums its token
// rows' pairs (carry_finalize, fixed order).  Launched after velocity_update_kernel with
// programmatic stream serialisation: scheduled while the update drains, it waits for its
// completion before reading.
__global__ void __launch_bounds__(kCacheThreads) carry_rows_finalize_kernel(const int32_t* __restrict__ idx,
                                                                           int ntiles, CarryOut carry,
                                                                           long long idx_limit, int* err) {
  __shared__ float red[2][32];
  pdl_wait_primary();
  const int i = idx[blockIdx.x];
  if (!index_ok(i, idx_limit, err)) return;      // uniform over the CTA
  carry_finalize(carry, i, ntiles, red);
}

// Scores when the two kinds of candidates left their partials in different groupings:
// skipped candidates per 8192-element chunk (nch), computed ones per token row (ntiles).
__global__ void score_finalize_split_kernel(const float* __restrict__ spart, int nch, const float* __restrict__ tpart,
                                            int ntiles, const uint8_t* __restrict__ skip_mask, int N,
                                            float* __restrict__ scores) {
  const int lane = threadIdx.x & 31;
  const int w0 = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, nw = (gridDim.x * blockDim.x) >> 5;
  for (int i = w0; i < N; i += nw) {
    const bool sk = skip_mask[i] != 0;
    const double s = sk ? warp_sum_partials(spart + (long long)i * nch, nch, 1, lane)
                        : warp_sum_partials(tpart + (long long)i * ntiles, ntiles, 1, lane);
    if (lane == 0) scores[i] = (float)(-sqrt(s));
  }
}

// -------------------------------------------------------------------- top-k ----
__global__ void topk_kernel(const float* __restrict__ scores, int N, int k, int32_t* __restrict__ idx) {
  extern __shared__ float s[];
  for (int i = threadIdx.x; i < N; i += blockDim.x) s[i] = scores[i];
  block_sync();
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    const float si = s[i];
    const bool ni = isnan(si);
    int rank = 0;
    for (int j = 0; j < N; ++j) {
      const float sj = s[j];
      const bool nj = isnan(sj);
      const bool greater = (!nj && ni) || (!nj && !ni && sj > si);
      const bool equal = (nj && ni) || (!nj && !ni && sj == si);
      rank += (greater || (equal && j < i)) ? 1 : 0;
    }
    if (rank < k) idx[rank] = i;
  }
}

// ------------------------------------------------------------------ refill ----
__global__ void __launch_bounds__(kCacheThreads) beam_refill_kernel(
    const float* __restrict__ sx, const float* __restrict__ sr, const float* __restrict__ sd,
    const float* __restrict__ sa, const uint8_t* __restrict__ sh, float* __restrict__ dx, float* __restrict__ dr,
    float* __restrict__ dd, float* __restrict__ da, uint8_t* __restrict__ dh, const int32_t* __restrict__ surv,
    int children, float sigma, const float* __restrict__ noise, long long D) {
  const int slot = blockIdx.y, c = blockIdx.x;
  const int p = slot / (children + 1), j = slot % (children + 1);
  const int src = surv[p];
  const long long lo = (long long)c * kChunkElems;
  const long long hi = min(D, lo + kChunkElems);
  const long long so = (long long)src * D, dof = (long long)slot * D;
  const float* nz = j > 0 ? noise + (long long)(p * children + j - 1) * D : nullptr;
  for (long long e = lo + threadIdx.x; e < hi; e += kCacheThreads) {
    float xv = sx[so + e];
    if (nz) xv += sigma * nz[e];
    dx[dof + e] = xv;
    dr[dof + e] = sr[so + e];
    dd[dof + e] = sd[so + e];
  }
  if (c == 0 && threadIdx.x == 0) {
    da[slot] = sa[src];
    dh[slot] = sh[src] ? 1 : 0;   // a carried drift belongs to the source slot's latent: not copied
  }
}

}  // namespace cs

using namespace cs;

// Workspace layout: drift partials [N][nch][2], score partials [N][nch], then (at a
// 256-byte boundary) the single-pass step's arrival counter and the skipped candidates'
// list with its count [N + 1].
static size_t counters_offset(int N, long long D) {
  return ((size_t)N * cache_chunks(D) * 3 * sizeof(float) + 255) / 256 * 256;
}

extern "C" size_t cs_cache_workspace_bytes(int N, long long D) {
  if (N <= 0 || D <= 0) return 0;
  return counters_offset(N, D) + sizeof(unsigned) + (size_t)(N + 1) * sizeof(int32_t) + 256;
}

extern "C" cs_status cs_cache_decide(const float* x, const float* x_ref, float* accum, uint8_t* has_ref, int N,
                                     long long D, int step_k, int T, float tau, int K_w, int K_c,
                                     const uint8_t* force, uint8_t* skip_mask, int32_t* idx, int32_t* n_compute,
                                     void* workspace, int* err, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && D > 0, "cs_cache_decide: need 0 < N <= 4096 and D > 0 (N=%d D=%lld)", N, D);
  CS_REQUIRE(x && x_ref && accum && has_ref && skip_mask && idx && n_compute && workspace,
             "cs_cache_decide: null pointer");
  CS_REQUIRE(step_k >= 1 && step_k <= T, "cs_cache_decide: step %d outside 1..T=%d", step_k, T);
  const int nch = cache_chunks(D);
  const int wf = window_forced(step_k, T, K_w, K_c) ? 1 : 0;
  float* partials = static_cast<float*>(workspace);
  if (!wf) {
    drift_partials_kernel<<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, has_ref, D, wf, N, partials);
    CS_LAUNCHED();
  }
  decide_finalize_kernel<<<1, 1024, N, stream>>>(partials, nch, accum, has_ref, N, wf, tau, force, skip_mask, idx,
                                                n_compute, err);
  CS_LAUNCHED();
  return CS_OK;
}

extern "C" cs_status cs_cache_apply(float* x, float* x_ref, float* delta, const float* v, const uint8_t* skip_mask,
                                    int N, long long D, float t_cur, float t_next, const float* target,
                                    float* scores, void* workspace, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && D > 0, "cs_cache_apply: need 0 < N <= 4096 and D > 0");
  CS_REQUIRE(x && x_ref && delta && v && skip_mask, "cs_cache_apply: null pointer");
  CS_REQUIRE(!target || (scores && workspace), "cs_cache_apply: scoring needs scores and workspace");
  const int nch = cache_chunks(D);
  const float h = t_next - t_cur;
  float* partials = workspace ? static_cast<float*>(workspace) + (size_t)N * nch * 2 : nullptr;
  if (target) {
    apply_kernel<true><<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, delta, v, skip_mask, D, h, t_next,
                                                                   target, partials);
    CS_LAUNCHED();
    score_finalize_kernel<<<(N + 3) / 4, 128, 0, stream>>>(partials, nch, N, scores);
    CS_LAUNCHED();
  } else {
    apply_kernel<false><<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, delta, v, skip_mask, D, h, t_next,
                                                                    nullptr, nullptr);
    CS_LAUNCHED();
  }
  return CS_OK;
}

extern "C" cs_status cs_cache_decide_cfg(const float* x, const float* x_ref, float* accum, uint8_t* has_ref, int N,
                                         long long D, int step_k, int T, float tau, int K_w, int K_c,
                                         const uint8_t* force, uint8_t* skip_mask, int32_t* idx,
                                         int32_t* n_compute, void* workspace, int* err, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && 2 * N <= 4096 && D > 0, "cs_cache_decide_cfg: need 0 < 2N <= 4096 and D > 0");
  CS_REQUIRE(x && x_ref && accum && has_ref && skip_mask && idx && n_compute && workspace,
             "cs_cache_decide_cfg: null pointer");
  CS_REQUIRE(step_k >= 1 && step_k <= T, "cs_cache_decide_cfg: step %d outside 1..T=%d", step_k, T);
  const int nch = cache_chunks(D), S = 2 * N;
  const int wf = window_forced(step_k, T, K_w, K_c) ? 1 : 0;
  float* partials = static_cast<float*>(workspace);
  if (!wf) {
    drift_partials_kernel<<<dim3(nch, S), kCacheThreads, 0, stream>>>(x, x_ref, has_ref, D, wf, N, partials);
    CS_LAUNCHED();
  }
  decide_finalize_kernel<<<1, 1024, S, stream>>>(partials, nch, accum, has_ref, S, wf, tau, force, skip_mask, idx,
                                                n_compute, err);
  CS_LAUNCHED();
  return CS_OK;
}

extern "C" cs_status cs_cache_apply_cfg(float* x, float* x_ref, float* delta, const float* v,
                                        const uint8_t* skip_mask, int N, long long D, float t_cur, float t_next,
                                        float w, const float* target, float* scores, void* workspace,
                                        cudaStream_t stream) {
  CS_REQUIRE(N > 0 && 2 * N <= 4096 && D > 0, "cs_cache_apply_cfg: need 0 < 2N <= 4096 and D > 0");
  CS_REQUIRE(x && x_ref && delta && v && skip_mask, "cs_cache_apply_cfg: null pointer");
  CS_REQUIRE(!target || (scores && workspace), "cs_cache_apply_cfg: scoring needs scores and workspace");
  const int nch = cache_chunks(D);
  const float h = t_next - t_cur;
  float* partials = workspace ? static_cast<float*>(workspace) + (size_t)2 * N * nch * 2 : nullptr;
  if (target) {
    apply_cfg_kernel<true><<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, delta, v, skip_mask, N, D, h,
                                                                       t_next, w, target, partials);
    CS_LAUNCHED();
    score_finalize_kernel<<<(N + 3) / 4, 128, 0, stream>>>(partials, nch, N, scores);
    CS_LAUNCHED();
  } else {
    apply_cfg_kernel<false><<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, delta, v, skip_mask, N, D, h,
                                                                        t_next, w, nullptr, nullptr);
    CS_LAUNCHED();
  }
  return CS_OK;
}

namespace cs {

// CTAs of 256 threads that fit on all SMs at once for `kernel` (dynamic shared memory
// `smem` bytes), looked up once per (kernel, smem).
static int resident_grid(const void* kernel, int smem) {
  static std::mutex mu;
  static std::vector<std::pair<std::pair<const void*, int>, int>> known;
  std::lock_guard<std::mutex> lock(mu);
  for (auto& k : known)
    if (k.first.first == kernel && k.first.second == smem) return k.second;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kCacheThreads, smem) != cudaSuccess || per_sm < 1) {
    (void)cudaGetLastError();
    per_sm = 4;
  }
  const int g = per_sm * num_sms();
  known.push_back({{kernel, smem}, g});
  return g;
}

// The single-pass decide + skip of cs_search_step.  sc.counter: the arrival counter, zero
// on entry (every completed call leaves it at zero; the model keeps its own, zeroed when
// allocated); sc.sidx: N + 1 ints (the skipped candidates and their count).
// sc.counter == nullptr: the pair inside the workspace, whose counter is cleared first.
cs_status decide_skip_run(float* x, const float* x_ref, const float* delta, float* accum, uint8_t* has_ref, int N,
                          long long D, int step_k, int T, float t_cur, float t_next, float tau, int K_w, int K_c,
                          const uint8_t* force, uint8_t* skip_mask, int32_t* idx, int32_t* n_compute,
                          const float* target, void* workspace, StepScratch sc, int* err, cudaStream_t stream) {
  const int nch = cache_chunks(D);
  const int wf = window_forced(step_k, T, K_w, K_c) ? 1 : 0;
  if (wf && !force) {
    decide_all_compute_kernel<<<1, 256, 0, stream>>>(accum, has_ref, N, skip_mask, idx, n_compute);
    CS_LAUNCHED();
    return CS_OK;
  }
  float* partials = static_cast<float*>(workspace);
  float* spart = partials + (size_t)N * nch * 2;
  const bool counter_zero = sc.counter != nullptr;
  if (!counter_zero) {
    sc.counter = reinterpret_cast<unsigned*>(static_cast<char*>(workspace) + counters_offset(N, D));
    sc.sidx = reinterpret_cast<int32_t*>(sc.counter + 1);
  }
  const int items = N * nch;
  // one wave of CTAs, each taking a contiguous range of chunks: a grid larger than what
  // fits on the SMs at once leaves a second, partial wave that ends late (measured on
  // GB300: 1024 one-chunk CTAs at 5 per SM took 14.6 us for what 512 two-chunk CTAs move
  // in about 10); no CTA waits for another, so residency is a speed matter only
  int grid = resident_grid((const void*)drift_decide_kernel, N);
  if (wf) {
    // forced mask inside the window: no drift is evaluated, one CTA decides
    decide_finalize_kernel<<<1, 1024, N, stream>>>(partials, nch, accum, has_ref, N, 1, tau, force, skip_mask, idx,
                                                  n_compute, err, sc.sidx);
    CS_LAUNCHED();
  } else {
    if (!counter_zero) CS_CUDA(cudaMemsetAsync(sc.counter, 0, sizeof(unsigned), stream));
    const int g1 = grid < items ? grid : items;   // contiguous ranges of items/g1 chunks
    drift_decide_kernel<<<g1, kCacheThreads, N, stream>>>(x, x_ref, accum, has_ref, N, D, nch, tau, force, skip_mask,
                                                         idx, n_compute, sc.sidx, partials, sc.counter, err);
    CS_LAUNCHED();
  }
  // the skip update's grid is sized before the decisions exist: CTAs without items return
  grid = resident_grid(target ? (const void*)skip_update_kernel<true> : (const void*)skip_update_kernel<false>, 0);
  if (grid > items) grid = items;
  const float h = t_next - t_cur;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kCacheThreads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const int32_t* sidx = sc.sidx;
  if (target)
    CS_CUDA(cudaLaunchKernelEx(&cfg, skip_update_kernel<true>, x, delta, sidx, N, D, nch, h, t_next, target, spart));
  else
    CS_CUDA(cudaLaunchKernelEx(&cfg, skip_update_kernel<false>, x, delta, sidx, N, D, nch, h, t_next,
                               (const float*)nullptr, (float*)nullptr));
  CS_LAUNCHED();
  return CS_OK;
}

// Load every cache kernel now (cudaFuncGetAttributes loads a kernel that lazy module
// loading has not loaded yet), so that no search step pays for a first launch: the
// decision pass and the skip update first run on the first free step, the scoring
// variants on the last step of a search.
cs_status load_cache_kernels() {
  const void* fns[] = {
      (const void*)drift_decide_kernel,          (const void*)skip_update_kernel<true>,
      (const void*)skip_update_kernel<false>,    (const void*)velocity_update_kernel<true, false>,
      (const void*)velocity_update_kernel<false, false>, (const void*)score_finalize_split_kernel,
      (const void*)velocity_update_kernel<true, true>, (const void*)velocity_update_kernel<false, true>,
      (const void*)carry_skip_kernel<true, true>,  (const void*)carry_skip_kernel<false, true>,
      (const void*)carry_skip_kernel<true, false>, (const void*)carry_skip_kernel<false, false>,
      (const void*)carry_rows_finalize_kernel,
      (const void*)decide_finalize_kernel,       (const void*)decide_all_compute_kernel,
      (const void*)drift_partials_kernel,        (const void*)apply_computed_kernel<true>,
      (const void*)apply_computed_kernel<false>, (const void*)score_finalize_kernel,
      (const void*)topk_kernel,                  (const void*)beam_refill_kernel,
  };
  for (const void* f : fns) {
    cudaFuncAttributes a;
    CS_CUDA(cudaFuncGetAttributes(&a, f));
  }
  return CS_OK;
}

cs_status apply_tokens_run(float* x, float* x_ref, float* delta, float* accum, uint8_t* has_ref, uint8_t* skip_mask,
                           const float* hout, const int32_t* idx, int n_c, int N, int C, int F, int H, int W,
                           float t_cur, float t_next, const float* target, float* scores, const float* spart,
                           float* tpart, long long idx_limit, int* err, cudaStream_t stream) {
  const long long D = (long long)C * F * H * W;
  const int ntiles = F * (H / 2);
  const float h = t_next - t_cur;
  const size_t smem = (size_t)(W / 4) * (2 * C + 1) * sizeof(float4);
  if (n_c > 0) {
    const dim3 grid(ntiles, n_c);
    if (target)
      velocity_update_kernel<true, false><<<grid, kCacheThreads, smem, stream>>>(
          hout, idx, C, F, H, W, x, x_ref, delta, accum, has_ref, skip_mask, h, t_next, target, tpart, CarryOut{},
          idx_limit, err);
    else
      velocity_update_kernel<false, false><<<grid, kCacheThreads, smem, stream>>>(
          hout, idx, C, F, H, W, x, x_ref, delta, accum, has_ref, skip_mask, h, t_next, nullptr, nullptr,
          CarryOut{}, idx_limit, err);
    CS_LAUNCHED();
  }
  if (target) {
    score_finalize_split_kernel<<<(N + 3) / 4, 128, 0, stream>>>(spart, cache_chunks(D), tpart, ntiles, skip_mask, N,
                                                                 scores);
    CS_LAUNCHED();
  }
  return CS_OK;
}

// ------------------------------------------------------------ carried form ----
// Step workspace of the carried form for `cap` candidate slots, each part at a 256-byte
// boundary: arrival counter; unit claim counter; skipped list [cap + 1]; carried
// sums [2][cap] (float2, by the parity of the step that reads them); partial pairs
// [cap][max(units, F*H/2)] (float2; units of 4096 elements); drift-pass partials
// [cap][nch][2]; skipped candidates' score partials [cap][units]; computed candidates'
// score partials [cap][F*H/2].
struct StepLayout {
  size_t counter, claim, sidx, drift, part, dpart, spart, tpart, total;
  int nch, nun, P;
};

static StepLayout step_layout(int cap, long long D, int ntiles) {
  StepLayout L;
  size_t o = 0;
  auto take = [&o](size_t bytes) {
    o = (o + 255) / 256 * 256;
    const size_t at = o;
    o += bytes;
    return at;
  };
  L.nch = cache_chunks(D);
  L.nun = carry_units(D);
  L.P = L.nun > ntiles ? L.nun : ntiles;
  L.counter = take(sizeof(unsigned));
  L.claim = take(sizeof(unsigned));
  L.sidx = take((size_t)(cap + 1) * sizeof(int32_t));
  L.drift = take((size_t)2 * cap * sizeof(float2));
  L.part = take((size_t)cap * L.P * sizeof(float2));
  L.dpart = take((size_t)cap * L.nch * 2 * sizeof(float));
  L.spart = take((size_t)cap * L.nun * sizeof(float));
  L.tpart = take((size_t)cap * ntiles * sizeof(float));
  L.total = (o + 255) / 256 * 256;
  return L;
}

size_t carry_state_bytes(int cap, long long D, int ntiles) { return step_layout(cap, D, ntiles).total; }

static CarryOut carry_out(const CarryState& cs, const StepLayout& L, int step_k) {
  char* b = static_cast<char*>(cs.base);
  return CarryOut{reinterpret_cast<float2*>(b + L.part), L.P,
                  reinterpret_cast<float2*>(b + L.drift) + (size_t)((step_k + 1) & 1) * cs.cap};
}

// The skip kernels' shared memory (the ring plus the list of up to 4096 candidates) is
// above the default limit: raised once per process for each instantiation.
static cs_status carry_skip_attributes() {
  static std::once_flag once;
  static cudaError_t e = cudaSuccess;
  std::call_once(once, [] {
    const int bytes = (int)carry_skip_smem(4096);
    const void* fns[] = {(const void*)carry_skip_kernel<true, true>, (const void*)carry_skip_kernel<false, true>,
                         (const void*)carry_skip_kernel<true, false>, (const void*)carry_skip_kernel<false, false>};
    for (const void* f : fns) {
      const cudaError_t r = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
      if (r != cudaSuccess && e == cudaSuccess) e = r;
    }
  });
  CS_CUDA(e);
  return CS_OK;
}

cs_status carry_decide_skip_run(float* x, const float* x_ref, const float* delta, float* accum, uint8_t* has_ref,
                                int N, int step_k, int T, float t_cur, float t_next, float tau, int K_w, int K_c,
                                const uint8_t* force, uint8_t* skip_mask, int32_t* idx, int32_t* n_compute,
                                const float* target, bool carried, const CarryState& cs, int* err,
                                cudaStream_t stream) {
  const long long D = cs.D;
  const int wf = window_forced(step_k, T, K_w, K_c) ? 1 : 0;
  if (wf && !force) {
    decide_all_compute_kernel<<<1, 256, 0, stream>>>(accum, has_ref, N, skip_mask, idx, n_compute);
    CS_LAUNCHED();
    return CS_OK;
  }
  const StepLayout L = step_layout(cs.cap, D, cs.ntiles);
  char* b = static_cast<char*>(cs.base);
  unsigned* counter = reinterpret_cast<unsigned*>(b + L.counter);
  unsigned* claim = reinterpret_cast<unsigned*>(b + L.claim);
  int32_t* sidx = reinterpret_cast<int32_t*>(b + L.sidx);
  const CarryOut co = carry_out(cs, L, step_k);
  const float2* din = reinterpret_cast<const float2*>(b + L.drift) + (size_t)(step_k & 1) * cs.cap;
  float* spart = reinterpret_cast<float*>(b + L.spart);
  const int nch = L.nch, nun = L.nun;
  if ((long long)N * nun >= (1ll << 31) || N > 4096) {
    set_error("carry_decide_skip_run: %d candidates of %lld elements exceed the item range", N, D);
    return CS_ERR_UNSUPPORTED;
  }
  const float h = t_next - t_cur;
  const size_t smem = carry_skip_smem(N);
  int grid = num_sms();                           // one CTA per SM (the ring takes its shared memory)
  if (grid > N * nun) grid = N * nun;
  CS_TRY(carry_skip_attributes());
  if (carried || wf) {
    // decisions from the carried drift (none is needed inside the window): one launch
    if (target)
      carry_skip_kernel<true, true><<<grid, kSkipThreads, smem, stream>>>(
          x, x_ref, delta, accum, has_ref, N, D, nun, wf, tau, force, skip_mask, idx, n_compute, nullptr, din, co,
          counter, claim, h, t_next, target, spart, err);
    else
      carry_skip_kernel<false, true><<<grid, kSkipThreads, smem, stream>>>(
          x, x_ref, delta, accum, has_ref, N, D, nun, wf, tau, force, skip_mask, idx, n_compute, nullptr, din, co,
          counter, claim, h, t_next, nullptr, nullptr, err);
    CS_LAUNCHED();
    return CS_OK;
  }
  // no carried drift: the drift pass decides, then the skip update follows it
  const int items = N * nch;
  int g1 = resident_grid((const void*)drift_decide_kernel, N);
  if (g1 > items) g1 = items;
  drift_decide_kernel<<<g1, kCacheThreads, N, stream>>>(x, x_ref, accum, has_ref, N, D, nch, tau, force, skip_mask,
                                                       idx, n_compute, sidx, reinterpret_cast<float*>(b + L.dpart),
                                                       counter, err);
  CS_LAUNCHED();
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kSkipThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const int32_t* csidx = sidx;
  const float2* no_drift = nullptr;
  float* no_accum = nullptr;
  uint8_t* no_u8 = nullptr;
  int32_t* no_i32 = nullptr;
  const uint8_t* no_force = nullptr;
  if (target)
    CS_CUDA(cudaLaunchKernelEx(&cfg, carry_skip_kernel<true, false>, x, x_ref, delta, no_accum, has_ref, N, D, nun, 0,
                               tau, no_force, no_u8, no_i32, no_i32, csidx, no_drift, co, counter, claim, h, t_next,
                               target, spart, err));
  else
    CS_CUDA(cudaLaunchKernelEx(&cfg, carry_skip_kernel<false, false>, x, x_ref, delta, no_accum, has_ref, N, D, nun,
                               0, tau, no_force, no_u8, no_i32, no_i32, csidx, no_drift, co, counter, claim, h,
                               t_next, (const float*)nullptr, (float*)nullptr, err));
  CS_LAUNCHED();
  return CS_OK;
}

cs_status carry_apply_tokens_run(float* x, float* x_ref, float* delta, float* accum, uint8_t* has_ref,
                                 uint8_t* skip_mask, const float* hout, const int32_t* idx, int n_c, int N, int C,
                                 int F, int H, int W, int step_k, float t_cur, float t_next, const float* target,
                                 float* scores, const CarryState& cs, long long idx_limit, int* err,
                                 cudaStream_t stream) {
  const long long D = cs.D;
  const int ntiles = F * (H / 2);
  const StepLayout L = step_layout(cs.cap, D, cs.ntiles);
  char* b = static_cast<char*>(cs.base);
  const CarryOut co = carry_out(cs, L, step_k);
  float* spart = reinterpret_cast<float*>(b + L.spart);
  float* tpart = reinterpret_cast<float*>(b + L.tpart);
  const float h = t_next - t_cur;
  const size_t smem = (size_t)(W / 4) * (2 * C + 1) * sizeof(float4);
  if (n_c > 0) {
    const dim3 grid(ntiles, n_c);
    if (target)
      velocity_update_kernel<true, true><<<grid, kCacheThreads, smem, stream>>>(
          hout, idx, C, F, H, W, x, x_ref, delta, accum, has_ref, skip_mask, h, t_next, target, tpart, co, idx_limit,
          err);
    else
      velocity_update_kernel<false, true><<<grid, kCacheThreads, smem, stream>>>(
          hout, idx, C, F, H, W, x, x_ref, delta, accum, has_ref, skip_mask, h, t_next, nullptr, nullptr, co,
          idx_limit, err);
    CS_LAUNCHED();
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(n_c);
    cfg.blockDim = dim3(kCacheThreads);
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    CS_CUDA(cudaLaunchKernelEx(&cfg, carry_rows_finalize_kernel, idx, ntiles, co, idx_limit, err));
    CS_LAUNCHED();
  }
  if (target) {
    score_finalize_split_kernel<<<(N + 3) / 4, 128, 0, stream>>>(spart, L.nun, tpart, ntiles, skip_mask, N, scores);
    CS_LAUNCHED();
  }
  return CS_OK;
}

// Whether apply_tokens_run handles this latent shape (16-byte rows along W and a staging
// tile that fits the default shared memory of a CTA).
bool apply_tokens_supported(int C, int F, int H, int W) {
  return C > 0 && F > 0 && H > 0 && W > 0 && (H % 2) == 0 && (W % 4) == 0 &&
         (size_t)(W / 4) * (2 * C + 1) * sizeof(float4) <= 48 * 1024;
}

}  // namespace cs

extern "C" cs_status cs_cache_decide_skip(float* x, const float* x_ref, const float* delta, float* accum,
                                          uint8_t* has_ref, int N, long long D, int step_k, int T, float t_cur,
                                          float t_next, float tau, int K_w, int K_c, const uint8_t* force,
                                          uint8_t* skip_mask, int32_t* idx, int32_t* n_compute,
                                          const float* target, void* workspace, int* err, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && D > 0, "cs_cache_decide_skip: need 0 < N <= 4096 and D > 0");
  CS_REQUIRE(x && x_ref && delta && accum && has_ref && skip_mask && idx && n_compute && workspace,
             "cs_cache_decide_skip: null pointer");
  CS_REQUIRE(step_k >= 1 && step_k <= T, "cs_cache_decide_skip: step %d outside 1..T=%d", step_k, T);
  CS_REQUIRE((D & 7) == 0 && (reinterpret_cast<uintptr_t>(x) & 31) == 0 &&
                 (reinterpret_cast<uintptr_t>(x_ref) & 31) == 0 && (reinterpret_cast<uintptr_t>(delta) & 31) == 0 &&
                 (!target || (reinterpret_cast<uintptr_t>(target) & 31) == 0),
             "cs_cache_decide_skip: needs D %% 8 == 0 and 32-byte aligned tensors");
  return decide_skip_run(x, x_ref, delta, accum, has_ref, N, D, step_k, T, t_cur, t_next, tau, K_w, K_c, force,
                         skip_mask, idx, n_compute, target, workspace, StepScratch{}, err, stream);
}

extern "C" cs_status cs_cache_apply_tokens(float* x, float* x_ref, float* delta, float* accum, uint8_t* has_ref,
                                           uint8_t* skip_mask, const float* hout, const int32_t* idx, int n_c, int N,
                                           int C, int F, int H, int W, float t_cur, float t_next,
                                           const float* target, float* scores, void* workspace, float* tile_partials,
                                           int* err, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && n_c >= 0 && n_c <= N, "cs_cache_apply_tokens: need 0 <= n_c <= N <= 4096");
  CS_REQUIRE(x && x_ref && delta && accum && has_ref && skip_mask && (n_c == 0 || (hout && idx)),
             "cs_cache_apply_tokens: null pointer");
  CS_REQUIRE(apply_tokens_supported(C, F, H, W), "cs_cache_apply_tokens: needs even H and W %% 4 == 0 (W=%d)", W);
  CS_REQUIRE(!target || (scores && workspace && tile_partials),
             "cs_cache_apply_tokens: scoring needs scores, workspace and tile_partials");
  const uintptr_t al = reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(x_ref) |
                       reinterpret_cast<uintptr_t>(delta) | reinterpret_cast<uintptr_t>(hout) |
                       reinterpret_cast<uintptr_t>(target);
  CS_REQUIRE((al & 15) == 0, "cs_cache_apply_tokens: tensors must be 16-byte aligned");
  const long long D = (long long)C * F * H * W;
  const float* spart = workspace ? static_cast<const float*>(workspace) + (size_t)N * cache_chunks(D) * 2 : nullptr;
  return apply_tokens_run(x, x_ref, delta, accum, has_ref, skip_mask, hout, idx, n_c, N, C, F, H, W, t_cur, t_next,
                          target, scores, spart, tile_partials, (long long)N, err, stream);
}

extern "C" size_t cs_cache_step_bytes(int N, int C, int F, int H, int W) {
  if (N <= 0 || !apply_tokens_supported(C, F, H, W)) return 0;
  return carry_state_bytes(N, (long long)C * F * H * W, F * (H / 2));
}

extern "C" cs_status cs_cache_decide_skip_carry(float* x, const float* x_ref, const float* delta, float* accum,
                                                uint8_t* has_ref, int N, int C, int F, int H, int W, int step_k,
                                                int T, float t_cur, float t_next, float tau, int K_w, int K_c,
                                                const uint8_t* force, uint8_t* skip_mask, int32_t* idx,
                                                int32_t* n_compute, const float* target, int carried,
                                                void* step_ws, int* err, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096, "cs_cache_decide_skip_carry: need 0 < N <= 4096 (N=%d)", N);
  CS_REQUIRE(apply_tokens_supported(C, F, H, W), "cs_cache_decide_skip_carry: latent %dx%dx%dx%d unsupported", C, F,
             H, W);
  CS_REQUIRE(x && x_ref && delta && accum && has_ref && skip_mask && idx && n_compute && step_ws,
             "cs_cache_decide_skip_carry: null pointer");
  CS_REQUIRE(step_k >= 1 && step_k <= T, "cs_cache_decide_skip_carry: step %d outside 1..T=%d", step_k, T);
  const CarryState cs{step_ws, N, (long long)C * F * H * W, F * (H / 2)};
  return carry_decide_skip_run(x, x_ref, delta, accum, has_ref, N, step_k, T, t_cur, t_next, tau, K_w, K_c, force,
                               skip_mask, idx, n_compute, target, carried != 0, cs, err, stream);
}

extern "C" cs_status cs_cache_apply_tokens_carry(float* x, float* x_ref, float* delta, float* accum,
                                                 uint8_t* has_ref, uint8_t* skip_mask, const float* hout,
                                                 const int32_t* idx, int n_c, int N, int C, int F, int H, int W,
                                                 int step_k, float t_cur, float t_next, const float* target,
                                                 float* scores, void* step_ws, int* err, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && n_c >= 0 && n_c <= N, "cs_cache_apply_tokens_carry: bad N=%d / n_c=%d", N, n_c);
  CS_REQUIRE(apply_tokens_supported(C, F, H, W), "cs_cache_apply_tokens_carry: latent %dx%dx%dx%d unsupported", C,
             F, H, W);
  CS_REQUIRE(x && x_ref && delta && accum && has_ref && skip_mask && step_ws && (n_c == 0 || (hout && idx)),
             "cs_cache_apply_tokens_carry: null pointer");
  CS_REQUIRE(!target || scores, "cs_cache_apply_tokens_carry: scoring needs scores");
  const CarryState cs{step_ws, N, (long long)C * F * H * W, F * (H / 2)};
  return carry_apply_tokens_run(x, x_ref, delta, accum, has_ref, skip_mask, hout, idx, n_c, N, C, F, H, W, step_k,
                                t_cur, t_next, target, scores, cs, N, err, stream);
}

extern "C" cs_status cs_cache_apply_computed(float* x, float* x_ref, float* delta, const float* v,
                                             const uint8_t* skip_mask, int N, long long D, float t_cur, float t_next,
                                             const float* target, float* scores, void* workspace,
                                             cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && D > 0 && (D & 3) == 0, "cs_cache_apply_computed: bad sizes");
  CS_REQUIRE(x && x_ref && delta && v && skip_mask, "cs_cache_apply_computed: null pointer");
  CS_REQUIRE(!target || (scores && workspace), "cs_cache_apply_computed: scoring needs scores and workspace");
  const int nch = cache_chunks(D);
  const float h = t_next - t_cur;
  float* spart = workspace ? static_cast<float*>(workspace) + (size_t)N * nch * 2 : nullptr;
  if (target) {
    apply_computed_kernel<true><<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, delta, v, skip_mask, D, h,
                                                                            t_next, target, spart);
    CS_LAUNCHED();
    score_finalize_kernel<<<(N + 3) / 4, 128, 0, stream>>>(spart, nch, N, scores);
    CS_LAUNCHED();
  } else {
    apply_computed_kernel<false><<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, delta, v, skip_mask, D, h,
                                                                             t_next, nullptr, nullptr);
    CS_LAUNCHED();
  }
  return CS_OK;
}

extern "C" cs_status cs_score(const float* x, const float* target, int N, long long D, float* scores,
                              void* workspace, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && D > 0 && x && target && scores && workspace, "cs_score: bad arguments");
  const int nch = cache_chunks(D);
  float* partials = static_cast<float*>(workspace) + (size_t)N * nch * 2;
  sqdist_partials_kernel<<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, target, D, partials);
  CS_LAUNCHED();
  score_finalize_kernel<<<(N + 3) / 4, 128, 0, stream>>>(partials, nch, N, scores);
  CS_LAUNCHED();
  return CS_OK;
}

extern "C" cs_status cs_select_topk(const float* scores, int N, int k, int32_t* idx, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && N <= 4096 && k >= 1 && k <= N && scores && idx, "cs_select_topk: need 1 <= k <= N <= 4096");
  topk_kernel<<<1, 256, N * sizeof(float), stream>>>(scores, N, k, idx);
  CS_LAUNCHED();
  return CS_OK;
}

extern "C" cs_status cs_beam_refill(const float* sx, const float* sr, const float* sd, const float* sa,
                                    const uint8_t* sh, float* dx, float* dr, float* dd, float* da, uint8_t* dh,
                                    const int32_t* surv, int keep, int children, float sigma, const float* noise,
                                    long long D, cudaStream_t stream) {
  CS_REQUIRE(keep > 0 && children >= 0 && D > 0, "cs_beam_refill: bad sizes");
  CS_REQUIRE(sx && sr && sd && sa && sh && dx && dr && dd && da && dh && surv && (children == 0 || noise),
             "cs_beam_refill: null pointer");
  CS_REQUIRE(sx != dx && sr != dr && sd != dd, "cs_beam_refill: source and destination must differ");
  const int slots = keep * (children + 1);
  beam_refill_kernel<<<dim3(cache_chunks(D), slots), kCacheThreads, 0, stream>>>(
      sx, sr, sd, sa, sh, dx, dr, dd, da, dh, surv, children, sigma, noise, D);
  CS_LAUNCHED();
  return CS_OK;
}

// ---------------------------------------------------------------------------
// Allocation-free variant of cs_cache_decide.
//
// Some callers cannot call cudaMalloc: a serving runtime whose memory pool has taken
// all device memory at start-up, or host code that must never let an allocation
// synchronise the device in the middle of a step.  For them the drift partial sums
// live in a fixed array compiled into this library instead of a caller workspace.
// The array exists once per GPU that loads the library and is held until the process
// exits; every call on that GPU shares it, so calls that overlap on the GPU (two
// streams, or two threads) race and must be serialised by the caller.  Each call
// writes every partial it later reads, so nothing carried over from an earlier call
// is ever used and nothing needs clearing.
// ---------------------------------------------------------------------------
namespace cs {

constexpr int kStaticMaxN = CS_NOALLOC_MAX_N;
constexpr int kStaticMaxChunks = CS_NOALLOC_MAX_CHUNKS;
static __device__ __align__(256) float g_decide_scratch[kStaticMaxN * kStaticMaxChunks * 2];

static std::mutex g_scratch_mu;
// Device address of g_decide_scratch per device ordinal, looked up once and kept for the
// life of the process (a cudaDeviceReset would leave it stale; the header says so).
static float* g_scratch_ptr[256] = {};

// Device address of the scratch array on the current device (looked up once per device).
static cs_status static_scratch(float** out) {
  int dev = 0;
  CS_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 256) {
    set_error("cs_cache_decide_noalloc: device ordinal %d out of range", dev);
    return CS_ERR_ARG;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_decide_scratch);
    if (e != cudaSuccess || !p) {
      set_error("cs_cache_decide_noalloc: cudaGetSymbolAddress failed on device %d: %s", dev, cudaGetErrorString(e));
      return CS_ERR_CUDA;
    }
    g_scratch_ptr[dev] = static_cast<float*>(p);
  }
  *out = g_scratch_ptr[dev];
  return CS_OK;
}

}  // namespace cs

extern "C" cs_status cs_cache_decide_noalloc(const float* x, const float* x_ref, float* accum, uint8_t* has_ref,
                                             int N, long long D, int step_k, int T, float tau, int K_w, int K_c,
                                             const uint8_t* force, uint8_t* skip_mask, int32_t* idx,
                                             int32_t* n_compute, int* err, cudaStream_t stream) {
  CS_REQUIRE(N > 0 && D > 0, "cs_cache_decide_noalloc: need N > 0 and D > 0 (N=%d D=%lld)", N, D);
  CS_REQUIRE(N <= kStaticMaxN, "cs_cache_decide_noalloc: N=%d exceeds the fixed scratch limit of %d candidates", N,
             kStaticMaxN);
  CS_REQUIRE(cache_chunks(D) <= kStaticMaxChunks,
             "cs_cache_decide_noalloc: D=%lld exceeds the fixed scratch limit of %lld elements per candidate", D,
             (long long)kStaticMaxChunks * kChunkElems);
  CS_REQUIRE(x && x_ref && accum && has_ref && skip_mask && idx && n_compute, "cs_cache_decide_noalloc: null pointer");
  CS_REQUIRE(step_k >= 1 && step_k <= T, "cs_cache_decide_noalloc: step %d outside 1..T=%d", step_k, T);
  float* partials = nullptr;
  CS_TRY(static_scratch(&partials));
  const int nch = cache_chunks(D);
  const int wf = window_forced(step_k, T, K_w, K_c) ? 1 : 0;
  if (!wf) {
    drift_partials_kernel<<<dim3(nch, N), kCacheThreads, 0, stream>>>(x, x_ref, has_ref, D, wf, N, partials);
    CS_LAUNCHED();
  }
  decide_finalize_kernel<<<1, 1024, N, stream>>>(partials, nch, accum, has_ref, N, wf, tau, force, skip_mask, idx,
                                                n_compute, err);
  CS_LAUNCHED();
  return CS_OK;
}
