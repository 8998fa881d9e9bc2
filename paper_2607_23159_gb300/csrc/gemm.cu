// tcgen05 GEMM for the DiT's Linear layers: C = A B^T, bf16 operands staged by TMA
// (128-byte swizzle) in a shared-memory ring, float32 accumulators in TMEM, fused
// epilogues (bias, GELU, gated residual add, attention-layout scatter).
//
// Persistent kernel, one CTA per SM, 6 warps:
//   warp 0      TMA producer (one lane): A tile 128 x 64 and B tile BN x 64 per stage
//   warp 1      TMEM allocator + MMA issuer (one lane): 4 x tcgen05.mma (K = 16) per stage
//   warps 2..5  epilogue: tcgen05.ld of the 128 x BN accumulator (warp w reads TMEM
//               lanes 32*(w%4)..+31), bias/activation, global stores
// Two TMEM accumulators (2 x BN columns) let the epilogue of tile i overlap the main
// loop of tile i+1.  Tiles are visited n-fastest so that the CTAs in flight share A
// rows and the whole of B in L2.
//
// BN = 256 runs as clusters of two CTAs on vertically adjacent tiles with the same B tile
// (MODE 2): rank 0 issues one M = 256 tcgen05.mma (cta_group::2) per K slice for the pair;
// each CTA's shared memory holds its 128 A rows and half of the B tile, both CTAs' TMA loads
// complete on rank 0's stage barrier, and the MMA commit releases the stage in both CTAs.
// Measured on GB300 (M 131040): the shared-memory writes of the B tile were the limit of
// the single-CTA kernel; MODE 2 halves them (1.66 -> 1.83 PFLOP/s at N 8960, K 1536).
// Every output element keeps the same K order in both modes.
#include <cuda.h>
#include <cuda_bf16.h>

#include "common.cuh"
#include "ptx.cuh"
#include "tma_host.h"

namespace cs {

struct GemmArgs {
  int M, N, K;
  const float* bias;
  const float* gate;
  void* out;
  int ldo;
  // attention-layout scatter (CS_EPI_QKV)
  __nv_bfloat16* q;
  __nv_bfloat16* k;
  __nv_bfloat16* vt;
  int L, d, heads, hd, hd_s, Lv, which_base;
  int tma_out;   // float32 epilogues: stage in shared memory and TMA-store / TMA-reduce-add the output
  int tma_qk;    // attention-layout epilogue: Q and K rows staged and TMA-stored (tmC = Q, tmD = K)
  int* err;
};

// MODE 0: one CTA per tile.  MODE 2: clusters of two running one M = 256 tcgen05.mma
// (cta_group::2) per K slice: each CTA holds its 128 A rows and half of the B tile, so every
// stage is half as large and the ring deeper.
template <int BN, int MODE = 0>
struct GemmCfg {
  static constexpr int BM = 128, BK = 64;
  static constexpr int B_ROWS = MODE == 2 ? BN / 2 : BN;   // B rows held in this CTA's shared memory
  static constexpr int STAGES = MODE == 2 ? 6 : (BN == 256 ? 4 : 6);
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = B_ROWS * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;
  static constexpr int OUT_BYTES = 4 * 2 * 32 * 128;   // per epilogue warp: two 32 x 32 float32 staging buffers
  static constexpr int SMEM = STAGES * STAGE_BYTES + OUT_BYTES + 1024 + 256;
  static constexpr uint32_t IDESC = idesc_bf16_f32(MODE == 2 ? 2 * BM : BM, BN);
};

// tanh on the SFU (tanh.approx.f32: the hardware instruction, relative error ~2^-11, below
// the bf16 rounding of the GELU output)
__device__ __forceinline__ float tanh_approx(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// tanh-GELU, 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))  (Hendrycks & Gimpel 2016), of two
// values at a time on the packed f32x2 pipe as 0.5 x + 0.5 x tanh(sqrt(2/pi) x (1 + 0.044715 x^2)):
// less than half the FP instructions of the scalar form, which the FFN-up GEMM measured as 3.7 %
// more throughput (its epilogue runs beside the next tile's main loop)
__device__ __forceinline__ void gelu_tanh2(float& a, float& b) {
  const uint64_t x = f2_pack(a, b);
  const uint64_t t = f2_fma(f2_mul(x, x), f2_pack(0.044715f, 0.044715f), f2_pack(1.f, 1.f));
  float ua, ub;
  f2_unpack(f2_mul(f2_mul(x, f2_pack(0.7978845608028654f, 0.7978845608028654f)), t), ua, ub);
  const uint64_t hx = f2_mul(x, f2_pack(0.5f, 0.5f));
  f2_unpack(f2_fma(hx, f2_pack(tanh_approx(ua), tanh_approx(ub)), hx), a, b);
}

// One thread's 32 consecutive accumulator columns [n, n+32) of row m.
template <int EPI>
__device__ __forceinline__ void epilogue_chunk(const GemmArgs& p, int m, int n, const uint32_t (&r)[32]) {
  float f[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) f[j] = __uint_as_float(r[j]);
  const bool full = (n + 32 <= p.N);
  if (p.bias) {
    if (full) {   // packed f32x2 adds (the same bits as scalar ones)
      const float4* b4 = reinterpret_cast<const float4*>(p.bias + n);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float4 b = __ldg(b4 + j);
        f2_unpack(f2_add(f2_pack(f[4 * j], f[4 * j + 1]), f2_pack(b.x, b.y)), f[4 * j], f[4 * j + 1]);
        f2_unpack(f2_add(f2_pack(f[4 * j + 2], f[4 * j + 3]), f2_pack(b.z, b.w)), f[4 * j + 2], f[4 * j + 3]);
      }
    } else {
      for (int j = 0; j < 32; ++j)
        if (n + j < p.N) f[j] += __ldg(p.bias + n + j);
    }
  }
  if constexpr (EPI == CS_EPI_F32) {
    float* o = static_cast<float*>(p.out) + (long long)m * p.ldo + n;
    if (full && (p.ldo % 4) == 0) {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        reinterpret_cast<float4*>(o)[j] = make_float4(f[4 * j], f[4 * j + 1], f[4 * j + 2], f[4 * j + 3]);
    } else {
      for (int j = 0; j < 32; ++j)
        if (n + j < p.N) o[j] = f[j];
    }
  } else if constexpr (EPI == CS_EPI_BF16 || EPI == CS_EPI_GELU_BF16) {
    if constexpr (EPI == CS_EPI_GELU_BF16) {
#pragma unroll
      for (int j = 0; j < 32; j += 2) gelu_tanh2(f[j], f[j + 1]);
    }
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(p.out) + (long long)m * p.ldo + n;
    if (full && (p.ldo % 8) == 0) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint4 u;
        u.x = pack_bf16x2(f[8 * j + 0], f[8 * j + 1]);
        u.y = pack_bf16x2(f[8 * j + 2], f[8 * j + 3]);
        u.z = pack_bf16x2(f[8 * j + 4], f[8 * j + 5]);
        u.w = pack_bf16x2(f[8 * j + 6], f[8 * j + 7]);
        reinterpret_cast<uint4*>(o)[j] = u;
      }
    } else {
      for (int j = 0; j < 32; ++j)
        if (n + j < p.N) o[j] = __float2bfloat16_rn(f[j]);
    }
  } else if constexpr (EPI == CS_EPI_RESID_F32) {
    float* o = static_cast<float*>(p.out) + (long long)m * p.ldo + n;
    if (full && (p.ldo % 4) == 0) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float4 x = reinterpret_cast<float4*>(o)[j];
        float4 g = p.gate ? __ldg(reinterpret_cast<const float4*>(p.gate + n) + j) : make_float4(1.f, 1.f, 1.f, 1.f);
        x.x += g.x * f[4 * j]; x.y += g.y * f[4 * j + 1]; x.z += g.z * f[4 * j + 2]; x.w += g.w * f[4 * j + 3];
        reinterpret_cast<float4*>(o)[j] = x;
      }
    } else {
      for (int j = 0; j < 32; ++j)
        if (n + j < p.N) o[j] += (p.gate ? __ldg(p.gate + n + j) : 1.f) * f[j];
    }
  } else if constexpr (EPI == CS_EPI_QKV) {
    // 32 | hd, so the chunk lies inside one head of one projection
    const int w = p.which_base + n / p.d;
    const int c0 = n % p.d;
    const int head = c0 / p.hd, e = c0 % p.hd;
    const int jb = m / p.L, l = m % p.L;
    const long long bh = (long long)jb * p.heads + head;
    if (w < 2) {
      __nv_bfloat16* o = (w == 0 ? p.q : p.k) + (bh * p.L + l) * p.hd_s + e;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint4 u;
        u.x = pack_bf16x2(f[8 * j + 0], f[8 * j + 1]);
        u.y = pack_bf16x2(f[8 * j + 2], f[8 * j + 3]);
        u.z = pack_bf16x2(f[8 * j + 4], f[8 * j + 5]);
        u.w = pack_bf16x2(f[8 * j + 6], f[8 * j + 7]);
        reinterpret_cast<uint4*>(o)[j] = u;
      }
    } else {
      __nv_bfloat16* o = p.vt + (bh * p.hd + e) * p.Lv + l;
#pragma unroll
      for (int j = 0; j < 32; ++j) o[(long long)j * p.Lv] = __float2bfloat16_rn(f[j]);
    }
  }
}

template <int BN, int EPI, int MODE>
__global__ void __launch_bounds__(192, 1)
    gemm_tcgen05_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmD,
                        const GemmArgs p) {
  using Cfg = GemmCfg<BN, MODE>;
  static_assert(MODE == 0 || MODE == 2, "MODE 0 (one CTA per tile) or 2 (two-SM MMA)");
  constexpr bool TWO_SM = MODE == 2;   // one cta_group::2 MMA stream issued by the cluster's rank 0
  constexpr bool PAIR = TWO_SM;        // clusters of two CTAs on vertically adjacent tiles
  constexpr int BM = Cfg::BM, BK = Cfg::BK, STAGES = Cfg::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * Cfg::A_BYTES;
  uint8_t* sOut = smem + STAGES * Cfg::STAGE_BYTES;   // 1024-aligned staging for float32 outputs
  uint64_t* full = reinterpret_cast<uint64_t*>(sOut + Cfg::OUT_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* teardown = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(teardown + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], TWO_SM ? 8 : 4);   // TWO_SM: rank 0's barrier, both CTAs' epilogue warps
    }
    mbar_init(teardown, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    if constexpr (TWO_SM) {
      tmem_alloc_2sm(tmem_slot, Cfg::TMEM_COLS);   // collective with the peer CTA's warp 1
      tmem_relinquish_2sm();
    } else {
      tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  block_sync();
  if (PAIR) cluster_sync();   // the peer's barriers exist before its loads complete on them
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int m_tiles = (p.M + BM - 1) / BM, n_tiles = (p.N + BN - 1) / BN;
  const int kblocks = p.K / BK;
  // work items, n-fastest: single CTA -> (m-tile, n-tile); PAIR -> (pair of m-tiles, n-tile),
  // of which the CTA of cluster rank r takes m-tile 2 * pair + r (rows past M are zero-filled
  // by TMA and never stored)
  const int rank = PAIR ? (int)cluster_ctarank() : 0;
  const int items = PAIR ? ((m_tiles + 1) / 2) * n_tiles : m_tiles * n_tiles;
  const int first = PAIR ? (int)blockIdx.x / 2 : (int)blockIdx.x;
  const int stride = PAIR ? (int)gridDim.x / 2 : (int)gridDim.x;
  auto item_m0 = [&](int it) { return (PAIR ? 2 * (it / n_tiles) + rank : it / n_tiles) * BM; };
  auto item_n0 = [&](int it) { return (it % n_tiles) * BN; };

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      for (int it = first; it < items && !*abort_flag; it += stride) {
        const int m0 = item_m0(it), n0 = item_n0(it);
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.err)) break;
          if constexpr (TWO_SM) {
            // both CTAs' halves complete on rank 0's barrier, which rank 0 arms for all of them
            if (rank == 0) mbar_arrive_expect_tx(&full[stage], 2 * Cfg::STAGE_BYTES);
            const uint32_t bar0 = cluster_map(&full[stage], 0);
            tma_load_2d_2sm(sA + stage * Cfg::A_BYTES, &tmA, bar0, kb * BK, m0);
            tma_load_2d_2sm(sB + stage * Cfg::B_BYTES, &tmB, bar0, kb * BK, n0 + rank * (BN / 2));
          } else {
            mbar_arrive_expect_tx(&full[stage], Cfg::STAGE_BYTES);
            tma_load_2d(sA + stage * Cfg::A_BYTES, &tmA, &full[stage], kb * BK, m0);
            tma_load_2d(sB + stage * Cfg::B_BYTES, &tmB, &full[stage], kb * BK, n0);
          }
          ++issued;
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
      }
      if (PAIR && !*abort_flag) {
        // every stage released by both CTAs' MMAs: no arrival from the peer is still on its way
        for (int i = 0; i < STAGES; ++i) {
          mbar_wait_teardown(&empty[stage], phase ^ 1);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
      }
      if (*abort_flag && !(TWO_SM && rank != 0)) {
        // drain: wait (bounded) for the loads of the last ring's worth of stages
        for (int back = 1; back <= STAGES && back <= issued; ++back) {
          int s = stage - back, ph = phase;
          if (s < 0) { s += STAGES; ph ^= 1; }
          mbar_wait_teardown(&full[s], ph);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && !(TWO_SM && rank != 0)) {   // TWO_SM: rank 0 issues for the pair
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (int it = first; it < items && !*abort_flag; it += stride) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag, p.err)) break;
        if constexpr (TWO_SM) fence_acq_rel_cluster();   // the peer's epilogue arrived from another CTA
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        bool ok = true;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, p.err)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + stage * Cfg::A_BYTES);
          const uint32_t b0 = smem_u32(sB + stage * Cfg::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            if constexpr (TWO_SM)
              umma_bf16_ss_2sm(d_tmem, sdesc_sw128(a0 + k * 32), sdesc_sw128(b0 + k * 32), Cfg::IDESC,
                               (kb | k) != 0 ? 1u : 0u);
            else
              umma_bf16_ss(d_tmem, sdesc_sw128(a0 + k * 32), sdesc_sw128(b0 + k * 32), Cfg::IDESC,
                           (kb | k) != 0 ? 1u : 0u);
          if constexpr (TWO_SM) umma_commit_2sm_mc(&empty[stage], 0x3);
          else umma_commit(&empty[stage]);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        if constexpr (TWO_SM) umma_commit_2sm_mc(&tfull[acc], 0x3);   // both CTAs' accumulators
        else umma_commit(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
      if (*abort_flag) {
        // every MMA issued so far must finish before TMEM is released
        if constexpr (TWO_SM) umma_commit_2sm_mc(teardown, 0x1);
        else umma_commit(teardown);
        mbar_wait_teardown(teardown, 0);
      }
    }
  } else {
    const int sp = warp & 3;
    const int row = sp * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    int nout = 0;   // chunks this warp has handed to TMA
    if (lane == 0 && (p.tma_out || p.tma_qk)) tma_prefetch_desc(&tmC);
    if (lane == 0 && p.tma_qk) tma_prefetch_desc(&tmD);
    for (int it = first; it < items; it += stride) {
      if (!__all_sync(0xffffffffu, mbar_wait(&tfull[acc], acc_phase, abort_flag, p.err))) break;
      tc_fence_after();
      const int m0 = item_m0(it), n0 = item_n0(it);
      const int m = m0 + row;
      const bool rows_in = m0 + sp * 32 < p.M;   // this warp has rows to store (uniform)
      const uint32_t tbase = tmem_base + ((uint32_t)(sp * 32) << 16) + acc * BN;
      if constexpr (EPI == CS_EPI_BF16 || EPI == CS_EPI_GELU_BF16) {
        if (p.tma_out) {
          // 64 columns at a time: 32 rows x 128 B of bf16 per warp -> staging -> one TMA store
#pragma unroll 1
          for (int c = 0; c < BN / 64; ++c) {
            const int n = n0 + c * 64;
            if (n >= p.N || !rows_in) break;   // uniform across the warp
            uint32_t r0[32], r1[32];
            tmem_ld32(tbase + c * 64, r0);
            tmem_ld32(tbase + c * 64 + 32, r1);
            uint8_t* buf = sOut + (sp * 2 + (nout & 1)) * 4096;
            if (lane == 0 && nout >= 2) bulk_wait_read_1();
            __syncwarp();
            const float4* b4 = p.bias ? reinterpret_cast<const float4*>(p.bias + n) : nullptr;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              float v[8];
#pragma unroll
              for (int j = 0; j < 8; ++j) v[j] = __uint_as_float(u < 4 ? r0[8 * u + j] : r1[8 * (u - 4) + j]);
              if (b4) {   // packed f32x2 adds: the same bits, half the instructions beside the main loop
                const float4 ba = __ldg(b4 + 2 * u), bb = __ldg(b4 + 2 * u + 1);
                f2_unpack(f2_add(f2_pack(v[0], v[1]), f2_pack(ba.x, ba.y)), v[0], v[1]);
                f2_unpack(f2_add(f2_pack(v[2], v[3]), f2_pack(ba.z, ba.w)), v[2], v[3]);
                f2_unpack(f2_add(f2_pack(v[4], v[5]), f2_pack(bb.x, bb.y)), v[4], v[5]);
                f2_unpack(f2_add(f2_pack(v[6], v[7]), f2_pack(bb.z, bb.w)), v[6], v[7]);
              }
              if constexpr (EPI == CS_EPI_GELU_BF16) {
#pragma unroll
                for (int j = 0; j < 8; j += 2) gelu_tanh2(v[j], v[j + 1]);
              }
              uint4 w;
              w.x = pack_bf16x2(v[0], v[1]);
              w.y = pack_bf16x2(v[2], v[3]);
              w.z = pack_bf16x2(v[4], v[5]);
              w.w = pack_bf16x2(v[6], v[7]);
              *reinterpret_cast<uint4*>(buf + lane * 128 + ((u ^ (lane & 7)) << 4)) = w;
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tmC, buf, n, m0 + sp * 32);
              bulk_commit();
            }
            ++nout;
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            if (TWO_SM) mbar_arrive_cluster(cluster_map(&tempty[acc], 0));
            else mbar_arrive(&tempty[acc]);
          }
          acc ^= 1;
          if (acc == 0) acc_phase ^= 1;
          continue;
        }
      }
      if constexpr (EPI == CS_EPI_QKV) {
        if (p.tma_qk) {
          // 64 columns (one head of Q or K) at a time: a warp whose 32 rows lie in one batch item
          // stages them and TMA-stores 32 consecutive (head, token) rows; V^T, rows that cross a
          // batch item or pass M go through the per-thread stores
#pragma unroll 1
          for (int c = 0; c < BN / 64; ++c) {
            const int n = n0 + c * 64;
            if (n >= p.N) break;   // uniform across the warp
            uint32_t r0[32], r1[32];
            tmem_ld32(tbase + c * 64, r0);
            tmem_ld32(tbase + c * 64 + 32, r1);
            const int w = p.which_base + n / p.d;
            const int mf = m0 + sp * 32;
            const int jb = mf / p.L;
            const bool staged = w < 2 && mf + 31 < p.M && (mf + 31) / p.L == jb;   // uniform across the warp
            if (!staged) {
              if (m < p.M) {
                epilogue_chunk<EPI>(p, m, n, r0);
                epilogue_chunk<EPI>(p, m, n + 32, r1);
              }
              continue;
            }
            const int c0 = n % p.d, head = c0 / p.hd, e = c0 % p.hd;
            uint8_t* buf = sOut + (sp * 2 + (nout & 1)) * 4096;
            if (lane == 0 && nout >= 2) bulk_wait_read_1();
            __syncwarp();
            const float4* b4 = p.bias ? reinterpret_cast<const float4*>(p.bias + n) : nullptr;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              float v[8];
#pragma unroll
              for (int j = 0; j < 8; ++j) v[j] = __uint_as_float(u < 4 ? r0[8 * u + j] : r1[8 * (u - 4) + j]);
              if (b4) {
                const float4 ba = __ldg(b4 + 2 * u), bb = __ldg(b4 + 2 * u + 1);
                f2_unpack(f2_add(f2_pack(v[0], v[1]), f2_pack(ba.x, ba.y)), v[0], v[1]);
                f2_unpack(f2_add(f2_pack(v[2], v[3]), f2_pack(ba.z, ba.w)), v[2], v[3]);
                f2_unpack(f2_add(f2_pack(v[4], v[5]), f2_pack(bb.x, bb.y)), v[4], v[5]);
                f2_unpack(f2_add(f2_pack(v[6], v[7]), f2_pack(bb.z, bb.w)), v[6], v[7]);
              }
              uint4 wv;
              wv.x = pack_bf16x2(v[0], v[1]);
              wv.y = pack_bf16x2(v[2], v[3]);
              wv.z = pack_bf16x2(v[4], v[5]);
              wv.w = pack_bf16x2(v[6], v[7]);
              *reinterpret_cast<uint4*>(buf + lane * 128 + ((u ^ (lane & 7)) << 4)) = wv;
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(w == 0 ? &tmC : &tmD, buf, e, (jb * p.heads + head) * p.L + (mf - jb * p.L));
              bulk_commit();
            }
            ++nout;
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            if (TWO_SM) mbar_arrive_cluster(cluster_map(&tempty[acc], 0));
            else mbar_arrive(&tempty[acc]);
          }
          acc ^= 1;
          if (acc == 0) acc_phase ^= 1;
          continue;
        }
      }
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        const int n = n0 + c * 32;
        if (n >= p.N) break;   // uniform across the warp
        uint32_t r[32];
        tmem_ld32(tbase + c * 32, r);
        if constexpr (EPI == CS_EPI_F32 || EPI == CS_EPI_RESID_F32) {
          if (p.tma_out) {
            if (!rows_in) continue;
            // this warp's 32 rows x 32 columns -> 128-byte-swizzled staging -> one TMA op
            // (a plain store, or for the residual an add performed in L2)
            uint8_t* buf = sOut + (sp * 2 + (nout & 1)) * 4096;
            if (lane == 0 && nout >= 2) bulk_wait_read_1();   // the op that last read this buffer is done
            __syncwarp();
            float f[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) f[j] = __uint_as_float(r[j]);
            const float4* b4 = p.bias ? reinterpret_cast<const float4*>(p.bias + n) : nullptr;
            const float4* g4 = (EPI == CS_EPI_RESID_F32 && p.gate) ? reinterpret_cast<const float4*>(p.gate + n)
                                                                   : nullptr;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              float4 v;
              uint64_t lo = f2_pack(f[4 * u], f[4 * u + 1]), hi = f2_pack(f[4 * u + 2], f[4 * u + 3]);
              if (b4) {   // packed f32x2 add and multiply: the same bits as scalar ones
                const float4 b = __ldg(b4 + u);
                lo = f2_add(lo, f2_pack(b.x, b.y));
                hi = f2_add(hi, f2_pack(b.z, b.w));
              }
              if (g4) {
                const float4 g = __ldg(g4 + u);
                lo = f2_mul(lo, f2_pack(g.x, g.y));
                hi = f2_mul(hi, f2_pack(g.z, g.w));
              }
              f2_unpack(lo, v.x, v.y);
              f2_unpack(hi, v.z, v.w);
              *reinterpret_cast<float4*>(buf + lane * 128 + ((u ^ (lane & 7)) << 4)) = v;
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              if constexpr (EPI == CS_EPI_RESID_F32) tma_reduce_add_2d(&tmC, buf, n, m0 + sp * 32);
              else tma_store_2d(&tmC, buf, n, m0 + sp * 32);
              bulk_commit();
            }
            ++nout;
            continue;
          }
        }
        if (m < p.M) epilogue_chunk<EPI>(p, m, n, r);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (TWO_SM) mbar_arrive_cluster(cluster_map(&tempty[acc], 0));
        else mbar_arrive(&tempty[acc]);
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1;
    }
    if (lane == 0 && nout > 0) bulk_wait_all();   // output writes complete before the CTA exits
  }

  tc_fence_before();
  block_sync();
  if (PAIR) cluster_sync();   // the peer's MMAs and arrivals on this CTA's barriers are done
  if (warp == 1) {
    tc_fence_after();
    if constexpr (TWO_SM) tmem_dealloc_2sm(tmem_base, Cfg::TMEM_COLS);
    else tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

template <int BN, int EPI, int MODE>
static cs_status launch_gemm(const void* A, const void* B, const GemmArgs& args, cudaStream_t stream) {
  using Cfg = GemmCfg<BN, MODE>;
  constexpr bool PAIR = MODE == 2;
  CUtensorMap ta, tb;
  const uint64_t da[2] = {(uint64_t)args.K, (uint64_t)args.M};
  const uint64_t sa[1] = {(uint64_t)args.K * 2};
  const uint32_t ba[2] = {64, 128};
  CS_TRY(make_tmap_bf16(&ta, A, 2, da, sa, ba));
  const uint64_t db[2] = {(uint64_t)args.K, (uint64_t)args.N};
  const uint32_t bb[2] = {64, (uint32_t)(PAIR ? BN / 2 : BN)};   // PAIR: each CTA loads half of the B tile
  CS_TRY(make_tmap_bf16(&tb, B, 2, db, sa, bb));
  // float32 outputs go through TMA when the output rows are TMA-addressable
  GemmArgs a = args;
  CUtensorMap tc = ta;   // unused unless a.tma_out
  a.tma_out = 0;
  if ((EPI == CS_EPI_F32 || EPI == CS_EPI_RESID_F32) && (args.N % 32) == 0 && (args.ldo % 4) == 0 &&
      (reinterpret_cast<uintptr_t>(args.out) & 15) == 0) {
    const uint64_t dc[2] = {(uint64_t)args.N, (uint64_t)args.M};
    const uint64_t sc[1] = {(uint64_t)args.ldo * 4};
    const uint32_t bc[2] = {32, 32};
    CS_TRY(make_tmap(&tc, args.out, 2, dc, sc, bc, true));
    a.tma_out = 1;
  }
  if ((EPI == CS_EPI_BF16 || EPI == CS_EPI_GELU_BF16) && (args.N % 64) == 0 && (args.ldo % 8) == 0 &&
      (reinterpret_cast<uintptr_t>(args.out) & 15) == 0) {
    const uint64_t dc[2] = {(uint64_t)args.N, (uint64_t)args.M};
    const uint64_t sc[1] = {(uint64_t)args.ldo * 2};
    const uint32_t bc[2] = {64, 32};
    CS_TRY(make_tmap(&tc, args.out, 2, dc, sc, bc, false));
    a.tma_out = 1;
  }
  CUtensorMap td = tc;   // unused unless a.tma_qk
  a.tma_qk = 0;
  if (EPI == CS_EPI_QKV && args.hd % 64 == 0 && args.d % 64 == 0 && args.N % 64 == 0 && args.q &&
      (reinterpret_cast<uintptr_t>(args.q) & 15) == 0 && (!args.k || (reinterpret_cast<uintptr_t>(args.k) & 15) == 0)) {
    // Q and K as 2-D [rows = (batch item, head, token), hd_s] bf16: a warp's 32 rows of one head
    // and one batch item are 32 consecutive rows there
    const uint64_t dq[2] = {(uint64_t)args.hd_s, (uint64_t)args.M * (uint64_t)args.heads};
    const uint64_t sq[1] = {(uint64_t)args.hd_s * 2};
    const uint32_t bq[2] = {64, 32};
    CS_TRY(make_tmap(&tc, args.q, 2, dq, sq, bq, false));
    td = tc;
    if (args.k) CS_TRY(make_tmap(&td, args.k, 2, dq, sq, bq, false));
    a.tma_qk = 1;
  }
  auto kern = gemm_tcgen05_kernel<BN, EPI, MODE>;
  CS_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM));
  const int m_tiles = (args.M + 127) / 128, n_tiles = (args.N + BN - 1) / BN;
  if (!PAIR) {
    const int tiles = m_tiles * n_tiles;
    const int grid = tiles < num_sms() ? tiles : num_sms();
    kern<<<grid, 192, Cfg::SMEM, stream>>>(ta, tb, tc, td, a);
    CS_LAUNCHED();
    return CS_OK;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = Cfg::SMEM;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(num_sms() / 2 * 2);
  static int max_clusters = -1;   // co-resident clusters of two (one CTA per SM); -1 = not asked yet
  if (max_clusters < 0) {
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    max_clusters = n;
  }
  if (max_clusters == 0) return launch_gemm<BN, EPI, 0>(A, B, args, stream);   // no cluster fits: one CTA per tile
  const int items = ((m_tiles + 1) / 2) * n_tiles;
  cfg.gridDim = dim3(2 * (items < max_clusters ? items : max_clusters));
  CS_CUDA(cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, td, a));
  CS_LAUNCHED();
  return CS_OK;
}

template <int EPI>
static cs_status dispatch_bn(const void* A, const void* B, const GemmArgs& args, cudaStream_t stream) {
  if (args.N >= 512) return launch_gemm<256, EPI, 2>(A, B, args, stream);
  return launch_gemm<128, EPI, 0>(A, B, args, stream);
}

cs_status gemm_run(const void* A, const void* B, int epi, const GemmArgs& args, cudaStream_t stream) {
  if (args.M <= 0 || args.N <= 0 || args.K <= 0 || (args.K % 64) != 0) {
    set_error("gemm: need M, N > 0 and K %% 64 == 0 (M=%d N=%d K=%d)", args.M, args.N, args.K);
    return CS_ERR_ARG;
  }
  if (!A || !B) {
    set_error("gemm: null operand");
    return CS_ERR_ARG;
  }
  switch (epi) {
    case CS_EPI_F32: return dispatch_bn<CS_EPI_F32>(A, B, args, stream);
    case CS_EPI_BF16: return dispatch_bn<CS_EPI_BF16>(A, B, args, stream);
    case CS_EPI_GELU_BF16: return dispatch_bn<CS_EPI_GELU_BF16>(A, B, args, stream);
    case CS_EPI_RESID_F32: return dispatch_bn<CS_EPI_RESID_F32>(A, B, args, stream);
    case CS_EPI_QKV: return dispatch_bn<CS_EPI_QKV>(A, B, args, stream);
  }
  set_error("gemm: unknown epilogue %d", epi);
  return CS_ERR_ARG;
}

}  // namespace cs

using namespace cs;

extern "C" cs_status cs_gemm_bf16(const void* A, const void* B, int M, int N, int K, int epi, const float* bias,
                                  const float* gate, void* out, int ldo, int* err, cudaStream_t stream) {
  CS_REQUIRE(epi != CS_EPI_QKV, "cs_gemm_bf16: use cs_gemm_qkv for the attention-layout epilogue");
  CS_REQUIRE(out && ldo >= N, "cs_gemm_bf16: need an output with ldo >= N");
  GemmArgs a{};
  a.M = M; a.N = N; a.K = K; a.bias = bias; a.gate = gate; a.out = out; a.ldo = ldo; a.err = err;
  return gemm_run(A, B, epi, a, stream);
}

extern "C" cs_status cs_gemm_qkv(const void* A, const void* B, int M, int N, int K, const float* bias, int L,
                                 int d, int heads, int which_base, void* q, void* k, void* vt, int Lv, int* err,
                                 cudaStream_t stream) {
  CS_REQUIRE(heads > 0 && d % heads == 0, "cs_gemm_qkv: d must be a multiple of heads");
  const int hd = d / heads;
  CS_REQUIRE(hd == 32 || hd == 128, "cs_gemm_qkv: head dim %d not supported (32 or 128)", hd);
  CS_REQUIRE(L > 0 && M % L == 0 && N % d == 0 && which_base >= 0 && which_base + N / d <= 3,
             "cs_gemm_qkv: inconsistent M=%d L=%d N=%d d=%d which_base=%d", M, L, N, d, which_base);
  CS_REQUIRE(Lv >= L && Lv % 8 == 0, "cs_gemm_qkv: Lv must be >= L and a multiple of 8");
  const int wmax = which_base + N / d;
  CS_REQUIRE((which_base > 0 || q) && (which_base > 1 || wmax <= 1 || k) && (wmax <= 2 || vt),
             "cs_gemm_qkv: missing output for a projection");
  GemmArgs a{};
  a.M = M; a.N = N; a.K = K; a.bias = bias; a.err = err;
  a.q = static_cast<__nv_bfloat16*>(q); a.k = static_cast<__nv_bfloat16*>(k);
  a.vt = static_cast<__nv_bfloat16*>(vt);
  a.L = L; a.d = d; a.heads = heads; a.hd = hd; a.hd_s = hd < 64 ? 64 : hd; a.Lv = Lv; a.which_base = which_base;
  return gemm_run(A, B, CS_EPI_QKV, a, stream);
}
