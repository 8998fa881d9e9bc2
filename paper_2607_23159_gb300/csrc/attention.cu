// Flash attention forward on the tcgen05 tensor cores (self- and cross-attention of
// the DiT blocks).  One CTA takes 256 query rows of one (batch item, head) as two
// 128-row tiles A and B and streams the keys in tiles of 128:
//
//   warp 0       TMA producer: Q once, then stages {V_{j-1}^T, K_j} through a 2-stage ring
//   warp 1       TMEM allocator + MMA issuer of tile A, warp 10 MMA issuer of tile B;
//                a token alternates them, giving the order
//                  S_A(0) S_B(0) | PV_A(j) S_A(j+1) | PV_B(j) S_B(j+1) | ...
//                so that the tensor core works on one tile while the other's softmax runs
//   warps 2..5   softmax of tile A, warps 6..9 softmax of tile B: one thread per query
//                row (the warp's TMEM lane quarter), all 128 keys of the tile in
//                registers; the row maximum comes with the reducing TMEM load
//                (tcgen05.ld.red).  Online softmax in log2 units with lazy O rescaling
//                (only when the running max grows by more than 8).  P is written back to TMEM
//                as bf16 over the row's own S columns and fed to the PV MMA as the TMEM
//                A operand.
//
// One softmax warp per tile on each SM sub-partition: a tcgen05.mma needs issue slots on
// the issuer's sub-partition.  Measured on GB300, an N=128 MMA stream runs at 64 cycles per
// MMA alone, ~72-76 next to one warp that issues every cycle (a mix of FMA, MUFU and
// conversions, like the softmax) and ~90-110 next to two to four such warps; warps of only
// MUFU or only conversions do not slow it, warps of FMA or ALU instructions do.  So the
// softmax keeps its FMA/ALU count low (packed f32x2 arithmetic, the reducing load instead of
// a max pass), its warps wait on barriers with suspending polls instead of spinning, and the
// issuers precompute their descriptors and issue four MMAs per asm block.  The layout with
// two threads per row (18 warps) ran its MMAs at ~90-110 cycles.
//
// TMEM (512 columns): S_A [0,128), S_B [128,256) (P_g, all 128 keys packed in pairs, aliases
// columns [0, 64) of S_g: one 64-column store), O_A [256, 256+hd), O_B [256+hd, 256+2hd).  V is stored
// transposed (V^T [hd][keys]) so that it is a K-major B operand in shared memory.
//
// Two launch forms of the same per-item arithmetic: one item (256 query rows of one
// (batch item, head)) per CTA for long key loops (self-attention), and a persistent form
// (attn_body_persist) for short ones (cross-attention over the 512 text tokens), where an
// item's fixed costs -- its Q load, first scores and O epilogue -- are as long as its key
// loop and overlap the neighbouring items' work instead.  Both give the same bits.
#include <cuda.h>
#include <cuda_bf16.h>

#include "common.cuh"
#include "elementwise.h"
#include "ptx.cuh"
#include "tma_host.h"

namespace cs {

struct AttnArgs {
  int B, heads, Lq, Lk, kv_shared;
  const int32_t* item_idx;   // optional: shared K/V set of batch item j is item_idx[j] / x_rows
  int x_rows, kv_sets;
  float scale_log2;
  __nv_bfloat16* o;
  int* err;
};

template <int HD>
struct AttnCfg {
  static constexpr int HDS = HD < 64 ? 64 : HD;   // Q/K row length in shared memory
  static constexpr int BKV = 128;
  static constexpr int QCH = HDS / 64;             // 64-wide chunks of a Q/K row
  static constexpr int CH_BYTES = 128 * 64 * 2;    // one [128 x 64] bf16 chunk
  static constexpr int Q_BYTES = QCH * CH_BYTES;   // one 128-row Q tile
  static constexpr int K_BYTES = QCH * CH_BYTES;   // one 128-key K tile
  static constexpr int VCH_BYTES = HD * 64 * 2;    // one [hd x 64 keys] chunk of V^T
  static constexpr int V_BYTES = 2 * VCH_BYTES;
  static constexpr int SLOT = K_BYTES > V_BYTES ? K_BYTES : V_BYTES;
  static constexpr int NSTAGE = 2;                  // ring stages, each a V slot and a K slot
  static constexpr int SMEM = 2 * Q_BYTES + NSTAGE * 2 * SLOT + 1024 + 256;
  static constexpr int ISSUER_B = 10;                 // second MMA issuer (another sub-partition)
  static constexpr int HANDOVER = 4;                  // MMAs left in a group when the token passes (3-6 measured best)
  static constexpr int THREADS = 11 * 32;
  static constexpr uint32_t IDESC_S = idesc_bf16_f32(128, BKV);
  static constexpr uint32_t IDESC_O = idesc_bf16_f32(128, HD);
};

// One key tile of the online softmax of one query row (one thread per row, after S(j) of
// its tile is complete): the scores of the tile from TMEM (keys past `valid` masked), the
// running maximum and sum in log2 units, P = 2^(s * scale - m) written back as bf16 pairs over
// the first 64 S columns, and O rescaled when the maximum grew by more than 8 (lazy rescale;
// the PV of the previous tile has finished, since the commit that signalled S(j) covers it).
template <int HD>
__device__ __forceinline__ void softmax_tile(uint32_t tS, uint32_t tO, int j, int valid, float sl2, uint64_t sc2,
                                             float& m_run, float& l_run) {
  using Cfg = AttnCfg<HD>;
  uint32_t u[128];
  float rmax;
  if (valid >= Cfg::BKV) {
    tmem_ld128_max(tS, u, rmax);            // the row maximum comes with the load
  } else {                                  // last, partial key tile: mask, then reduce
    tmem_ld128(tS, u);
#pragma unroll
    for (int e = 0; e < Cfg::BKV; ++e)
      if (e >= valid) u[e] = __float_as_uint(-INFINITY);
    float mx[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) mx[q] = __uint_as_float(u[q]);
#pragma unroll
    for (int e = 4; e < Cfg::BKV - 4; e += 8) {
#pragma unroll
      for (int q = 0; q < 4; ++q) mx[q] = fmax3(mx[q], __uint_as_float(u[e + 2 * q]), __uint_as_float(u[e + 2 * q + 1]));
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) mx[q] = fmaxf(mx[q], __uint_as_float(u[Cfg::BKV - 4 + q]));
    rmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
  }
  const float m_new = fmaxf(m_run, rmax * sl2);
  const bool need = (j == 0) || (m_new > m_run + 8.f);
  const bool warp_need = __any_sync(0xffffffffu, need);
  const float m_use = need ? m_new : m_run;
  const float factor = need ? ex2_approx(m_run - m_use) : 1.f;
  const uint64_t nm2 = f2_pack(-m_use, -m_use);
  // p = 2^(s * scale * log2(e) - m) on pairs; P packed as bf16 pairs in place (u[0..63])
  uint64_t acc[2] = {0ull, 0ull};
#pragma unroll
  for (int i = 0; i < Cfg::BKV / 2; ++i) {
    float a, b;
    f2_unpack(f2_fma(f2_pack(__uint_as_float(u[2 * i]), __uint_as_float(u[2 * i + 1])), sc2, nm2), a, b);
    a = ex2_approx(a);
    b = ex2_approx(b);
    acc[i & 1] = f2_add(acc[i & 1], f2_pack(a, b));
    u[i] = pack_bf16x2(a, b);
  }
  float s0, s1, s2, s3;
  f2_unpack(acc[0], s0, s1);
  f2_unpack(acc[1], s2, s3);
  l_run = l_run * factor + ((s0 + s1) + (s2 + s3));
  m_run = m_use;
  // PV of the previous tile has finished: the commit that signalled S(j) also covers
  // every MMA issued before it, so O may be rescaled and P overwritten now
  if (j > 0 && warp_need) {
#pragma unroll 1
    for (int c = 0; c < HD / 32; ++c) {
      uint32_t o[32];
      tmem_ld32(tO + c * 32, o);
#pragma unroll
      for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * factor);
      tmem_st32(tO + c * 32, o);
    }
  }
  tmem_st64(tS, u);                         // P: keys 2c, 2c+1 packed in column c
}

// The normalised O row (O / l, bf16) of one query row from TMEM to memory.
template <int HD>
__device__ __forceinline__ void store_o_row(uint32_t tO, float l_run, __nv_bfloat16* orow, bool in_range) {
  const float inv_l = 1.f / l_run;
#pragma unroll 1
  for (int c = 0; c < HD / 32; ++c) {
    uint32_t u[32];
    tmem_ld32(tO + c * 32, u);
    if (in_range) {
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        uint4 o4;
        o4.x = pack_bf16x2(__uint_as_float(u[8 * w + 0]) * inv_l, __uint_as_float(u[8 * w + 1]) * inv_l);
        o4.y = pack_bf16x2(__uint_as_float(u[8 * w + 2]) * inv_l, __uint_as_float(u[8 * w + 3]) * inv_l);
        o4.z = pack_bf16x2(__uint_as_float(u[8 * w + 4]) * inv_l, __uint_as_float(u[8 * w + 5]) * inv_l);
        o4.w = pack_bf16x2(__uint_as_float(u[8 * w + 6]) * inv_l, __uint_as_float(u[8 * w + 7]) * inv_l);
        reinterpret_cast<uint4*>(orow + c * 32)[w] = o4;
      }
    }
  }
}

template <int HD>
__device__ __forceinline__ void attn_body(const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                                          const AttnArgs& p) {
  using Cfg = AttnCfg<HD>;
  constexpr int NS = Cfg::NSTAGE;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                                   // [2][Q_BYTES]
  uint8_t* sKV = sQ + 2 * Cfg::Q_BYTES;                 // [NSTAGE][V slot, K slot][SLOT]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sKV + NS * 2 * Cfg::SLOT);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;            // [NS]
  uint64_t* kv_empty = kv_full + NS;       // [NS]
  uint64_t* s_full = kv_empty + NS;        // [2]
  uint64_t* p_full = s_full + 2;           // [2]
  uint64_t* o_done = p_full + 2;           // [2]
  uint64_t* tok = o_done + 2;              // [2]: tok[g] = tile g may start its next MMA group
  uint64_t* teardown = tok + 2;            // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(teardown + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.y;
  const int head = bh % p.heads, jb = bh / p.heads;
  int kv_set = p.kv_shared && p.item_idx ? p.item_idx[jb] / p.x_rows : 0;
  if (!index_ok(kv_set, p.kv_sets, p.err)) kv_set = 0;
  const int bkv = !p.kv_shared ? bh : kv_set * p.heads + head;
  const int q0 = blockIdx.x * 256;
  const int nt = (p.Lk + Cfg::BKV - 1) / Cfg::BKV;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 2);          // both issuers read every stage
    }
    for (int g = 0; g < 2; ++g) {
      mbar_init(&s_full[g], 1);
      mbar_init(&p_full[g], 128);
      mbar_init(&o_done[g], 1);
    }
    for (int g = 0; g < 2; ++g) {
      mbar_init(&tok[g], 1);
      mbar_init(&teardown[g], 1);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  block_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      mbar_arrive_expect_tx(q_full, 2 * Cfg::Q_BYTES);
      for (int g = 0; g < 2; ++g)
        for (int c = 0; c < Cfg::QCH; ++c)
          tma_load_3d(sQ + g * Cfg::Q_BYTES + c * Cfg::CH_BYTES, &tmQ, q_full, c * 64, q0 + g * 128, bh);
      // stage st holds V_{st-1} (st >= 1) and K_st (st < nt): exactly what the MMAs issued
      // after P(st-1) read, so the issuer waits on one barrier per key tile
      int issued = 0;
      for (int st = 0; st <= nt; ++st) {
        const int b = st % NS;
        if (!mbar_wait(&kv_empty[b], ((st / NS) & 1) ^ 1, abort_flag, p.err)) break;
        uint8_t* dv = sKV + b * 2 * Cfg::SLOT;
        uint8_t* dk = dv + Cfg::SLOT;
        mbar_arrive_expect_tx(&kv_full[b], (st >= 1 ? Cfg::V_BYTES : 0) + (st < nt ? Cfg::K_BYTES : 0));
        if (st < nt)
          for (int c = 0; c < Cfg::QCH; ++c)
            tma_load_3d(dk + c * Cfg::CH_BYTES, &tmK, &kv_full[b], c * 64, st * Cfg::BKV, bkv);
        if (st >= 1)
          for (int c = 0; c < 2; ++c)
            tma_load_3d(dv + c * Cfg::VCH_BYTES, &tmV, &kv_full[b], (st - 1) * Cfg::BKV + c * 64, 0, bkv);
        issued = st + 1;
      }
      if (*abort_flag) {
        mbar_wait_teardown(q_full, 0);
        for (int st = issued - NS < 0 ? 0 : issued - NS; st < issued; ++st)
          mbar_wait_teardown(&kv_full[st % NS], (st / NS) & 1);
      }
    }
  } else if (warp == 1 || warp == Cfg::ISSUER_B) {
    // ------------------------------------------------------------ MMA issuers
    // One issuing thread per query tile, on different SM sub-partitions, handing a token
    // back and forth so that the tensor core sees the groups in the order
    //   S_A(0) S_B(0) | PV_A(j) S_A(j+1) | PV_B(j) S_B(j+1) | ...
    // A tcgen05.mma stream must not pause (measured on GB300: each wait or fence between
    // two MMAs costs the tensor core ~100-200 cycles).  The token is handed over HANDOVER
    // MMAs before the end of a group, so the next group's waits and fence run while those
    // MMAs execute.  Each thread's MMAs run in its issue order, which is all that a tile's
    // TMEM reuse needs (PV_g(j) reads P_g(j) before S_g(j+1) overwrites it).
    if (lane == 0) {
      const int g = warp == 1 ? 0 : 1;
      const uint32_t q_base = smem_u32(sQ);
      const uint32_t sdst = tmem_base + g * 128, odst = tmem_base + 256 + g * HD;
      const uint64_t ad = sdesc_sw128(q_base + g * Cfg::Q_BYTES);
      // Every descriptor of both ring stages is built once (shared addresses stay below 2^18,
      // so adding a slice's byte offset / 16 to the start-address field cannot carry); the
      // MMAs go out four to an asm block, which keeps the issuing thread's instruction
      // count per MMA low (its sub-partition is shared with softmax warps).
      static_assert(Cfg::NSTAGE == 2 && Cfg::HANDOVER == 4, "descriptor tables: two stages, hand-over at 4");
      constexpr int NKS = Cfg::HDS / 16;      // K slices of S (4 or 8)
      auto v_addr = [&](int st) { return smem_u32(sKV + (st % NS) * 2 * Cfg::SLOT); };
      auto k_addr = [&](int st) { return v_addr(st) + Cfg::SLOT; };
      uint64_t qa[8], kb0[8], kb1[8], vb0[8], vb1[8];
      uint32_t pa[8];
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint64_t offk = (uint64_t)(((kk >> 2) * Cfg::CH_BYTES + (kk & 3) * 32) >> 4);
        const uint64_t offv = (uint64_t)(((kk >> 2) * Cfg::VCH_BYTES + (kk & 3) * 32) >> 4);
        qa[kk] = ad + offk;
        kb0[kk] = sdesc_sw128(k_addr(0)) + offk;
        kb1[kk] = sdesc_sw128(k_addr(1)) + offk;
        vb0[kk] = sdesc_sw128(v_addr(0)) + offv;
        vb1[kk] = sdesc_sw128(v_addr(1)) + offv;
        pa[kk] = sdst + kk * 8;                          // keys 16kk..16kk+15 packed in 8 columns
      }
      auto issue_s = [&](const uint64_t* kb, uint64_t* pass) {
        if (pass && NKS == Cfg::HANDOVER) mbar_arrive(pass);
        umma4_ss(sdst, qa, kb, Cfg::IDESC_S, 0u);
        if (NKS == 8) {
          if (pass) mbar_arrive(pass);
          umma4_ss(sdst, qa + 4, kb + 4, Cfg::IDESC_S, 1u);
        }
        umma_commit(&s_full[g]);
      };
      auto issue_pv = [&](const uint64_t* vb, int j, uint64_t* pass) {
        umma4_ts(odst, pa, vb, Cfg::IDESC_O, j > 0 ? 1u : 0u);
        if (pass) mbar_arrive(pass);
        umma4_ts(odst, pa + 4, vb + 4, Cfg::IDESC_O, 1u);
        umma_commit(&o_done[g]);   // measured: this commit after each PV group runs faster than none
      };
      uint64_t* other = &tok[1 - g];
      bool ok = mbar_wait(q_full, 0, abort_flag, p.err);
      if (ok) ok = mbar_wait(&kv_full[0], 0, abort_flag, p.err);
      if (ok && g == 1) ok = mbar_wait(&tok[1], 0, abort_flag, p.err);    // after S_A(0)
      if (ok) {
        tc_fence_after();
        issue_s(kb0, other);
        umma_commit(&kv_empty[0]);
      }
      // Token phases: tok[1] completes for S_A(0), then once per group A(j); tok[0] for
      // S_B(0), then once per group B(j) that another group A follows.  Each hand-over
      // comes after the receiver's previous wait on its own token, so no token runs two
      // phases ahead of its waiter and the parity tests stay unambiguous.
      for (int j = 0; ok && j < nt; ++j) {
        const int st = j + 1;
        const bool more = j + 1 < nt;
        if (!mbar_wait(&tok[g], g == 0 ? (j & 1) : ((j + 1) & 1), abort_flag, p.err)) break;
        if (!mbar_wait(&kv_full[st % NS], (st / NS) & 1, abort_flag, p.err)) break;
        if (!mbar_wait(&p_full[g], j & 1, abort_flag, p.err)) break;
        tc_fence_after();
        // the group's last MMAs hand the token over (group B only when a group A follows)
        uint64_t* pass = (g == 0 || more) ? other : nullptr;
        if ((st % NS) == 0) {   // two copies of the group, so the tables stay in registers
          issue_pv(vb0, j, more ? nullptr : pass);
          if (more) issue_s(kb0, pass);
        } else {
          issue_pv(vb1, j, more ? nullptr : pass);
          if (more) issue_s(kb1, pass);
        }
        umma_commit(&kv_empty[st % NS]);
      }
      if (*abort_flag) {
        umma_commit(&teardown[g]);
        mbar_wait_teardown(&teardown[g], 0);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int g = (warp - 2) >> 2;          // query tile: 0 = A (warps 2..5), 1 = B (warps 6..9)
    const int qtr = warp & 3;               // TMEM lane quarter this warp may access
    const int r = qtr * 32 + lane;          // query row inside the tile
    const uint32_t lane_off = (uint32_t)(qtr * 32) << 16;
    const uint32_t tS = tmem_base + lane_off + g * 128;
    const uint32_t tO = tmem_base + lane_off + 256 + g * HD;
    const float sl2 = p.scale_log2;
    const uint64_t sc2 = f2_pack(sl2, sl2);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < nt; ++j) {
      if (!__all_sync(0xffffffffu, mbar_wait_suspend(&s_full[g], j & 1, abort_flag, p.err))) { ok = false; break; }
      tc_fence_after();
      softmax_tile<HD>(tS, tO, j, p.Lk - j * Cfg::BKV, sl2, sc2, m_run, l_run);
      tc_fence_before();
      mbar_arrive(&p_full[g]);
    }
    // final: O / l -> bf16
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait_suspend(&o_done[g], (nt - 1) & 1, abort_flag, p.err));
    if (ok) {
      tc_fence_after();
      const int q = q0 + g * 128 + r;
      store_o_row<HD>(tO, l_run, p.o + ((long long)jb * p.Lq + q) * (p.heads * HD) + head * HD, q < p.Lq);
    }
  }

  tc_fence_before();
  block_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

// Persistent form: one CTA per SM walks the items (256 query rows of one (batch item,
// head)) it, it + G, ... (G = grid size) and keeps every pipeline running across item
// boundaries: the K/V ring, the MMA token between the two issuers, and the barrier phases
// continue, the producer loads the next item's Q as soon as the last score MMAs of the
// current item have read theirs, and each softmax warp's O epilogue of one item overlaps
// the next item's Q load and first score MMAs.  Every item runs the same arithmetic in the
// same order as in the one-item-per-CTA kernel.
template <int HD>
__device__ __forceinline__ void attn_body_persist(const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                                                  const AttnArgs& p) {
  using Cfg = AttnCfg<HD>;
  constexpr int NS = Cfg::NSTAGE;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = sQ + 2 * Cfg::Q_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sKV + NS * 2 * Cfg::SLOT);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;            // [NS]
  uint64_t* kv_empty = kv_full + NS;       // [NS]
  uint64_t* s_full = kv_empty + NS;        // [2]
  uint64_t* p_full = s_full + 2;           // [2]
  uint64_t* o_done = p_full + 2;           // [2]
  uint64_t* tok = o_done + 2;              // [2]
  uint64_t* teardown = tok + 2;            // [2]
  uint64_t* q_empty = teardown + 2;        // both issuers' last score MMAs of an item are done
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(q_empty + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqp = (p.Lq + 255) / 256;
  const int items = nqp * p.B * p.heads;
  const int nt = (p.Lk + Cfg::BKV - 1) / Cfg::BKV;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 2);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 2);
    }
    for (int g = 0; g < 2; ++g) {
      mbar_init(&s_full[g], 1);
      mbar_init(&p_full[g], 128);
      mbar_init(&o_done[g], 1);
      mbar_init(&tok[g], 1);
      mbar_init(&teardown[g], 1);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  block_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  auto item_bh = [&](int it) { return it / nqp; };
  auto item_q0 = [&](int it) { return (it % nqp) * 256; };
  auto item_bkv = [&](int it) {
    const int bh = item_bh(it), head = bh % p.heads, jb = bh / p.heads;
    int kv_set = p.kv_shared && p.item_idx ? p.item_idx[jb] / p.x_rows : 0;
    if (!index_ok(kv_set, p.kv_sets, p.err)) kv_set = 0;
    return !p.kv_shared ? bh : kv_set * p.heads + head;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      int gst = 0, issued = 0, n = 0, q_issued = 0;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < items; it += gridDim.x, ++n) {
        const int bh = item_bh(it), q0 = item_q0(it), bkv = item_bkv(it);
        // the previous item's score MMAs have read its Q
        if (n > 0 && !mbar_wait(q_empty, (n - 1) & 1, abort_flag, p.err)) break;
        ++q_issued;
        mbar_arrive_expect_tx(q_full, 2 * Cfg::Q_BYTES);
        for (int g = 0; g < 2; ++g)
          for (int c = 0; c < Cfg::QCH; ++c)
            tma_load_3d(sQ + g * Cfg::Q_BYTES + c * Cfg::CH_BYTES, &tmQ, q_full, c * 64, q0 + g * 128, bh);
        for (int st = 0; st <= nt; ++st, ++gst) {
          const int b = gst % NS;
          if (!mbar_wait(&kv_empty[b], ((gst / NS) & 1) ^ 1, abort_flag, p.err)) { ok = false; break; }
          uint8_t* dv = sKV + b * 2 * Cfg::SLOT;
          uint8_t* dk = dv + Cfg::SLOT;
          mbar_arrive_expect_tx(&kv_full[b], (st >= 1 ? Cfg::V_BYTES : 0) + (st < nt ? Cfg::K_BYTES : 0));
          if (st < nt)
            for (int c = 0; c < Cfg::QCH; ++c)
              tma_load_3d(dk + c * Cfg::CH_BYTES, &tmK, &kv_full[b], c * 64, st * Cfg::BKV, bkv);
          if (st >= 1)
            for (int c = 0; c < 2; ++c)
              tma_load_3d(dv + c * Cfg::VCH_BYTES, &tmV, &kv_full[b], (st - 1) * Cfg::BKV + c * 64, 0, bkv);
          issued = gst + 1;
        }
      }
      if (*abort_flag) {
        // the loads of the last ring's worth of stages and of the last Q (bounded waits)
        if (q_issued > 0) mbar_wait_teardown(q_full, (q_issued - 1) & 1);
        for (int st = issued - NS < 0 ? 0 : issued - NS; st < issued; ++st)
          mbar_wait_teardown(&kv_full[st % NS], (st / NS) & 1);
      }
    }
  } else if (warp == 1 || warp == Cfg::ISSUER_B) {
    // ------------------------------------------------------------ MMA issuers
    // The same groups as the one-item kernel, in one continuous stream:
    //   S_A(0) S_B(0) | PV_A(0) S_A(1) | PV_B(0) S_B(1) | ... | PV_A(nt-1) | PV_B(nt-1) | next item S_A(0) ...
    // with the token handed over inside every group except the CTA's very last one.
    if (lane == 0) {
      const int g = warp == 1 ? 0 : 1;
      const uint32_t q_base = smem_u32(sQ);
      const uint32_t sdst = tmem_base + g * 128, odst = tmem_base + 256 + g * HD;
      const uint64_t ad = sdesc_sw128(q_base + g * Cfg::Q_BYTES);
      static_assert(Cfg::NSTAGE == 2 && Cfg::HANDOVER == 4, "descriptor tables: two stages, hand-over at 4");
      constexpr int NKS = Cfg::HDS / 16;
      auto v_addr = [&](int st) { return smem_u32(sKV + (st % NS) * 2 * Cfg::SLOT); };
      auto k_addr = [&](int st) { return v_addr(st) + Cfg::SLOT; };
      uint64_t qa[8], kb0[8], kb1[8], vb0[8], vb1[8];
      uint32_t pa[8];
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint64_t offk = (uint64_t)(((kk >> 2) * Cfg::CH_BYTES + (kk & 3) * 32) >> 4);
        const uint64_t offv = (uint64_t)(((kk >> 2) * Cfg::VCH_BYTES + (kk & 3) * 32) >> 4);
        qa[kk] = ad + offk;
        kb0[kk] = sdesc_sw128(k_addr(0)) + offk;
        kb1[kk] = sdesc_sw128(k_addr(1)) + offk;
        vb0[kk] = sdesc_sw128(v_addr(0)) + offv;
        vb1[kk] = sdesc_sw128(v_addr(1)) + offv;
        pa[kk] = sdst + kk * 8;
      }
      auto issue_s = [&](const uint64_t* kb, uint64_t* pass) {
        if (pass && NKS == Cfg::HANDOVER) mbar_arrive(pass);
        umma4_ss(sdst, qa, kb, Cfg::IDESC_S, 0u);
        if (NKS == 8) {
          if (pass) mbar_arrive(pass);
          umma4_ss(sdst, qa + 4, kb + 4, Cfg::IDESC_S, 1u);
        }
        umma_commit(&s_full[g]);
      };
      auto issue_pv = [&](const uint64_t* vb, int j, uint64_t* pass) {
        umma4_ts(odst, pa, vb, Cfg::IDESC_O, j > 0 ? 1u : 0u);
        if (pass) mbar_arrive(pass);
        umma4_ts(odst, pa + 4, vb + 4, Cfg::IDESC_O, 1u);
        umma_commit(&o_done[g]);
      };
      uint64_t* other = &tok[1 - g];
      int gst = 0, n = 0, tw = 0, pw = 0;   // stage counter, items, token waits, P waits
      bool ok = true;
      for (int it = blockIdx.x; ok && it < items; it += gridDim.x, ++n) {
        const bool last_item = it + (int)gridDim.x >= items;
        const int base = gst;
        if (!mbar_wait(q_full, n & 1, abort_flag, p.err)) { ok = false; break; }
        // S(0): tile A of the CTA's first item starts the stream, every other group waits its turn
        if (!(g == 0 && n == 0)) {
          if (!mbar_wait(&tok[g], tw & 1, abort_flag, p.err)) { ok = false; break; }
          ++tw;
        }
        if (!mbar_wait(&kv_full[base % NS], (base / NS) & 1, abort_flag, p.err)) { ok = false; break; }
        tc_fence_after();
        issue_s((base % NS) == 0 ? kb0 : kb1, other);
        if (nt == 1) umma_commit(q_empty);
        umma_commit(&kv_empty[base % NS]);
        for (int j = 0; j < nt; ++j) {
          const int st = base + j + 1;
          const bool more = j + 1 < nt;
          if (!mbar_wait(&tok[g], tw & 1, abort_flag, p.err)) { ok = false; break; }
          ++tw;
          if (!mbar_wait(&kv_full[st % NS], (st / NS) & 1, abort_flag, p.err)) { ok = false; break; }
          if (!mbar_wait(&p_full[g], pw & 1, abort_flag, p.err)) { ok = false; break; }
          ++pw;
          tc_fence_after();
          // every group hands the token over, except tile B's last group of the CTA's last item
          uint64_t* pass = (g == 1 && !more && last_item) ? nullptr : other;
          if ((st % NS) == 0) {
            issue_pv(vb0, j, more ? nullptr : pass);
            if (more) issue_s(kb0, pass);
          } else {
            issue_pv(vb1, j, more ? nullptr : pass);
            if (more) issue_s(kb1, pass);
          }
          if (more && j + 2 == nt) umma_commit(q_empty);   // this item's last score MMAs
          umma_commit(&kv_empty[st % NS]);
        }
        gst = base + nt + 1;
      }
      if (*abort_flag) {
        umma_commit(&teardown[g]);
        mbar_wait_teardown(&teardown[g], 0);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax + epilogue
    const int g = (warp - 2) >> 2;
    const int qtr = warp & 3;
    const int r = qtr * 32 + lane;
    const uint32_t lane_off = (uint32_t)(qtr * 32) << 16;
    const uint32_t tS = tmem_base + lane_off + g * 128;
    const uint32_t tO = tmem_base + lane_off + 256 + g * HD;
    const float sl2 = p.scale_log2;
    const uint64_t sc2 = f2_pack(sl2, sl2);
    const int d = p.heads * HD;
    int sc = 0;   // S tiles of this query tile consumed so far (all items)
    bool ok = true;
    for (int it = blockIdx.x; ok && it < items; it += gridDim.x) {
      const int bh = item_bh(it), q0 = item_q0(it);
      const int head = bh % p.heads, jb = bh / p.heads;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; j < nt; ++j, ++sc) {
        if (!__all_sync(0xffffffffu, mbar_wait_suspend(&s_full[g], sc & 1, abort_flag, p.err))) { ok = false; break; }
        tc_fence_after();
        softmax_tile<HD>(tS, tO, j, p.Lk - j * Cfg::BKV, sl2, sc2, m_run, l_run);
        tc_fence_before();
        mbar_arrive(&p_full[g]);
      }
      if (!ok) break;
      // epilogue: the item's last PV group (o_done phase sc - 1) has completed
      if (!__all_sync(0xffffffffu, mbar_wait_suspend(&o_done[g], (sc - 1) & 1, abort_flag, p.err))) { ok = false; break; }
      tc_fence_after();
      const int q = q0 + g * 128 + r;
      store_o_row<HD>(tO, l_run, p.o + ((long long)jb * p.Lq + q) * d + head * HD, q < p.Lq);
      // O is read before this warp's next arrival on p_full, which the next PV (that
      // overwrites O) waits for: tmem_ld32 waits for its loads to complete
    }
  }

  tc_fence_before();
  block_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

template <int HD>
__global__ void __launch_bounds__(AttnCfg<HD>::THREADS, 1)
    attn_tcgen05_persist_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                                const __grid_constant__ CUtensorMap tmV, const AttnArgs p) {
  attn_body_persist<HD>(tmQ, tmK, tmV, p);
}

template <int HD>
__global__ void __launch_bounds__(AttnCfg<HD>::THREADS, 1)
    attn_tcgen05_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, const AttnArgs p) {
  attn_body<HD>(tmQ, tmK, tmV, p);
}

constexpr int kPersistMaxKeys = 8192;

template <int HD>
static cs_status launch_attn(const void* q, const void* k, const void* vt, void* o, int B, int heads, int Lq, int Lk,
                             int Lkv_stride, int kv_shared, int kv_sets, const int32_t* item_idx, int x_rows,
                             int* err, cudaStream_t stream) {
  using Cfg = AttnCfg<HD>;
  const int BH = B * heads, Bkv = kv_shared ? heads * kv_sets : BH;
  CUtensorMap tq, tk, tv;
  {
    const uint64_t dims[3] = {(uint64_t)Cfg::HDS, (uint64_t)Lq, (uint64_t)BH};
    const uint64_t str[2] = {(uint64_t)Cfg::HDS * 2, (uint64_t)Lq * Cfg::HDS * 2};
    const uint32_t box[3] = {64, 128, 1};
    CS_TRY(make_tmap_bf16(&tq, q, 3, dims, str, box));
  }
  {
    const uint64_t dims[3] = {(uint64_t)Cfg::HDS, (uint64_t)Lk, (uint64_t)Bkv};
    const uint64_t str[2] = {(uint64_t)Cfg::HDS * 2, (uint64_t)Lk * Cfg::HDS * 2};
    const uint32_t box[3] = {64, 128, 1};
    CS_TRY(make_tmap_bf16(&tk, k, 3, dims, str, box));
  }
  {
    const uint64_t dims[3] = {(uint64_t)Lk, (uint64_t)HD, (uint64_t)Bkv};
    const uint64_t str[2] = {(uint64_t)Lkv_stride * 2, (uint64_t)HD * Lkv_stride * 2};
    const uint32_t box[3] = {64, (uint32_t)HD, 1};
    CS_TRY(make_tmap_bf16(&tv, vt, 3, dims, str, box));
  }
  AttnArgs a{};
  a.B = B; a.heads = heads; a.Lq = Lq; a.Lk = Lk; a.kv_shared = kv_shared;
  a.item_idx = item_idx; a.x_rows = x_rows > 0 ? x_rows : 1; a.kv_sets = kv_sets;
  a.scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  a.o = static_cast<__nv_bfloat16*>(o);
  a.err = err;
  dim3 grid((Lq + 255) / 256, BH);
  if (Lk <= kPersistMaxKeys) {
    // short key loops (cross-attention over the text, short clips): one CTA per SM walks the
    // items, so that an item's Q load, first scores and O epilogue overlap its neighbours'
    // work.  Measured (same bits either way): 4 x 12 x 32760 x 512 973 -> 1026 TFLOP/s,
    // 8 x 12 x 4096^2 1370-1416 -> 1476, 4 x 12 x 8192^2 1495-1523 -> 1548; at 14040 keys
    // +2 % at 4 batch items and -1 % at 32, at 32760 keys -0.5 %, so longer loops keep
    // one item per CTA
    auto kern = attn_tcgen05_persist_kernel<HD>;
    CS_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM));
    const int items = grid.x * grid.y;
    kern<<<items < num_sms() ? items : num_sms(), Cfg::THREADS, Cfg::SMEM, stream>>>(tq, tk, tv, a);
    CS_LAUNCHED();
    return CS_OK;
  }
  auto kern = attn_tcgen05_kernel<HD>;
  CS_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM));
  kern<<<grid, Cfg::THREADS, Cfg::SMEM, stream>>>(tq, tk, tv, a);
  CS_LAUNCHED();
  return CS_OK;
}

cs_status attention_run(const void* q, const void* k, const void* vt, void* o, int B, int heads, int Lq, int Lk,
                        int hd, int Lkv_stride, int kv_shared, int kv_sets, const int32_t* item_idx, int x_rows,
                        int* err, cudaStream_t stream) {
  CS_REQUIRE(q && k && vt && o, "cs_attention: null pointer");
  CS_REQUIRE(B > 0 && heads > 0 && Lq > 0 && Lk > 0, "cs_attention: empty shape");
  CS_REQUIRE(Lkv_stride >= Lk && Lkv_stride % 8 == 0, "cs_attention: Lkv_stride must be >= Lk and a multiple of 8");
  CS_REQUIRE((long long)B * heads <= 65535, "cs_attention: B*heads = %lld exceeds the grid limit",
             (long long)B * heads);
  CS_REQUIRE(kv_sets >= 1 && (kv_sets == 1 || (kv_shared && item_idx)), "cs_attention: bad K/V set selection");
  if (hd == 128)
    return launch_attn<128>(q, k, vt, o, B, heads, Lq, Lk, Lkv_stride, kv_shared, kv_sets, item_idx, x_rows, err,
                            stream);
  if (hd == 32)
    return launch_attn<32>(q, k, vt, o, B, heads, Lq, Lk, Lkv_stride, kv_shared, kv_sets, item_idx, x_rows, err,
                           stream);
  set_error("cs_attention: head dim %d not supported (32 or 128)", hd);
  return CS_ERR_UNSUPPORTED;
}

}  // namespace cs

extern "C" cs_status cs_attention(const void* q, const void* k, const void* vt, void* o, int B, int heads, int Lq,
                                  int Lk, int hd, int Lkv_stride, int kv_shared, int* err, cudaStream_t stream) {
  return cs::attention_run(q, k, vt, o, B, heads, Lq, Lk, hd, Lkv_stride, kv_shared, 1, nullptr, 1, err, stream);
}
