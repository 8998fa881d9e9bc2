// The model object and the step-level C ABI: weight storage, the prompt's text K/V,
// the DiT forward of a compacted candidate subset, and cs_search_step, which runs
//   cache decide (Eq. indicator) -> DiT on the computing candidates -> cache apply
//   (Eq. delta / Eq. skip / Eq. euler, optional x0-estimate score)
// on one stream.  All arithmetic runs in this library's kernels.
#include <cmath>
#include <algorithm>
#include <cstring>
#include <vector>

#include <cuda_bf16.h>

#include "common.cuh"
#include "elementwise.h"

using bf16 = __nv_bfloat16;

namespace {

constexpr int kClasses = 5;   // 0 self-attn, 1 cross-attn, 2 GEMM, 3 cache, 4 other

struct Timing {
  long long launches = 0;
  double ms = 0.0, work = 0.0;
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending;
  std::vector<double> pending_work;
};

struct BlockW {
  bf16 *qkv_w, *o_w, *cq_w, *ckv_w, *co_w, *ff1_w, *ff2_w;
  float *mod_off, *qkv_b, *o_b, *cq_b, *ckv_b, *co_b, *ff1_b, *ff2_b;
};

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

struct cs_model {
  cs_model_config cfg;
  int hd, hd_s, P, Kp, L, Lv, Ltv;
  long long D;
  int device;
  // weights (one allocation)
  void* wmem = nullptr;
  bf16 *patch_w, *head_w, *text_w1, *text_w2, *time_w1, *time_w2, *mod_w, *head_mod_w;
  float *patch_b, *time_b1, *time_b2, *mod_b, *text_b1, *text_b2, *head_mod_b, *head_b;
  std::vector<BlockW> blk;
  float** mod_offs_dev = nullptr;
  // text K/V (per block) and its scratch
  bf16 *ktext, *vttext, *txt1, *txt, *ctx_bf16;   // ktext [block][set][H][Lt][hd_s], vttext [block][set][H][hd][Ltv]
  bool text_set = false, null_text_set = false;
  // workspace (one allocation)
  void* ws = nullptr;
  bf16 *tok, *hbuf, *obuf, *q, *k, *vt, *fbuf;
  float *resid, *hout, *cond_scratch, *mods, *hmod, *v, *x_host_stage;
  int32_t *idx, *n_compute;
  int32_t* idx_all;   // 0, 1, ..., max_batch - 1: the compaction list of an all-compute step
  unsigned* cache_counter;    // arrival counter of the decision pass (zero between steps)
  int32_t* cache_sidx;        // skipped candidates [max_batch] and their count
  float* tpart;       // score partials of computed candidates per token row [max_batch][F*H/2]
  bool tokens_update = false;   // computed update straight from the head's token output
  // carried drift (token-layout update only): per candidate slot, the drift sums of the
  // latent the last step left, and which state buffers and step they belong to
  void* carry_ws = nullptr;
  cs::CarryState carry{};
  struct {
    const void *x = nullptr, *x_ref = nullptr, *delta = nullptr, *accum = nullptr, *has_ref = nullptr;
    int N = 0, k = 0;
    bool valid = false;
  } carry_tag;
  uint8_t* skip_tmp;
  void* cache_ws;
  int* err;
  int32_t* n_host = nullptr;   // pinned
  // profiling
  bool profiling = false;
  Timing timing[kClasses];
};

namespace {

cs_status record_begin(cs_model* m, int cls, cudaStream_t s, cudaEvent_t* ev) {
  if (!m->profiling) return CS_OK;
  CS_CUDA(cudaEventCreate(&ev[0]));
  CS_CUDA(cudaEventCreate(&ev[1]));
  CS_CUDA(cudaEventRecord(ev[0], s));
  (void)cls;
  return CS_OK;
}

cs_status record_end(cs_model* m, int cls, cudaStream_t s, cudaEvent_t* ev, double work) {
  if (!m->profiling) return CS_OK;
  CS_CUDA(cudaEventRecord(ev[1], s));
  m->timing[cls].pending.emplace_back(ev[0], ev[1]);
  m->timing[cls].pending_work.push_back(work);
  return CS_OK;
}

// Work of a class that launched nothing more: added to its last timed region.
cs_status add_work(cs_model* m, int cls, double work) {
  if (!m->profiling) return CS_OK;
  Timing& t = m->timing[cls];
  if (!t.pending_work.empty()) t.pending_work.back() += work;
  else t.work += work;
  return CS_OK;
}

cs_status fold_timing(cs_model* m) {
  for (int c = 0; c < kClasses; ++c) {
    Timing& t = m->timing[c];
    for (size_t i = 0; i < t.pending.size(); ++i) {
      float ms = 0.f;
      CS_CUDA(cudaEventSynchronize(t.pending[i].second));
      CS_CUDA(cudaEventElapsedTime(&ms, t.pending[i].first, t.pending[i].second));
      t.ms += ms;
      t.work += t.pending_work[i];
      t.launches += 1;
      cudaEventDestroy(t.pending[i].first);
      cudaEventDestroy(t.pending[i].second);
    }
    t.pending.clear();
    t.pending_work.clear();
  }
  return CS_OK;
}

cs_status gemm(cs_model* m, const void* A, const void* B, int epi, const float* bias, const float* gate, void* out,
               int ldo, int M, int N, int K, cudaStream_t s) {
  cudaEvent_t ev[2];
  CS_TRY(record_begin(m, 2, s, ev));
  CS_TRY(cs_gemm_bf16(A, B, M, N, K, epi, bias, gate, out, ldo, m->err, s));
  return record_end(m, 2, s, ev, 2.0 * M * N * K);
}

cs_status gemm_qkv(cs_model* m, const void* A, const void* B, int M, int N, int K, const float* bias, int L,
                   int which_base, void* q, void* k, void* vt, int Lv, cudaStream_t s) {
  cudaEvent_t ev[2];
  CS_TRY(record_begin(m, 2, s, ev));
  CS_TRY(cs_gemm_qkv(A, B, M, N, K, bias, L, m->cfg.d, m->cfg.heads, which_base, q, k, vt, Lv, m->err, s));
  return record_end(m, 2, s, ev, 2.0 * M * N * K);
}

cs_status attention(cs_model* m, int cls, const void* q, const void* k, const void* vt, void* o, int B, int Lq,
                    int Lk, int Lkv_stride, int kv_shared, cudaStream_t s) {
  cudaEvent_t ev[2];
  CS_TRY(record_begin(m, cls, s, ev));
  CS_TRY(cs_attention(q, k, vt, o, B, m->cfg.heads, Lq, Lk, m->hd, Lkv_stride, kv_shared, m->err, s));
  return record_end(m, cls, s, ev, 4.0 * B * m->cfg.heads * (double)Lq * Lk * m->hd);
}

cs_status cross_attention(cs_model* m, const void* q, const void* k, const void* vt, void* o, int B, int Lq, int Lk,
                          int Lkv_stride, int kv_sets, const int32_t* idx, int x_rows, cudaStream_t s) {
  cudaEvent_t ev[2];
  CS_TRY(record_begin(m, 1, s, ev));
  CS_TRY(cs::attention_run(q, k, vt, o, B, m->cfg.heads, Lq, Lk, m->hd, Lkv_stride, 1, kv_sets,
                           kv_sets > 1 ? idx : nullptr, x_rows, m->err, s));
  return record_end(m, 1, s, ev, 4.0 * B * m->cfg.heads * (double)Lq * Lk * m->hd);
}

bool valid_cfg(const cs_model_config* c) {
  if (!c) return false;
  if (c->C <= 0 || c->F <= 0 || c->H <= 0 || c->W <= 0 || (c->H & 1) || (c->W & 1)) return false;
  if (c->d <= 0 || c->heads <= 0 || c->d % c->heads || c->ffn <= 0 || c->blocks <= 0) return false;
  if (c->f_dim <= 0 || (c->f_dim & 1) || c->d_text <= 0 || c->Lt <= 0 || c->max_batch <= 0) return false;
  return true;
}

}  // namespace

// One run of the search step's cache kernels (both decision-pass kernels, with and without
// scores, and the computed update) on scratch inside the residual-stream buffer, so that
// the first free step of a search does not pay their first launch (measured on GB300: the
// first decision pass of a process took ~25 us longer than the next one even with the
// kernels loaded).  Leaves the model's counter at zero and its error word clear.
static cs_status warm_cache_kernels(cs_model* m) {
  const cs_model_config& c = m->cfg;
  if (!m->tokens_update) return CS_OK;
  const long long D = m->D;
  float* x = m->resid;                      // 3 latents + a target + small state, all scratch
  float* xr = x + D;
  float* dl = xr + D;
  float* y = dl + D;
  float* small = y + D;                     // accum, scores, tile partials
  uint8_t* bytes = reinterpret_cast<uint8_t*>(small + 8 + c.F * (c.H / 2));
  uint8_t* has_ref = bytes;
  uint8_t* skip = bytes + 16;
  if ((size_t)(4 * D + 64 + c.F * (c.H / 2)) > (size_t)c.max_batch * m->L * c.d) return CS_OK;   // too small to hold it
  CS_CUDA(cudaMemset(x, 0, (4 * D + 8 + c.F * (c.H / 2)) * sizeof(float) + 64));
  for (int score = 0; score < 2; ++score) {
    // a cached candidate far from a non-zero reference under an infinite threshold: a
    // finite drift, and the candidate skips (the skip update runs)
    CS_CUDA(cudaMemset(has_ref, 1, 1));
    CS_CUDA(cudaMemset(xr, 0x3f, D * sizeof(float)));
    CS_TRY(cs::decide_skip_run(x, xr, dl, small, has_ref, 1, D, 2, 3, 1.f, 0.5f, 1e30f, 0, 0, nullptr, skip, m->idx,
                               m->n_compute, score ? y : nullptr, m->cache_ws,
                               cs::StepScratch{m->cache_counter, m->cache_sidx}, m->err, 0));
    CS_TRY(cs::apply_tokens_run(x, xr, dl, small, has_ref, skip, m->hout, m->idx_all, 1, 1, c.C, c.F, c.H, c.W, 1.f,
                                0.5f, score ? y : nullptr, small + 1, reinterpret_cast<float*>(m->cache_ws) + 2 * ((D + 8191) / 8192),
                                small + 8, 1, m->err, 0));
  }
  // the carried form: the drift pass with the carrying skip update, the decision from the
  // carried drift, and the carrying computed update (slot 0 of the model's carry state;
  // the model's step uses a carried drift only after a step of its own wrote it)
  for (int score = 0; score < 2; ++score) {
    CS_CUDA(cudaMemset(has_ref, 1, 1));
    CS_TRY(cs::carry_decide_skip_run(x, xr, dl, small, has_ref, 1, 2, 4, 1.f, 0.75f, 1e30f, 0, 0, nullptr, skip,
                                     m->idx, m->n_compute, score ? y : nullptr, false, m->carry, m->err, 0));
    CS_TRY(cs::carry_decide_skip_run(x, xr, dl, small, has_ref, 1, 3, 4, 0.75f, 0.5f, 1e30f, 0, 0, nullptr, skip,
                                     m->idx, m->n_compute, score ? y : nullptr, true, m->carry, m->err, 0));
    CS_TRY(cs::carry_apply_tokens_run(x, xr, dl, small, has_ref, skip, m->hout, m->idx_all, 1, 1, c.C, c.F, c.H, c.W,
                                      4, 0.5f, 0.25f, score ? y : nullptr, small + 1, m->carry, 1, m->err, 0));
  }
  CS_CUDA(cudaDeviceSynchronize());
  CS_CUDA(cudaMemset(m->err, 0, sizeof(int)));
  return CS_OK;
}

extern "C" size_t cs_param_count(const cs_model_config* c) {
  if (!valid_cfg(c)) return 0;
  const size_t d = c->d, P = 4 * (size_t)c->C, F = c->ffn;
  size_t n = d * P + d + d * c->f_dim + d + d * d + d + 6 * d * d + 6 * d + d * c->d_text + d + d * d + d +
             2 * d * d + 2 * d + P * d + P;
  const size_t per = 6 * d + 3 * d * d + 3 * d + d * d + d + d * d + d + 2 * d * d + 2 * d + d * d + d + F * d + F +
                     d * F + d;
  return n + per * c->blocks;
}

extern "C" cs_status cs_init_model(const cs_model_config* cfg, cs_model** out) {
  CS_REQUIRE(out, "cs_init_model: out is NULL");
  *out = nullptr;
  CS_REQUIRE(valid_cfg(cfg), "cs_init_model: invalid configuration");
  const int hd = cfg->d / cfg->heads;
  if (hd != 32 && hd != 128) {
    cs::set_error("cs_init_model: head dim %d not supported (32 or 128)", hd);
    return CS_ERR_UNSUPPORTED;
  }
  CS_REQUIRE(cfg->d % 64 == 0 && cfg->ffn % 64 == 0 && cfg->d_text % 64 == 0,
             "cs_init_model: d, ffn and d_text must be multiples of 64");
  CS_REQUIRE(4 * cfg->C <= 256, "cs_init_model: 4*C = %d patch features exceed 256", 4 * cfg->C);
  cs_model* m = new cs_model();
  m->cfg = *cfg;
  m->hd = hd;
  m->hd_s = hd < 64 ? 64 : hd;
  m->P = 4 * cfg->C;
  m->Kp = (int)align_up(m->P, 64);
  m->L = cfg->F * (cfg->H / 2) * (cfg->W / 2);
  m->Lv = (int)align_up(m->L, 8);
  m->Ltv = (int)align_up(cfg->Lt, 8);
  m->D = (long long)cfg->C * cfg->F * cfg->H * cfg->W;
  cudaGetDevice(&m->device);
  const size_t d = cfg->d, F = cfg->ffn, P = m->P, nb = cfg->blocks;

  // ---- weights
  struct Item { void** dst; size_t bytes; };
  std::vector<Item> items;
  auto addb = [&](bf16** p, size_t n) { items.push_back({reinterpret_cast<void**>(p), n * sizeof(bf16)}); };
  auto addf = [&](float** p, size_t n) { items.push_back({reinterpret_cast<void**>(p), n * sizeof(float)}); };
  addb(&m->patch_w, d * m->Kp); addf(&m->patch_b, d);
  addb(&m->time_w1, d * cfg->f_dim); addf(&m->time_b1, d);
  addb(&m->time_w2, d * d); addf(&m->time_b2, d);
  addb(&m->mod_w, 6 * d * d); addf(&m->mod_b, 6 * d);
  addb(&m->text_w1, d * cfg->d_text); addf(&m->text_b1, d);
  addb(&m->text_w2, d * d); addf(&m->text_b2, d);
  addb(&m->head_mod_w, 2 * d * d); addf(&m->head_mod_b, 2 * d);
  addb(&m->head_w, P * d); addf(&m->head_b, P);
  m->blk.resize(nb);
  for (size_t b = 0; b < nb; ++b) {
    BlockW& w = m->blk[b];
    addf(&w.mod_off, 6 * d);
    addb(&w.qkv_w, 3 * d * d); addf(&w.qkv_b, 3 * d);
    addb(&w.o_w, d * d); addf(&w.o_b, d);
    addb(&w.cq_w, d * d); addf(&w.cq_b, d);
    addb(&w.ckv_w, 2 * d * d); addf(&w.ckv_b, 2 * d);
    addb(&w.co_w, d * d); addf(&w.co_b, d);
    addb(&w.ff1_w, F * d); addf(&w.ff1_b, F);
    addb(&w.ff2_w, d * F); addf(&w.ff2_b, d);
  }
  // text K/V cache + text scratch
  const size_t kt = 2 * nb * cfg->heads * (size_t)cfg->Lt * m->hd_s, vtt = 2 * nb * cfg->heads * (size_t)hd * m->Ltv;
  addb(&m->ktext, kt);
  addb(&m->vttext, vtt);
  addb(&m->txt1, (size_t)cfg->Lt * d);
  addb(&m->txt, (size_t)cfg->Lt * d);
  addb(&m->ctx_bf16, (size_t)cfg->Lt * cfg->d_text);
  size_t total = 0;
  for (auto& it : items) total = align_up(total, 256) + it.bytes;
  if (cudaMalloc(&m->wmem, total) != cudaSuccess) {
    cudaGetLastError();
    cs::set_error("cs_init_model: cannot allocate %zu bytes of weights", total);
    delete m;
    return CS_ERR_NOMEM;
  }
  size_t off = 0;
  for (auto& it : items) {
    off = align_up(off, 256);
    *it.dst = static_cast<char*>(m->wmem) + off;
    off += it.bytes;
  }
  cudaMemset(m->wmem, 0, total);   // also zeroes the Q/K head-dim padding of the text cache

  // ---- workspace
  const size_t R = (size_t)cfg->max_batch * m->L;   // token rows
  const size_t BH = (size_t)cfg->max_batch * cfg->heads;
  items.clear();
  addb(&m->tok, R * m->Kp);
  addb(&m->hbuf, R * d);
  addb(&m->obuf, R * d);
  addb(&m->q, BH * m->L * m->hd_s);
  addb(&m->k, BH * m->L * m->hd_s);
  addb(&m->vt, BH * hd * m->Lv);
  addb(&m->fbuf, R * F);
  addf(&m->resid, R * d);
  addf(&m->hout, R * P);
  addf(&m->cond_scratch, cfg->f_dim + 9 * d);
  addf(&m->mods, nb * 6 * d);
  addf(&m->hmod, 2 * d);
  addf(&m->v, (size_t)cfg->max_batch * m->D);
  addf(&m->x_host_stage, (size_t)cfg->max_batch * m->D);
  items.push_back({reinterpret_cast<void**>(&m->idx), (size_t)cfg->max_batch * 4});
  items.push_back({reinterpret_cast<void**>(&m->idx_all), (size_t)cfg->max_batch * 4});
  items.push_back({reinterpret_cast<void**>(&m->cache_counter), 4});
  items.push_back({reinterpret_cast<void**>(&m->cache_sidx), (size_t)(cfg->max_batch + 1) * 4});
  addf(&m->tpart, (size_t)cfg->max_batch * cfg->F * (cfg->H / 2));
  items.push_back({reinterpret_cast<void**>(&m->n_compute), 16});
  items.push_back({reinterpret_cast<void**>(&m->skip_tmp), (size_t)cfg->max_batch});
  items.push_back({&m->cache_ws, cs_cache_workspace_bytes(cfg->max_batch, m->D)});
  items.push_back({&m->carry_ws, cs::carry_state_bytes(cfg->max_batch, m->D, cfg->F * (cfg->H / 2))});
  items.push_back({reinterpret_cast<void**>(&m->err), 16});
  items.push_back({reinterpret_cast<void**>(&m->mod_offs_dev), nb * sizeof(float*)});
  total = 0;
  for (auto& it : items) total = align_up(total, 256) + it.bytes;
  if (cudaMalloc(&m->ws, total) != cudaSuccess) {
    cudaGetLastError();
    cs::set_error("cs_init_model: cannot allocate %zu bytes of workspace", total);
    cudaFree(m->wmem);
    delete m;
    return CS_ERR_NOMEM;
  }
  off = 0;
  for (auto& it : items) {
    off = align_up(off, 256);
    *it.dst = static_cast<char*>(m->ws) + off;
    off += it.bytes;
  }
  cudaMemset(m->ws, 0, total);   // Q/K head-dim padding and the cache step's counters start at zero
  std::vector<int32_t> iota(cfg->max_batch);
  for (int i = 0; i < cfg->max_batch; ++i) iota[i] = i;
  cudaMemcpy(m->idx_all, iota.data(), iota.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  m->tokens_update = cs::apply_tokens_supported(cfg->C, cfg->F, cfg->H, cfg->W);
  m->carry = cs::CarryState{m->carry_ws, cfg->max_batch, m->D, cfg->F * (cfg->H / 2)};
  if (cs::load_cache_kernels() != CS_OK || warm_cache_kernels(m) != CS_OK) {
    cudaFree(m->ws);
    cudaFree(m->wmem);
    delete m;
    return CS_ERR_CUDA;
  }
  std::vector<float*> offs(nb);
  for (size_t b = 0; b < nb; ++b) offs[b] = m->blk[b].mod_off;
  cudaMemcpy(m->mod_offs_dev, offs.data(), nb * sizeof(float*), cudaMemcpyHostToDevice);
  if (cudaMallocHost(&m->n_host, 64) != cudaSuccess) {
    cudaGetLastError();
    cs::set_error("cs_init_model: cannot allocate pinned host memory");
    cudaFree(m->ws);
    cudaFree(m->wmem);
    delete m;
    return CS_ERR_NOMEM;
  }
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cs::set_error("cs_init_model: %s", cudaGetErrorString(e));
    return CS_ERR_CUDA;
  }
  *out = m;
  return CS_OK;
}

extern "C" cs_status cs_destroy_model(cs_model* m) {
  if (!m) return CS_OK;
  cudaDeviceSynchronize();
  fold_timing(m);
  cudaFree(m->ws);
  cudaFree(m->wmem);
  cudaFreeHost(m->n_host);
  delete m;
  return CS_OK;
}

namespace {
// One parameter tensor of the flat layout: a bf16 GEMM weight (rows x cols, stored with
// row stride ld) or a float32 vector copied as is.
struct ParamSlot {
  bf16* w;
  float* f;
  size_t rows, cols, ld;
  size_t count() const { return w ? rows * cols : rows; }
};

std::vector<ParamSlot> param_slots(cs_model* m) {
  const cs_model_config& c = m->cfg;
  const size_t d = c.d, F = c.ffn, P = m->P;
  std::vector<ParamSlot> v;
  auto W = [&](bf16* p, size_t r, size_t cc, size_t ld) { v.push_back({p, nullptr, r, cc, ld}); };
  auto V = [&](float* p, size_t n) { v.push_back({nullptr, p, n, 1, 1}); };
  W(m->patch_w, d, P, m->Kp); V(m->patch_b, d);
  W(m->time_w1, d, c.f_dim, c.f_dim); V(m->time_b1, d);
  W(m->time_w2, d, d, d); V(m->time_b2, d);
  W(m->mod_w, 6 * d, d, d); V(m->mod_b, 6 * d);
  W(m->text_w1, d, c.d_text, c.d_text); V(m->text_b1, d);
  W(m->text_w2, d, d, d); V(m->text_b2, d);
  W(m->head_mod_w, 2 * d, d, d); V(m->head_mod_b, 2 * d);
  W(m->head_w, P, d, d); V(m->head_b, P);
  for (int b = 0; b < c.blocks; ++b) {
    BlockW& bw = m->blk[b];
    V(bw.mod_off, 6 * d);
    W(bw.qkv_w, 3 * d, d, d); V(bw.qkv_b, 3 * d);
    W(bw.o_w, d, d, d); V(bw.o_b, d);
    W(bw.cq_w, d, d, d); V(bw.cq_b, d);
    W(bw.ckv_w, 2 * d, d, d); V(bw.ckv_b, 2 * d);
    W(bw.co_w, d, d, d); V(bw.co_b, d);
    W(bw.ff1_w, F, d, d); V(bw.ff1_b, F);
    W(bw.ff2_w, d, F, F); V(bw.ff2_b, d);
  }
  return v;
}

// Device float32 source -> destination slot (conversion to bf16 with padding for weights).
cs_status store_slot(const ParamSlot& sl, const float* src_dev, cudaStream_t s) {
  if (sl.w) return cs::to_bf16_pad(src_dev, (long long)sl.rows, (int)sl.cols, (int)sl.ld, sl.w, s);
  CS_CUDA(cudaMemcpyAsync(sl.f, src_dev, sl.rows * sizeof(float), cudaMemcpyDeviceToDevice, s));
  return CS_OK;
}

cs_status load_slot(cs_model* m, const ParamSlot& sl, const float* src, int on_device, float* stage,
                    cudaStream_t s) {
  if (on_device) return store_slot(sl, src, s);
  if (!sl.w) {
    CS_CUDA(cudaMemcpyAsync(sl.f, src, sl.rows * sizeof(float), cudaMemcpyHostToDevice, s));
    return CS_OK;
  }
  CS_CUDA(cudaMemcpyAsync(stage, src, sl.count() * sizeof(float), cudaMemcpyHostToDevice, s));
  CS_TRY(store_slot(sl, stage, s));
  CS_CUDA(cudaStreamSynchronize(s));   // the staging buffer is reused by the next tensor
  (void)m;
  return CS_OK;
}
}  // namespace

extern "C" int cs_param_tensor_count(const cs_model_config* c) {
  if (!c) return 0;
  return 16 + 15 * c->blocks;
}

extern "C" cs_status cs_load_weights(cs_model* m, const float* params, size_t count, int on_device,
                                     cudaStream_t s) {
  CS_REQUIRE(m && params, "cs_load_weights: null pointer");
  const size_t want = cs_param_count(&m->cfg);
  CS_REQUIRE(count == want, "cs_load_weights: got %zu floats, the model has %zu", count, want);
  std::vector<ParamSlot> slots = param_slots(m);
  size_t biggest = 0;
  for (auto& sl : slots) biggest = std::max(biggest, sl.count());
  float* stage = nullptr;
  if (!on_device) CS_CUDA(cudaMalloc(&stage, biggest * sizeof(float)));
  size_t off = 0;
  cs_status st = CS_OK;
  for (auto& sl : slots) {
    st = load_slot(m, sl, params + off, on_device, stage, s);
    if (st != CS_OK) break;
    off += sl.count();
  }
  cudaError_t e = cudaStreamSynchronize(s);
  if (stage) cudaFree(stage);
  if (st != CS_OK) return st;
  if (e != cudaSuccess) {
    cs::set_error("cs_load_weights: %s", cudaGetErrorString(e));
    return CS_ERR_CUDA;
  }
  m->text_set = m->null_text_set = false;
  return CS_OK;
}

extern "C" cs_status cs_load_param(cs_model* m, int index, const float* data, size_t count, int on_device,
                                   cudaStream_t s) {
  CS_REQUIRE(m && data, "cs_load_param: null pointer");
  std::vector<ParamSlot> slots = param_slots(m);
  CS_REQUIRE(index >= 0 && index < (int)slots.size(), "cs_load_param: tensor index %d outside 0..%d", index,
             (int)slots.size() - 1);
  const ParamSlot& sl = slots[index];
  CS_REQUIRE(count == sl.count(), "cs_load_param: tensor %d has %zu floats, got %zu", index, sl.count(), count);
  float* stage = nullptr;
  if (!on_device && sl.w) CS_CUDA(cudaMalloc(&stage, count * sizeof(float)));
  cs_status st = load_slot(m, sl, data, on_device, stage, s);
  cudaError_t e = cudaStreamSynchronize(s);
  if (stage) cudaFree(stage);
  if (st != CS_OK) return st;
  if (e != cudaSuccess) {
    cs::set_error("cs_load_param: %s", cudaGetErrorString(e));
    return CS_ERR_CUDA;
  }
  m->text_set = m->null_text_set = false;
  return CS_OK;
}

// Project a text context into K/V set `set` of every block (0: the prompt, 1: the
// unconditional context of classifier-free guidance).
static cs_status project_text(cs_model* m, const float* ctx, int set, cudaStream_t s) {
  const cs_model_config& c = m->cfg;
  const int d = c.d;
  CS_TRY(cs::to_bf16_pad(ctx, c.Lt, c.d_text, c.d_text, m->ctx_bf16, s));
  // text = W2 GELU(W1 ctx + b1) + b2
  CS_TRY(gemm(m, m->ctx_bf16, m->text_w1, CS_EPI_GELU_BF16, m->text_b1, nullptr, m->txt1, d, c.Lt, d, c.d_text, s));
  CS_TRY(gemm(m, m->txt1, m->text_w2, CS_EPI_BF16, m->text_b2, nullptr, m->txt, d, c.Lt, d, d, s));
  const size_t kt = (size_t)c.heads * c.Lt * m->hd_s, vtt = (size_t)c.heads * m->hd * m->Ltv;
  for (int b = 0; b < c.blocks; ++b) {
    // per block: [K | V] = text W_ckv^T + b_ckv, laid out per head (K) and transposed (V)
    CS_TRY(gemm_qkv(m, m->txt, m->blk[b].ckv_w, c.Lt, 2 * d, d, m->blk[b].ckv_b, c.Lt, 1, nullptr,
                    m->ktext + (2 * b + set) * kt, m->vttext + (2 * b + set) * vtt, m->Ltv, s));
  }
  return CS_OK;
}

extern "C" cs_status cs_set_text_context(cs_model* m, const float* ctx, cudaStream_t s) {
  CS_REQUIRE(m && ctx, "cs_set_text_context: null pointer");
  CS_TRY(project_text(m, ctx, 0, s));
  m->text_set = true;
  return CS_OK;
}

extern "C" cs_status cs_set_null_text_context(cs_model* m, const float* ctx, cudaStream_t s) {
  CS_REQUIRE(m && ctx, "cs_set_null_text_context: null pointer");
  CS_TRY(project_text(m, ctx, 1, s));
  m->null_text_set = true;
  return CS_OK;
}

// DiT forward of items j < n_c: latent row idx[j] % x_rows, cross-attention K/V set
// idx[j] / x_rows (kv_sets = 2 for guidance), velocity written to v[idx[j]].
static cs_status dit_forward_impl(cs_model* m, const float* x, const int32_t* idx, int n_c, int x_rows, int kv_sets,
                                  float t, float* v, cudaStream_t s) {
  // v == nullptr: stop after the head Linear; the velocity rows stay in m->hout (token layout)
  if (n_c == 0) return CS_OK;
  const cs_model_config& c = m->cfg;
  const int d = c.d, L = m->L, M = n_c * L;
  // valid state indices, checked by builds with CS_DEBUG_CHECKS: the search steps name
  // states [0, x_rows * kv_sets); a caller of cs_dit_forward any non-negative row
  const long long idx_limit = x_rows == (1 << 30) ? (1ll << 62) : (long long)x_rows * kv_sets;
  cudaEvent_t ev[2];
  CS_TRY(record_begin(m, 4, s, ev));
  cs::CondWeights cw{d, c.f_dim, c.blocks, m->time_w1, m->time_w2, m->mod_w, m->head_mod_w,
                     m->time_b1, m->time_b2, m->mod_b, m->head_mod_b, m->mod_offs_dev};
  CS_TRY(cs::timestep_conditioning(cw, t, m->cond_scratch, m->mods, m->hmod, s));
  CS_TRY(cs::patchify(x, idx, n_c, x_rows, c.C, c.F, c.H, c.W, m->Kp, m->tok, idx_limit, m->err, s));
  CS_TRY(record_end(m, 4, s, ev, 0.0));
  CS_TRY(gemm(m, m->tok, m->patch_w, CS_EPI_F32, m->patch_b, nullptr, m->resid, d, M, d, m->Kp, s));
  const size_t kt = (size_t)c.heads * c.Lt * m->hd_s, vtt = (size_t)c.heads * m->hd * m->Ltv;
  for (int b = 0; b < c.blocks; ++b) {
    const BlockW& w = m->blk[b];
    const float* mod = m->mods + (size_t)b * 6 * d;   // shift1 scale1 gate1 shift2 scale2 gate2
    // h = LN(x)(1 + scale1) + shift1 ; x += gate1 * SA(h)
    CS_TRY(record_begin(m, 4, s, ev));
    CS_TRY(cs::layernorm_modulate(m->resid, mod + 0 * d, mod + 1 * d, m->hbuf, M, d, s));
    CS_TRY(record_end(m, 4, s, ev, 0.0));
    CS_TRY(gemm_qkv(m, m->hbuf, w.qkv_w, M, 3 * d, d, w.qkv_b, L, 0, m->q, m->k, m->vt, m->Lv, s));
    CS_TRY(attention(m, 0, m->q, m->k, m->vt, m->obuf, n_c, L, L, m->Lv, 0, s));
    CS_TRY(gemm(m, m->obuf, w.o_w, CS_EPI_RESID_F32, w.o_b, mod + 2 * d, m->resid, d, M, d, d, s));
    // x += CA(LN(x), text)
    CS_TRY(record_begin(m, 4, s, ev));
    CS_TRY(cs::layernorm_modulate(m->resid, nullptr, nullptr, m->hbuf, M, d, s));
    CS_TRY(record_end(m, 4, s, ev, 0.0));
    CS_TRY(gemm_qkv(m, m->hbuf, w.cq_w, M, d, d, w.cq_b, L, 0, m->q, nullptr, nullptr, m->Lv, s));
    CS_TRY(cross_attention(m, m->q, m->ktext + 2 * b * kt, m->vttext + 2 * b * vtt, m->obuf, n_c, L, c.Lt, m->Ltv,
                           kv_sets, idx, x_rows, s));
    CS_TRY(gemm(m, m->obuf, w.co_w, CS_EPI_RESID_F32, w.co_b, nullptr, m->resid, d, M, d, d, s));
    // h = LN(x)(1 + scale2) + shift2 ; x += gate2 * FFN(h)
    CS_TRY(record_begin(m, 4, s, ev));
    CS_TRY(cs::layernorm_modulate(m->resid, mod + 3 * d, mod + 4 * d, m->hbuf, M, d, s));
    CS_TRY(record_end(m, 4, s, ev, 0.0));
    CS_TRY(gemm(m, m->hbuf, w.ff1_w, CS_EPI_GELU_BF16, w.ff1_b, nullptr, m->fbuf, c.ffn, M, c.ffn, d, s));
    CS_TRY(gemm(m, m->fbuf, w.ff2_w, CS_EPI_RESID_F32, w.ff2_b, mod + 5 * d, m->resid, d, M, d, c.ffn, s));
  }
  // head: LN(x)(1 + scale) + shift -> Linear(d -> 4C) -> unpatchify into v[idx[j]]
  CS_TRY(record_begin(m, 4, s, ev));
  CS_TRY(cs::layernorm_modulate(m->resid, m->hmod, m->hmod + d, m->hbuf, M, d, s));
  CS_TRY(record_end(m, 4, s, ev, 0.0));
  CS_TRY(gemm(m, m->hbuf, m->head_w, CS_EPI_F32, m->head_b, nullptr, m->hout, m->P, M, m->P, d, s));
  if (!v) return CS_OK;
  CS_TRY(record_begin(m, 4, s, ev));
  CS_TRY(cs::unpatchify(m->hout, idx, n_c, c.C, c.F, c.H, c.W, v, idx_limit, m->err, s));
  CS_TRY(record_end(m, 4, s, ev, 0.0));
  return CS_OK;
}

extern "C" cs_status cs_dit_forward(cs_model* m, const float* x, const int32_t* idx, int n_c, float t, float* v,
                                    cudaStream_t s) {
  CS_REQUIRE(m && x && idx && v, "cs_dit_forward: null pointer");
  CS_REQUIRE(n_c >= 0 && n_c <= m->cfg.max_batch, "cs_dit_forward: n_c=%d outside 0..max_batch=%d", n_c,
             m->cfg.max_batch);
  CS_REQUIRE(m->text_set, "cs_dit_forward: call cs_set_text_context first");
  return dit_forward_impl(m, x, idx, n_c, 1 << 30, 1, t, v, s);
}

static cs_status step_impl(cs_model* m, float* x, float* x_ref, float* delta, float* accum, uint8_t* has_ref, int N,
                           int k, int T, float t_cur, float t_next, float tau, int K_w, int K_c,
                           const uint8_t* force, uint8_t* skip, const float* target, float* scores, int* n_out,
                           const void* tag_x, cudaStream_t s) {
  CS_REQUIRE(m && x && x_ref && delta && accum && has_ref && skip, "cs_search_step: null pointer");
  CS_REQUIRE(N > 0 && N <= m->cfg.max_batch, "cs_search_step: N=%d outside 1..max_batch=%d", N, m->cfg.max_batch);
  CS_REQUIRE(!target || scores, "cs_search_step: scoring needs scores");
  CS_REQUIRE(k >= 1 && k <= T, "cs_search_step: step %d outside 1..T=%d", k, T);
  const long long D = m->D;
  const cs_model_config& c = m->cfg;
  cudaEvent_t ev[2];
  const bool wf = k <= K_w || k > T - K_c;
  const bool tokens = m->tokens_update;
  // the drift sums the previous step left apply when that step ran on the same state
  // buffers and N and was step k - 1 (and each candidate's has_ref = 3 says they still
  // belong to its latent)
  auto& tag = m->carry_tag;
  const bool carry_ok = tokens && tag.valid && tag.x == tag_x && tag.x_ref == x_ref && tag.delta == delta &&
                        tag.accum == accum && tag.has_ref == has_ref && tag.N == N && tag.k + 1 == k;
  tag.valid = false;
  bool carried = false;   // decisions taken from carried drifts on a free step
  int n_c = N;
  const int32_t* idx = m->idx;
  auto read_decisions = [&]() -> cs_status {
    CS_CUDA(cudaMemcpyAsync(m->n_host, m->n_compute, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    CS_CUDA(cudaMemcpyAsync(m->n_host + 1, m->err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    CS_CUDA(cudaStreamSynchronize(s));
    if (m->n_host[1] != 0) {
      cs::set_error("cs_search_step: device error %d recorded before step %d", m->n_host[1], k);
      const int code = m->n_host[1];
      cudaMemsetAsync(m->err, 0, sizeof(int), s);
      return (cs_status)code;
    }
    return CS_OK;
  };
  if (tokens && wf && !force) {
    // warm-up / cool-down: every candidate computes and no drift is evaluated (Sec. 3.1);
    // the computed update below writes the state (a = 0, has_ref = 3, skip = 0)
    idx = m->idx_all;
  } else if (tokens) {
    // decisions + the update of skipped candidates; computed ones after the DiT
    CS_TRY(record_begin(m, 3, s, ev));
    CS_TRY(cs::carry_decide_skip_run(x, x_ref, delta, accum, has_ref, N, k, T, t_cur, t_next, tau, K_w, K_c, force,
                                     skip, m->idx, m->n_compute, target, carry_ok, m->carry, m->err, s));
    CS_TRY(record_end(m, 3, s, ev, 0.0));
    CS_TRY(read_decisions());
    carried = carry_ok && !wf;
    if (m->n_host[0] < 0) {
      // a cached candidate carries no drift (its state was written outside these calls):
      // nothing was changed; take the drift pass
      carried = false;
      CS_TRY(record_begin(m, 3, s, ev));
      CS_TRY(cs::carry_decide_skip_run(x, x_ref, delta, accum, has_ref, N, k, T, t_cur, t_next, tau, K_w, K_c, force,
                                       skip, m->idx, m->n_compute, target, false, m->carry, m->err, s));
      CS_TRY(record_end(m, 3, s, ev, 0.0));
      CS_TRY(read_decisions());
    }
    n_c = m->n_host[0];
  } else {
    CS_TRY(record_begin(m, 3, s, ev));
    CS_TRY(cs::decide_skip_run(x, x_ref, delta, accum, has_ref, N, D, k, T, t_cur, t_next, tau, K_w, K_c, force, skip,
                               m->idx, m->n_compute, target, m->cache_ws,
                               cs::StepScratch{m->cache_counter, m->cache_sidx}, m->err, s));
    CS_TRY(record_end(m, 3, s, ev, 0.0));
    CS_TRY(read_decisions());
    n_c = m->n_host[0];
  }
  if (n_out) *n_out = n_c;
  CS_TRY(dit_forward_impl(m, x, idx, n_c, N, 1, t_cur, tokens ? nullptr : m->v, s));
  // algorithmic bytes of indicator + update (each tensor read or written once):
  //   skipped: read x, x_ref, Delta, write x                                 16 D
  //   computed: read x, v, write x, Delta, x_ref                             20 D
  //   (+ read x_ref for the drift of a free step whose drift was not carried: 24 D)
  const double skipped = N - n_c;
  double bytes = skipped * 16.0 * D + n_c * ((wf || carried) ? 20.0 : 24.0) * D;
  if (target) bytes += 4.0 * D * N;
  if (n_c == 0 && !target) {
    // the decision pass did the whole update
    if (tokens) tag = {tag_x, x_ref, delta, accum, has_ref, N, k, true};
    return add_work(m, 3, bytes);
  }
  CS_TRY(record_begin(m, 3, s, ev));
  if (tokens) {
    CS_TRY(cs::carry_apply_tokens_run(x, x_ref, delta, accum, has_ref, skip, m->hout, idx, n_c, N, c.C, c.F, c.H, c.W,
                                      k, t_cur, t_next, target, scores, m->carry, N, m->err, s));
  } else {
    CS_TRY(cs_cache_apply_computed(x, x_ref, delta, m->v, skip, N, D, t_cur, t_next, target, scores, m->cache_ws, s));
  }
  CS_TRY(record_end(m, 3, s, ev, bytes));
  if (tokens) tag = {tag_x, x_ref, delta, accum, has_ref, N, k, true};
  return CS_OK;
}

extern "C" cs_status cs_search_step(cs_model* m, float* x, float* x_ref, float* delta, float* accum,
                                    uint8_t* has_ref, int N, int k, int T, float t_cur, float t_next, float tau,
                                    int K_w, int K_c, const uint8_t* force, uint8_t* skip, const float* target,
                                    float* scores, int* n_computed, cudaStream_t s) {
  return step_impl(m, x, x_ref, delta, accum, has_ref, N, k, T, t_cur, t_next, tau, K_w, K_c, force, skip, target,
                   scores, n_computed, x, s);
}

extern "C" cs_status cs_search_step_cfg(cs_model* m, float* x, float* x_ref, float* delta, float* accum,
                                        uint8_t* has_ref, int N, int k, int T, float t_cur, float t_next, float tau,
                                        int K_w, int K_c, float w, const uint8_t* force, uint8_t* skip,
                                        const float* target, float* scores, int* n_out, cudaStream_t s) {
  CS_REQUIRE(m && x && x_ref && delta && accum && has_ref && skip, "cs_search_step_cfg: null pointer");
  CS_REQUIRE(N > 0 && 2 * N <= m->cfg.max_batch, "cs_search_step_cfg: 2N=%d exceeds max_batch=%d", 2 * N,
             m->cfg.max_batch);
  CS_REQUIRE(m->text_set && m->null_text_set, "cs_search_step_cfg: set both text contexts first");
  CS_REQUIRE(!target || scores, "cs_search_step_cfg: scoring needs scores");
  m->carry_tag.valid = false;   // the guided step carries no drift
  const long long D = m->D;
  cudaEvent_t ev[2];
  const bool wf = k <= K_w || k > T - K_c;
  CS_TRY(record_begin(m, 3, s, ev));
  CS_TRY(cs_cache_decide_cfg(x, x_ref, accum, has_ref, N, D, k, T, tau, K_w, K_c, force, skip, m->idx, m->n_compute,
                             m->cache_ws, m->err, s));
  CS_TRY(record_end(m, 3, s, ev, 0.0));
  CS_CUDA(cudaMemcpyAsync(m->n_host, m->n_compute, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  CS_CUDA(cudaMemcpyAsync(m->n_host + 1, m->err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  CS_CUDA(cudaStreamSynchronize(s));
  const int n_c = m->n_host[0];
  if (m->n_host[1] != 0) {
    cs::set_error("cs_search_step_cfg: device error %d recorded before step %d", m->n_host[1], k);
    const int code = m->n_host[1];
    cudaMemsetAsync(m->err, 0, sizeof(int), s);
    return (cs_status)code;
  }
  if (n_out) *n_out = n_c;
  // branch items: state rows < N are conditional (K/V set 0), rows >= N unconditional (set 1)
  CS_TRY(dit_forward_impl(m, x, m->idx, n_c, N, 2, t_cur, m->v, s));
  CS_TRY(record_begin(m, 3, s, ev));
  CS_TRY(cs_cache_apply_cfg(x, x_ref, delta, m->v, skip, N, D, t_cur, t_next, w, target, scores, m->cache_ws, s));
  const double skipped = 2.0 * N - n_c;
  double bytes = 4.0 * D * N * 2 + skipped * 8.0 * D + n_c * (wf ? 12.0 : 16.0) * D;   // x in/out + per branch
  if (target) bytes += 4.0 * D * N;
  CS_TRY(record_end(m, 3, s, ev, bytes));
  return CS_OK;
}

extern "C" cs_status cs_search_step_host(cs_model* m, float* x_host, float* x_ref, float* delta, float* accum,
                                         uint8_t* has_ref, int N, int k, int T, float t_cur, float t_next, float tau,
                                         int K_w, int K_c, uint8_t* skip_host, int* n_computed, cudaStream_t s) {
  CS_REQUIRE(m && x_host && skip_host, "cs_search_step_host: null pointer");
  CS_REQUIRE(N > 0 && N <= m->cfg.max_batch, "cs_search_step_host: N outside 1..max_batch");
  const size_t bytes = (size_t)N * m->D * sizeof(float);
  CS_CUDA(cudaMemcpyAsync(m->x_host_stage, x_host, bytes, cudaMemcpyHostToDevice, s));
  CS_TRY(step_impl(m, m->x_host_stage, x_ref, delta, accum, has_ref, N, k, T, t_cur, t_next, tau, K_w, K_c, nullptr,
                   m->skip_tmp, nullptr, nullptr, n_computed, x_host, s));
  CS_CUDA(cudaMemcpyAsync(x_host, m->x_host_stage, bytes, cudaMemcpyDeviceToHost, s));
  CS_CUDA(cudaMemcpyAsync(skip_host, m->skip_tmp, N, cudaMemcpyDeviceToHost, s));
  CS_CUDA(cudaStreamSynchronize(s));
  return CS_OK;
}

extern "C" cs_status cs_device_error(cs_model* m, int* code, cudaStream_t s) {
  CS_REQUIRE(m && code, "cs_device_error: null pointer");
  CS_CUDA(cudaMemcpyAsync(m->n_host + 2, m->err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  CS_CUDA(cudaMemsetAsync(m->err, 0, sizeof(int32_t), s));
  CS_CUDA(cudaStreamSynchronize(s));
  *code = m->n_host[2];
  return CS_OK;
}

extern "C" cs_status cs_set_profiling(cs_model* m, int enable) {
  CS_REQUIRE(m, "cs_set_profiling: null model");
  m->profiling = enable != 0;
  return CS_OK;
}

extern "C" cs_status cs_kernel_stats(cs_model* m, int cls, long long* launches, double* total_ms, double* work) {
  CS_REQUIRE(m && cls >= 0 && cls < kClasses, "cs_kernel_stats: bad arguments");
  CS_TRY(fold_timing(m));
  if (launches) *launches = m->timing[cls].launches;
  if (total_ms) *total_ms = m->timing[cls].ms;
  if (work) *work = m->timing[cls].work;
  return CS_OK;
}

extern "C" cs_status cs_reset_kernel_stats(cs_model* m) {
  CS_REQUIRE(m, "cs_reset_kernel_stats: null model");
  CS_TRY(fold_timing(m));
  for (auto& t : m->timing) {
    t.launches = 0;
    t.ms = 0.0;
    t.work = 0.0;
  }
  return CS_OK;
}
