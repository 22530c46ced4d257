// Host side of libvp: argument checking, workspace ownership, launch planning
// and the extern "C" entry points declared in include/vp.h.
#include <cuda_runtime.h>
#include <cmath>
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <string>
#include <vector>

#include "vp.h"
#include "vp_internal.h"

struct vp_ctx {
  vp_config cfg;
  int device = 0;
  int num_sms = 0;
  vp::WsLayout lay;
  void* ws = nullptr;
  size_t ws_bytes = 0;
  float* z_ws = nullptr;
  float* split_st = nullptr;
  float* split_o = nullptr;
  float* gpart_o = nullptr;
  float* gpart_st = nullptr;
  float* mt_o = nullptr;
  float* mt_st = nullptr;
  float* hmax = nullptr;
  float diag_delta = 0.f;          // diagnostics (vp_set_diagnostics)
  int32_t* diag_n_act = nullptr;
  uint32_t* diag_bits = nullptr;
  int32_t score_path = VP_SCORE_AUTO;  // vp_set_score_path
  unsigned* tickets = nullptr;
  unsigned* err = nullptr;
  std::string last_error;
  std::vector<cudaEvent_t> tev;  // stage-timing events, 4 per slot
  int32_t tslots = 0;
  int64_t tcalls = 0;
  int32_t last_score_path = 0;  // vp_last_launch: score kernel and kernel count of the last call
  int32_t last_kernels = 0;
};

namespace {


constexpr int64_t kPpm = 1000000;
constexpr int kMaxVisual = 32768;  // score keys of one sequence fit in shared memory
constexpr int kMaxHeads = 128;
constexpr int kMaxGroup = 16;

vp_status fail(vp_ctx* ctx, vp_status st, const std::string& msg) {
  if (ctx) ctx->last_error = msg;
  else vp::context_free_error() = msg;
  return st;
}

vp_status cuda_fail(vp_ctx* ctx, const char* what, cudaError_t e) {
  return fail(ctx, VP_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }


// Largest K_t the budget yields for n visual tokens (K_t is non-decreasing in
// N_v in every mode, so the bound for max_visual covers every sequence).
int32_t max_kept(const vp_budget& bd, int32_t n) {
  if (n <= 0) return 0;
  switch (bd.mode) {
    case VP_DENSE:
    case VP_TOP_P: return n;
    case VP_FIXED_K: return bd.fixed_k < n ? (bd.fixed_k < 0 ? 0 : bd.fixed_k) : n;
    case VP_FIXED_RATIO: {
      int64_t k = ceil_div((int64_t)bd.ratio_ppm * n, kPpm);
      if (k < 1) k = 1;
      return (int32_t)(k < n ? k : n);
    }
    case VP_ADAPTIVE: {
      const int64_t k_lo = ceil_div((int64_t)bd.r_lo_ppm * n, kPpm);
      int64_t k_hi = (int64_t)bd.r_hi_ppm * n / kPpm;
      if (k_hi < k_lo) k_hi = k_lo;
      return (int32_t)(k_hi < n ? k_hi : n);
    }
    default: return -1;
  }
}

bool budget_ok(const vp_budget& bd, std::string* why) {
  if (bd.mode < VP_ADAPTIVE || bd.mode > VP_TOP_P) { *why = "budget.mode out of range"; return false; }
  if (!(bd.tau > 0.f) || !isfinite(bd.tau)) { *why = "budget.tau must be finite and > 0"; return false; }
  if (!(bd.scale >= 0.f) || !isfinite(bd.scale)) { *why = "budget.scale must be finite and >= 0"; return false; }
  if (bd.r_lo_ppm < 0 || bd.r_lo_ppm > kPpm || bd.r_hi_ppm < 0 || bd.r_hi_ppm > kPpm) {
    *why = "budget clamp ratios must lie in [0, 1000000] ppm"; return false;
  }
  if (bd.ratio_ppm < 0 || bd.ratio_ppm > kPpm) { *why = "budget.ratio_ppm must lie in [0, 1000000]"; return false; }
  if (bd.fixed_k < 0) { *why = "budget.fixed_k must be >= 0"; return false; }
  if (bd.granularity != 0 && bd.granularity != 1) { *why = "budget.granularity must be 0 or 1"; return false; }
  if (bd.mode == VP_TOP_P && bd.granularity != 0) { *why = "the top-p budget needs granularity 0"; return false; }
  return true;
}

bool kv_ok(const vp_ctx* ctx, const vp_kv* kv, const char* name, std::string* why) {
  const size_t esz = ctx->cfg.dtype == VP_BF16 ? 2 : 4;
  char buf[160];
  if (!kv || !kv->data) { snprintf(buf, sizeof buf, "%s: NULL cache", name); *why = buf; return false; }
  if (!aligned16(kv->data)) { snprintf(buf, sizeof buf, "%s: data must be 16-byte aligned", name); *why = buf; return false; }
  const int64_t strides[3] = {kv->stride_b, kv->stride_h, kv->stride_t};
  for (int64_t s : strides) {
    if (s < 0 || ((uint64_t)s * esz) % 16 != 0) {
      snprintf(buf, sizeof buf, "%s: strides must be >= 0 and multiples of 16 bytes", name); *why = buf; return false;
    }
  }
  if (ctx->cfg.paged) {
    if (!kv->block_table || kv->max_pages < 1 || kv->num_pages < 1) {
      snprintf(buf, sizeof buf, "%s: paged cache needs block_table, max_pages >= 1, num_pages >= 1", name);
      *why = buf; return false;
    }
  } else if (kv->block_table) {
    snprintf(buf, sizeof buf, "%s: block_table given but the context is not paged", name); *why = buf; return false;
  }
  return true;
}

}  // namespace

std::string& vp::context_free_error() {
  static thread_local std::string msg;
  return msg;
}

extern "C" {

int32_t vp_max_kept(const vp_budget* budget, int32_t n_visual) {
  if (!budget || n_visual < 0) return -1;
  std::string why;
  if (!budget_ok(*budget, &why)) return -1;
  return max_kept(*budget, n_visual);
}

vp_status vp_init(const vp_config* cfg, vp_ctx** out_ctx) {
  if (!out_ctx) return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: out_ctx is NULL");
  *out_ctx = nullptr;
  if (!cfg) return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: cfg is NULL");
  const vp_config& c = *cfg;
  if (c.max_batch < 1 || c.num_q_heads < 1 || c.num_kv_heads < 1)
    return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: max_batch, num_q_heads and num_kv_heads must be >= 1");
  if (c.num_q_heads % c.num_kv_heads != 0)
    return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: num_q_heads must be a multiple of num_kv_heads");
  if (c.dtype != VP_BF16 && c.dtype != VP_FP32)
    return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: dtype must be VP_BF16 or VP_FP32");
  if (c.max_visual < 0 || c.max_seq < c.max_visual + 1)
    return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: need 0 <= max_visual and max_seq >= max_visual + 1");
  if (c.paged != 0 && c.paged != 1) return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: paged must be 0 or 1");
  if (c.paged && (c.page_size < 1 || c.page_size > 256 || (c.page_size & (c.page_size - 1))))
    return fail(nullptr, VP_ERR_INVALID_ARG, "vp_init: page_size must be a power of two in [1, 256]");
  if (c.head_dim != 64 && c.head_dim != 128)
    return fail(nullptr, VP_ERR_UNSUPPORTED, "vp_init: head_dim must be 64 or 128");
  if (c.num_q_heads / c.num_kv_heads > kMaxGroup || c.num_q_heads > kMaxHeads)
    return fail(nullptr, VP_ERR_UNSUPPORTED, "vp_init: needs G = H / Hkv <= 16 and H <= 128");
  if (c.max_visual > kMaxVisual)
    return fail(nullptr, VP_ERR_UNSUPPORTED, "vp_init: max_visual above 32768 is not supported");

  vp_ctx* ctx = new vp_ctx();
  ctx->cfg = c;
  cudaError_t e = cudaGetDevice(&ctx->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, ctx->device);
  if (e != cudaSuccess) {
    vp_status st = cuda_fail(nullptr, "vp_init: no usable CUDA device", e);
    delete ctx;
    return st;
  }
  ctx->lay = vp::ws_layout(c.max_batch, c.num_q_heads, c.num_kv_heads, c.head_dim, c.max_visual, c.max_seq,
                          ctx->num_sms);
  const vp::WsLayout& L = ctx->lay;
  const size_t off = L.total;
  ctx->ws_bytes = off;
  e = cudaMalloc(&ctx->ws, ctx->ws_bytes);
  if (e != cudaSuccess) {
    vp_status st = cuda_fail(nullptr, "vp_init: workspace allocation failed", e);
    delete ctx;
    return st;
  }
  char* base = static_cast<char*>(ctx->ws);
  ctx->z_ws = reinterpret_cast<float*>(base + L.o_z);
  ctx->split_st = reinterpret_cast<float*>(base + L.o_st);
  ctx->split_o = reinterpret_cast<float*>(base + L.o_o);
  ctx->gpart_o = reinterpret_cast<float*>(base + L.o_go);
  ctx->gpart_st = reinterpret_cast<float*>(base + L.o_gs);
  ctx->mt_o = reinterpret_cast<float*>(base + L.o_mo);
  ctx->mt_st = reinterpret_cast<float*>(base + L.o_ms);
  ctx->hmax = reinterpret_cast<float*>(base + L.o_hm);
  ctx->tickets = reinterpret_cast<unsigned*>(base + L.o_tickets);
  ctx->err = reinterpret_cast<unsigned*>(base + L.o_err);
  e = cudaMemset(ctx->ws, 0, ctx->ws_bytes);
  if (e == cudaSuccess) e = vp::configure_kernels(c.max_visual, c.num_q_heads, L.nsp_max);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    vp_status st = cuda_fail(nullptr, "vp_init: workspace set-up failed", e);
    cudaFree(ctx->ws);
    delete ctx;
    return st;
  }
  *out_ctx = ctx;
  return VP_OK;
}

vp_status vp_decode_step(vp_ctx* ctx, int32_t batch, const void* q,
                         const vp_kv* k_cache, const vp_kv* v_cache,
                         const vp_span* visual_span, const int32_t* text_len,
                         const vp_budget* budget, void* out,
                         int32_t* kept_idx, int32_t kept_cap, int32_t* kept_count,
                         float* mass, float* mass_stats, void* cuda_stream) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  ctx->last_error.clear();
  const vp_config& c = ctx->cfg;
  if (batch < 0) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_step: batch < 0");
  if (batch > c.max_batch) return fail(ctx, VP_ERR_CAPACITY, "vp_decode_step: batch exceeds max_batch");
  if (!budget) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_step: budget is NULL");
  std::string why;
  if (!budget_ok(*budget, &why)) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_step: " + why);
  const int32_t need = max_kept(*budget, c.max_visual);
  if (kept_cap < 0 || kept_cap < need) {
    return fail(ctx, VP_ERR_CAPACITY, "vp_decode_step: kept_cap " + std::to_string(kept_cap) +
                " is below the largest budget " + std::to_string(need));
  }
  if (batch == 0) return VP_OK;
  if (!q || !out || !text_len || !visual_span || !visual_span->vis_start || !visual_span->vis_len ||
      !kept_count || !mass || (kept_cap > 0 && !kept_idx))
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_step: NULL tensor argument");
  if (!aligned16(q) || !aligned16(out)) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_step: q and out must be 16-byte aligned");
  if (!kv_ok(ctx, k_cache, "k_cache", &why) || !kv_ok(ctx, v_cache, "v_cache", &why))
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_step: " + why);

  const int H = c.num_q_heads, Hkv = c.num_kv_heads;
  vp::StepParams p;
  memset(&p, 0, sizeof p);
  p.dtype = c.dtype;
  p.B = batch; p.H = H; p.Hkv = Hkv; p.G = H / Hkv; p.D = c.head_dim;
  p.max_visual = c.max_visual; p.max_seq = c.max_seq;
  p.paged = c.paged; p.page_size = c.paged ? c.page_size : 1;
  p.page_shift = 0;
  while ((1 << p.page_shift) < p.page_size) ++p.page_shift;
  p.q = q;
  p.k = vp::KvView{k_cache->data, k_cache->stride_b, k_cache->stride_h, k_cache->stride_t,
                   k_cache->block_table, k_cache->max_pages, k_cache->num_pages};
  p.v = vp::KvView{v_cache->data, v_cache->stride_b, v_cache->stride_h, v_cache->stride_t,
                   v_cache->block_table, v_cache->max_pages, v_cache->num_pages};
  p.vis_start = visual_span->vis_start;
  p.vis_len = visual_span->vis_len;
  p.text_len = text_len;
  p.mode = budget->mode;
  p.granularity = budget->granularity;
  p.inv_tau = 1.0f / budget->tau;
  const float scale = budget->scale > 0.f ? budget->scale : 1.0f / sqrtf((float)c.head_dim);
  p.c_log2 = scale * 1.4426950408889634f;
  p.r_lo_ppm = budget->r_lo_ppm; p.r_hi_ppm = budget->r_hi_ppm;
  p.ratio_ppm = budget->ratio_ppm; p.fixed_k = budget->fixed_k;
  p.out = out; p.kept_idx = kept_idx; p.kept_cap = kept_cap; p.kept_count = kept_count;
  p.mass = mass; p.mass_stats = mass_stats;
  p.z_ws = ctx->z_ws; p.split_st = ctx->split_st; p.split_o = ctx->split_o;
  p.gpart_o = ctx->gpart_o; p.gpart_st = ctx->gpart_st; p.tickets = ctx->tickets; p.err = ctx->err;
  p.hp = ctx->lay.hp;
  p.nsp_max = ctx->lay.nsp_max;
  p.nk_max = ctx->lay.nk_max;
  if (!vp::plan_step(p, ctx->num_sms, kept_cap, budget->granularity, ctx->score_path))
    return fail(ctx, VP_ERR_UNSUPPORTED, "vp_decode_step: the tcgen05 score kernel (VP_SCORE_TC) cannot serve this "
                "call (needs bf16, head_dim 128, G <= 16, pages of >= 8 tokens, a tensor-descriptor layout)");
  p.mt_o = ctx->mt_o; p.mt_st = ctx->mt_st; p.hmax = ctx->hmax;
  if (ctx->diag_n_act || ctx->diag_bits) {
    memcpy(&p.act_delta_bits, &ctx->diag_delta, sizeof(float));
    p.n_act = ctx->diag_n_act;
    p.act_bits = ctx->diag_bits;
    p.act_words = (c.max_visual + 31) / 32;
  }
  p.fused = vp::select_kind(p, kept_cap);

  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  cudaEvent_t* tev = nullptr;
  unsigned rec_flags = cudaEventRecordDefault;
  if (ctx->tslots > 0) {
    tev = &ctx->tev[4 * (size_t)(ctx->tcalls++ % ctx->tslots)];
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
      rec_flags = cudaEventRecordExternal;
  }
  cudaError_t e = cudaSuccess;
  if (tev) e = cudaEventRecordWithFlags(tev[0], st, rec_flags);
  if (e == cudaSuccess) e = vp::launch_score(p, st);
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_decode_step: score kernel launch", e);
  if (tev) e = cudaEventRecordWithFlags(tev[1], st, rec_flags);
  if (e == cudaSuccess) e = vp::launch_select(p, st);
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_decode_step: select kernel launch", e);
  if (tev) e = cudaEventRecordWithFlags(tev[2], st, rec_flags);
  if (e == cudaSuccess) e = vp::launch_gather(p, st);
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_decode_step: gather kernel launch", e);
  if (tev) e = cudaEventRecordWithFlags(tev[3], st, rec_flags);
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_decode_step: timing event", e);
  ctx->last_score_path = p.use_tc ? VP_SCORE_TC : VP_SCORE_MMA;
  ctx->last_kernels = p.fused == 1 ? 2 : 3;
  return VP_OK;
}

const char* vp_last_error(const vp_ctx* ctx) {
  return ctx ? ctx->last_error.c_str() : vp::context_free_error().c_str();
}

vp_status vp_decode_gather(vp_ctx* ctx, int32_t batch, const void* q,
                           const vp_kv* k_cache, const vp_kv* v_cache,
                           const vp_span* visual_span, const int32_t* text_len,
                           const int32_t* kept_idx, int32_t kept_cap, const int32_t* kept_count,
                           int32_t granularity, float scale, void* out, void* cuda_stream) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  ctx->last_error.clear();
  const vp_config& c = ctx->cfg;
  if (batch < 0) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_gather: batch < 0");
  if (batch > c.max_batch) return fail(ctx, VP_ERR_CAPACITY, "vp_decode_gather: batch exceeds max_batch");
  if (granularity != 0 && granularity != 1) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_gather: granularity must be 0 or 1");
  if (kept_cap < 0) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_gather: kept_cap < 0");
  if (!(scale >= 0.f) || !std::isfinite(scale)) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_gather: scale must be finite and >= 0");
  if (c.dtype != VP_BF16) return fail(ctx, VP_ERR_UNSUPPORTED, "vp_decode_gather: needs bf16 caches");
  if (batch == 0) return VP_OK;
  if (!q || !out || !text_len || !visual_span || !visual_span->vis_start || !visual_span->vis_len || !kept_count ||
      (kept_cap > 0 && !kept_idx))
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_gather: NULL tensor argument");
  if (!aligned16(q) || !aligned16(out)) return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_gather: q and out must be 16-byte aligned");
  std::string why;
  if (!kv_ok(ctx, k_cache, "k_cache", &why) || !kv_ok(ctx, v_cache, "v_cache", &why))
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_decode_gather: " + why);

  const int H = c.num_q_heads, Hkv = c.num_kv_heads, D = c.head_dim;
  vp::StepParams p;
  memset(&p, 0, sizeof p);
  p.dtype = c.dtype;
  p.B = batch; p.H = H; p.Hkv = Hkv; p.G = H / Hkv; p.D = D;
  p.max_visual = c.max_visual; p.max_seq = c.max_seq;
  p.paged = c.paged; p.page_size = c.paged ? c.page_size : 1;
  while ((1 << p.page_shift) < p.page_size) ++p.page_shift;
  p.q = q;
  p.k = vp::KvView{k_cache->data, k_cache->stride_b, k_cache->stride_h, k_cache->stride_t,
                   k_cache->block_table, k_cache->max_pages, k_cache->num_pages};
  p.v = vp::KvView{v_cache->data, v_cache->stride_b, v_cache->stride_h, v_cache->stride_t,
                   v_cache->block_table, v_cache->max_pages, v_cache->num_pages};
  p.vis_start = visual_span->vis_start;
  p.vis_len = visual_span->vis_len;
  p.text_len = text_len;
  p.anchor = 1;
  p.granularity = granularity;
  p.inv_tau = 1.f;
  p.c_log2 = (scale > 0.f ? scale : 1.0f / sqrtf((float)D)) * 1.4426950408889634f;
  p.kept_idx = const_cast<int32_t*>(kept_idx);
  p.kept_cap = kept_cap;
  p.kept_count = const_cast<int32_t*>(kept_count);
  p.out = out;
  p.z_ws = ctx->z_ws; p.split_st = ctx->split_st; p.split_o = ctx->split_o;
  p.gpart_o = ctx->gpart_o; p.gpart_st = ctx->gpart_st; p.tickets = ctx->tickets; p.err = ctx->err;
  p.mt_o = ctx->mt_o; p.mt_st = ctx->mt_st; p.hmax = ctx->hmax;
  // Score splits as planned for the decode step; their weight covers the
  // cache outside the visual span plus the kept rows.  The merge of the
  // splits is the chunk gather with no kept chunks.
  const vp::Plan pl = vp::make_plan(batch, Hkv, D, ctx->num_sms, c.max_visual, c.max_seq, 0, granularity);
  p.hp = ctx->lay.hp;
  p.ns = pl.ns; p.nsp_max = ctx->lay.nsp_max; p.cl = 1;
  {
    long long w = 2LL * ((c.max_seq + 31) / 32 - c.max_visual / 32 + (kept_cap + 31) / 32);
    if (w < 1) w = 1;
    p.split_w = (int)((w + pl.ns - 1) / pl.ns);
  }
  p.nk = 0; p.nk_max = ctx->lay.nk_max;
  p.nm = pl.ns > 1 ? (D / 16 < 8 ? D / 16 : 8) : 0;
  p.nc = p.nm > 0 ? p.nm : 1;
  p.gslice = 0;
  vp::encode_kv_maps(p);
  if (!p.use_tma)
    return fail(ctx, VP_ERR_UNSUPPORTED, "vp_decode_gather: the cache layout needs the bulk-tensor path "
                "(token axis not outermost, pages of at least 8 tokens)");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = vp::launch_score(p, st);
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_decode_gather: score kernel launch", e);
  e = vp::launch_gather(p, st);
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_decode_gather: merge kernel launch", e);
  ctx->last_score_path = VP_SCORE_MMA;
  ctx->last_kernels = 2;
  return VP_OK;
}

vp_status vp_set_diagnostics(vp_ctx* ctx, float delta, int32_t* n_act, uint32_t* active_bits) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  ctx->last_error.clear();
  if ((n_act || active_bits) && !(delta > 0.f && std::isfinite(delta)))
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_set_diagnostics: delta must be finite and > 0");
  if ((n_act && (reinterpret_cast<uintptr_t>(n_act) & 3u)) || (active_bits && (reinterpret_cast<uintptr_t>(active_bits) & 3u)))
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_set_diagnostics: arrays must be 4-byte aligned");
  ctx->diag_delta = delta;
  ctx->diag_n_act = n_act;
  ctx->diag_bits = active_bits;
  return VP_OK;
}

vp_status vp_compact_kv(vp_ctx* ctx, int32_t batch, const vp_kv* src, const vp_kv* dst,
                        const vp_span* visual_span, const int32_t* text_len,
                        const int32_t* kept_idx, int32_t kept_cap, const int32_t* kept_count,
                        void* cuda_stream) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  ctx->last_error.clear();
  const vp_config& c = ctx->cfg;
  if (batch < 0) return fail(ctx, VP_ERR_INVALID_ARG, "vp_compact_kv: batch < 0");
  if (batch > c.max_batch) return fail(ctx, VP_ERR_CAPACITY, "vp_compact_kv: batch exceeds max_batch");
  if (kept_cap < 0) return fail(ctx, VP_ERR_INVALID_ARG, "vp_compact_kv: kept_cap < 0");
  if (batch == 0) return VP_OK;
  if (!text_len || !visual_span || !visual_span->vis_start || !visual_span->vis_len || !kept_count ||
      (kept_cap > 0 && !kept_idx))
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_compact_kv: NULL tensor argument");
  std::string why;
  if (!kv_ok(ctx, src, "src", &why)) return fail(ctx, VP_ERR_INVALID_ARG, "vp_compact_kv: " + why);
  const size_t esz = c.dtype == VP_BF16 ? 2 : 4;
  if (!dst || !dst->data || !aligned16(dst->data) || dst->block_table)
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_compact_kv: dst must be a contiguous cache with 16-byte-aligned data");
  for (int64_t st : {dst->stride_b, dst->stride_h, dst->stride_t})
    if (st < 0 || ((uint64_t)st * esz) % 16 != 0)
      return fail(ctx, VP_ERR_INVALID_ARG, "vp_compact_kv: dst strides must be >= 0 and multiples of 16 bytes");
  if (dst->data == src->data) return fail(ctx, VP_ERR_INVALID_ARG, "vp_compact_kv: dst must not overlap src");
  vp::CompactParams p;
  memset(&p, 0, sizeof p);
  p.src = vp::KvView{src->data, src->stride_b, src->stride_h, src->stride_t, src->block_table, src->max_pages,
                     src->num_pages};
  p.paged = c.paged;
  p.page_size = c.paged ? c.page_size : 1;
  while ((1 << p.page_shift) < p.page_size) ++p.page_shift;
  p.dst = const_cast<void*>(dst->data);  // the destination cache is written
  p.dsb = dst->stride_b; p.dsh = dst->stride_h; p.dst_t = dst->stride_t;
  p.vis_start = visual_span->vis_start; p.vis_len = visual_span->vis_len; p.text_len = text_len;
  p.kept_idx = kept_idx; p.kept_cap = kept_cap; p.kept_count = kept_count;
  p.B = batch; p.Hkv = c.num_kv_heads; p.D = c.head_dim; p.esz = (int)esz;
  p.max_visual = c.max_visual; p.max_seq = c.max_seq;
  p.err = ctx->err;
  const cudaError_t e = vp::launch_compact(p, static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_compact_kv: launch", e);
  return VP_OK;
}

vp_status vp_set_score_path(vp_ctx* ctx, int32_t path) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  ctx->last_error.clear();
  if (path != VP_SCORE_AUTO && path != VP_SCORE_MMA && path != VP_SCORE_TC)
    return fail(ctx, VP_ERR_INVALID_ARG, "vp_set_score_path: path must be VP_SCORE_AUTO, VP_SCORE_MMA or VP_SCORE_TC");
  ctx->score_path = path;
  return VP_OK;
}

vp_status vp_last_launch(const vp_ctx* ctx, int32_t* score_path, int32_t* kernels) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  if (score_path) *score_path = ctx->last_score_path;
  if (kernels) *kernels = ctx->last_kernels;
  return VP_OK;
}

vp_status vp_check_errors(vp_ctx* ctx, void* cuda_stream) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = cudaStreamSynchronize(st);
  unsigned word = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&word, ctx->err, sizeof word, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && word) e = cudaMemset(ctx->err, 0, sizeof word);
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_check_errors", e);
  if (!word) { ctx->last_error.clear(); return VP_OK; }
  std::string msg = "device checks failed:";
  if (word & vp::ERR_SPAN) msg += " visual span outside the live cache or above max_visual;";
  if (word & vp::ERR_TEXT) msg += " text_len < 1;";
  if (word & vp::ERR_LEN) msg += " vis_len + text_len above max_seq;";
  if (word & vp::ERR_PAGE) msg += " block table entry outside the pool;";
  if (word & vp::ERR_KEPT) msg += " kept index outside the visual span;";
  if (word & vp::ERR_NONFINITE) msg += " non-finite importance score;";
  if (word & vp::ERR_TIMEOUT) msg += " an asynchronous copy did not complete in time;";
  return fail(ctx, VP_ERR_DEVICE_PRECOND, msg);
}

vp_status vp_timing_enable(vp_ctx* ctx, int32_t slots) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  if (slots < 0) return fail(ctx, VP_ERR_INVALID_ARG, "vp_timing_enable: slots < 0");
  cudaDeviceSynchronize();
  for (cudaEvent_t ev : ctx->tev) cudaEventDestroy(ev);
  ctx->tev.clear();
  ctx->tslots = 0;
  ctx->tcalls = 0;
  for (int64_t i = 0; i < 4LL * slots; ++i) {
    cudaEvent_t ev;
    cudaError_t e = cudaEventCreate(&ev);
    if (e != cudaSuccess) {
      for (cudaEvent_t x : ctx->tev) cudaEventDestroy(x);
      ctx->tev.clear();
      return cuda_fail(ctx, "vp_timing_enable: cudaEventCreate", e);
    }
    ctx->tev.push_back(ev);
  }
  ctx->tslots = slots;
  return VP_OK;
}

vp_status vp_timing_read(vp_ctx* ctx, float* ms, int32_t max_slots, int32_t* n_slots) {
  if (!ctx) return VP_ERR_NOT_INITIALIZED;
  if (!ms || !n_slots || max_slots < 0) return fail(ctx, VP_ERR_INVALID_ARG, "vp_timing_read: bad arguments");
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(ctx, "vp_timing_read", e);
  const int64_t n = std::min<int64_t>({(int64_t)max_slots, (int64_t)ctx->tslots, ctx->tcalls});
  for (int64_t s = 0; s < n; ++s) {
    for (int k = 0; k < 3; ++k) {
      float t = -1.f;
      if (cudaEventElapsedTime(&t, ctx->tev[4 * s + k], ctx->tev[4 * s + k + 1]) != cudaSuccess) t = -1.f;
      ms[3 * s + k] = t;
    }
  }
  cudaGetLastError();  // an event that never fired leaves a sticky-free error code
  *n_slots = (int32_t)n;
  return VP_OK;
}

void vp_free(vp_ctx* ctx) {
  if (!ctx) return;
  if (!ctx->tev.empty()) {
    cudaDeviceSynchronize();
    for (cudaEvent_t ev : ctx->tev) cudaEventDestroy(ev);
  }
  if (ctx->ws) cudaFree(ctx->ws);
  delete ctx;
}

}  // extern "C"
