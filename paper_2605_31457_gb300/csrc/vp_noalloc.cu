// vp_decode_step_noalloc: the decode step for callers that cannot allocate
// device memory, with its scratch in a fixed, file-scope device array.
//
// Who needs it: code that runs where cudaMalloc is off limits -- a plugin or
// custom-op host whose framework owns every byte of device memory through its
// own pool and forbids allocations on the inference path, or a caller that
// must not introduce the device-wide synchronisation an allocation can imply
// in the middle of a latency-critical loop.  Such callers still own and pass
// every input and output; only the intermediate scratch moves here.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <mutex>
#include <string>

#include "vp.h"
#include "vp_internal.h"

namespace {

// The scratch every call shares.  Each GPU that loads the library holds these
// bytes until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[VP_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Shapes a scratch layout was planned for.
struct LayoutKey {
  int batch = -1, H = 0, Hkv = 0, D = 0, max_visual = 0, max_seq = 0;
  bool operator==(const LayoutKey& o) const {
    return batch == o.batch && H == o.H && Hkv == o.Hkv && D == o.D && max_visual == o.max_visual &&
           max_seq == o.max_seq;
  }
};

struct DeviceSlot {
  bool ready = false;
  void* scratch = nullptr;  // device address of g_noalloc_scratch on this device
  int num_sms = 0;
  // The last call's scratch layout (planning it walks every batch size), and
  // the largest visual span the select kernel's shared memory was raised for.
  LayoutKey key;
  vp::WsLayout lay;
  int configured_visual = -1;
};

std::mutex g_mu;
DeviceSlot g_slots[kMaxDevices];

// Failure text goes where vp_last_error(NULL) reads it, in this thread.
vp_status fail(vp_status st, const std::string& msg) {
  vp::context_free_error() = msg;
  return st;
}

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Largest K_t of the budget for n visual tokens (same rule as vp_max_kept).
int64_t max_kept(const vp_budget& bd, int64_t n) {
  if (n <= 0) return 0;
  switch (bd.mode) {
    case VP_DENSE:
    case VP_TOP_P: return n;
    case VP_FIXED_K: return std::min<int64_t>(std::max<int64_t>(bd.fixed_k, 0), n);
    case VP_FIXED_RATIO: return std::min<int64_t>(std::max<int64_t>(ceil_div((int64_t)bd.ratio_ppm * n, 1000000), 1), n);
    case VP_ADAPTIVE: {
      const int64_t lo = ceil_div((int64_t)bd.r_lo_ppm * n, 1000000);
      return std::min<int64_t>(std::max<int64_t>(lo, (int64_t)bd.r_hi_ppm * n / 1000000), n);
    }
    default: return -1;
  }
}

// Once per device, with that device current: resolve the array's device
// address (in host code the symbol is only a stand-in, not a device address)
// and read the SM count the launch plan needs.
vp_status setup_device(int dev, DeviceSlot** out) {
  if (dev < 0 || dev >= kMaxDevices) return fail(VP_ERR_UNSUPPORTED, "vp_decode_step_noalloc: device index too large");
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceSlot& s = g_slots[dev];
  if (!s.ready) {
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess)
      return fail(VP_ERR_CUDA, std::string("vp_decode_step_noalloc: cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess)
      return fail(VP_ERR_CUDA, std::string("vp_decode_step_noalloc: device query: ") + cudaGetErrorString(e));
    s.scratch = ptr;
    s.num_sms = sms;
    s.ready = true;
  }
  *out = &s;
  return VP_OK;
}

}  // namespace

extern "C" vp_status vp_decode_step_noalloc(const vp_config* cfg, int32_t batch, const void* q,
                                            const vp_kv* k_cache, const vp_kv* v_cache,
                                            const vp_span* visual_span, const int32_t* text_len,
                                            const vp_budget* budget, void* out, int32_t* kept_idx,
                                            int32_t kept_cap, int32_t* kept_count, float* mass,
                                            float* mass_stats, void* cuda_stream) {
  vp::context_free_error().clear();
  if (!cfg || !budget) return fail(VP_ERR_INVALID_ARG, "vp_decode_step_noalloc: cfg and budget are required");
  const vp_config& c = *cfg;
  if (c.max_batch < 1 || c.num_q_heads < 1 || c.num_kv_heads < 1 || c.num_q_heads % c.num_kv_heads ||
      (c.dtype != VP_BF16 && c.dtype != VP_FP32) || c.max_visual < 0 || c.max_seq < c.max_visual + 1 ||
      c.paged < 0 || c.paged > 1 ||
      (c.paged && (c.page_size < 1 || c.page_size > 256 || (c.page_size & (c.page_size - 1)))))
    return fail(VP_ERR_INVALID_ARG, "vp_decode_step_noalloc: malformed cfg");
  if ((c.head_dim != 64 && c.head_dim != 128) || c.num_q_heads / c.num_kv_heads > 16 ||
      c.num_q_heads > 128 || c.max_visual > 32768)
    return fail(VP_ERR_UNSUPPORTED, "vp_decode_step_noalloc: shape not supported");
  if (batch < 0 || batch > c.max_batch) return fail(VP_ERR_CAPACITY, "vp_decode_step_noalloc: batch outside [0, max_batch]");
  if (!(budget->tau > 0.f) || !isfinite(budget->tau) || !(budget->scale >= 0.f) || !isfinite(budget->scale) ||
      budget->mode < VP_ADAPTIVE || budget->mode > VP_TOP_P || (budget->mode == VP_TOP_P && budget->granularity != 0) || budget->r_lo_ppm < 0 || budget->r_lo_ppm > 1000000 ||
      budget->r_hi_ppm < 0 || budget->r_hi_ppm > 1000000 || budget->ratio_ppm < 0 || budget->ratio_ppm > 1000000 ||
      budget->fixed_k < 0 || (budget->granularity != 0 && budget->granularity != 1))
    return fail(VP_ERR_INVALID_ARG, "vp_decode_step_noalloc: malformed budget");
  if (kept_cap < 0 || kept_cap < max_kept(*budget, c.max_visual))
    return fail(VP_ERR_CAPACITY, "vp_decode_step_noalloc: kept_cap " + std::to_string(kept_cap) +
                " is negative or below the largest budget " + std::to_string(max_kept(*budget, c.max_visual)));
  if (batch == 0) return VP_OK;
  if (!q || !out || !text_len || !visual_span || !visual_span->vis_start || !visual_span->vis_len || !kept_count ||
      !mass || (kept_cap > 0 && !kept_idx) || !k_cache || !v_cache || !k_cache->data || !v_cache->data)
    return fail(VP_ERR_INVALID_ARG, "vp_decode_step_noalloc: NULL tensor argument");
  const size_t esz = c.dtype == VP_BF16 ? 2 : 4;
  for (const vp_kv* kv : {k_cache, v_cache}) {
    if (!aligned16(kv->data) || kv->stride_b < 0 || kv->stride_h < 0 || kv->stride_t < 0 ||
        ((uint64_t)kv->stride_b * esz) % 16 || ((uint64_t)kv->stride_h * esz) % 16 || ((uint64_t)kv->stride_t * esz) % 16 ||
        (c.paged ? (!kv->block_table || kv->max_pages < 1 || kv->num_pages < 1) : kv->block_table != nullptr))
      return fail(VP_ERR_INVALID_ARG, "vp_decode_step_noalloc: malformed cache view");
  }
  if (!aligned16(q) || !aligned16(out)) return fail(VP_ERR_INVALID_ARG, "vp_decode_step_noalloc: q and out must be 16-byte aligned");

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(VP_ERR_CUDA, std::string("vp_decode_step_noalloc: ") + cudaGetErrorString(e));
  DeviceSlot* slot = nullptr;
  vp_status st = setup_device(dev, &slot);
  if (st != VP_OK) return st;

  // Scratch layout for this call (the partial formats of a context's
  // workspace), planned again only when the shapes change.
  const int H = c.num_q_heads, Hkv = c.num_kv_heads, G = H / Hkv, D = c.head_dim;
  const LayoutKey key{batch, H, Hkv, D, c.max_visual, c.max_seq};
  vp::WsLayout L;
  bool configure = false;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!(slot->key == key)) {
      slot->lay = vp::ws_layout(batch, H, Hkv, D, c.max_visual, c.max_seq, slot->num_sms);
      slot->key = key;
    }
    L = slot->lay;
    configure = c.max_visual > slot->configured_visual;
  }
  if (L.total > (size_t)VP_NOALLOC_SCRATCH_BYTES)
    return fail(VP_ERR_CAPACITY, "vp_decode_step_noalloc: this batch and cfg need " + std::to_string(L.total) +
                " scratch bytes; the fixed scratch holds " + std::to_string((size_t)VP_NOALLOC_SCRATCH_BYTES));
  if (configure) {  // kernel attributes: the select kernel's shared memory grows with max_visual
    e = vp::configure_kernels(c.max_visual, H, L.nsp_max);
    if (e != cudaSuccess) return fail(VP_ERR_CUDA, std::string("vp_decode_step_noalloc: ") + cudaGetErrorString(e));
    std::lock_guard<std::mutex> lock(g_mu);
    if (c.max_visual > slot->configured_visual) slot->configured_visual = c.max_visual;
  }

  char* base = static_cast<char*>(slot->scratch);
  vp::StepParams p;
  memset(&p, 0, sizeof p);
  p.dtype = c.dtype;
  p.B = batch; p.H = H; p.Hkv = Hkv; p.G = G; p.D = D;
  p.max_visual = c.max_visual; p.max_seq = c.max_seq;
  p.paged = c.paged; p.page_size = c.paged ? c.page_size : 1;
  while ((1 << p.page_shift) < p.page_size) ++p.page_shift;
  p.q = q;
  p.k = vp::KvView{k_cache->data, k_cache->stride_b, k_cache->stride_h, k_cache->stride_t,
                   k_cache->block_table, k_cache->max_pages, k_cache->num_pages};
  p.v = vp::KvView{v_cache->data, v_cache->stride_b, v_cache->stride_h, v_cache->stride_t,
                   v_cache->block_table, v_cache->max_pages, v_cache->num_pages};
  p.vis_start = visual_span->vis_start; p.vis_len = visual_span->vis_len; p.text_len = text_len;
  p.mode = budget->mode; p.granularity = budget->granularity;
  p.inv_tau = 1.0f / budget->tau;
  const float scale = budget->scale > 0.f ? budget->scale : 1.0f / sqrtf((float)D);
  p.c_log2 = scale * 1.4426950408889634f;
  p.r_lo_ppm = budget->r_lo_ppm; p.r_hi_ppm = budget->r_hi_ppm;
  p.ratio_ppm = budget->ratio_ppm; p.fixed_k = budget->fixed_k;
  p.out = out; p.kept_idx = kept_idx; p.kept_cap = kept_cap; p.kept_count = kept_count;
  p.mass = mass; p.mass_stats = mass_stats;
  p.tickets = reinterpret_cast<unsigned*>(base + L.o_tickets);
  p.err = reinterpret_cast<unsigned*>(base + L.o_err);
  p.z_ws = reinterpret_cast<float*>(base + L.o_z);
  p.split_st = reinterpret_cast<float*>(base + L.o_st);
  p.split_o = reinterpret_cast<float*>(base + L.o_o);
  p.gpart_o = reinterpret_cast<float*>(base + L.o_go);
  p.gpart_st = reinterpret_cast<float*>(base + L.o_gs);
  p.mt_o = reinterpret_cast<float*>(base + L.o_mo);
  p.mt_st = reinterpret_cast<float*>(base + L.o_ms);
  p.hmax = reinterpret_cast<float*>(base + L.o_hm);
  p.hp = L.hp;
  p.nsp_max = L.nsp_max;
  p.nk_max = L.nk_max;
  if (!vp::plan_step(p, slot->num_sms, kept_cap, budget->granularity))
    return fail(VP_ERR_UNSUPPORTED, "vp_decode_step_noalloc: no launch plan serves this call");
  p.fused = vp::select_kind(p, kept_cap);

  // Only now that every check has passed: clear the counters, then launch.
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  e = cudaMemsetAsync(base, 0, L.zero_bytes, stream);
  if (e == cudaSuccess) e = vp::launch_score(p, stream);
  if (e == cudaSuccess) e = vp::launch_select(p, stream);
  if (e == cudaSuccess) e = vp::launch_gather(p, stream);
  if (e != cudaSuccess) return fail(VP_ERR_CUDA, std::string("vp_decode_step_noalloc: launch: ") + cudaGetErrorString(e));
  return VP_OK;
}

