// CUDA kernels of one VisionPulse decode step (arxiv 2605.31457, Sec. 4.2-4.3).
//
//   k_score   per (sequence, kv-head, split): logits of the G query heads of the
//             kv-head against every key of the split (Eq. 6's Z).  Visual logits
//             go to the workspace; visual and text tokens get separate online
//             softmax statistics at tau = 1 and at tau (the two sums of Eq. 6);
//             text tokens also accumulate their unnormalised attention output.
//   k_select  per sequence (or per kv-head): merges the split statistics into
//             the visual mass per head (Eq. 5) and its head-max (Sec. 4.3), the
//             budget K_t (Eq. 7 + clamp of Sec. 5.2), the importance score S_i
//             (Eq. 2) and the Top-K_t set (Eq. 3) by radix select, ties to the
//             lower index, emitted in ascending order.
//   k_gather  per (sequence, kv-head, chunk of the kept set): attention of the
//             kept visual tokens, reading V only for them; the last chunk to
//             finish merges every partial (text splits and kept chunks) in
//             log-sum-exp form and writes the output (Sec. 4.2, Sec. 5.7).
//
// Logits are carried in log2 units (z * log2 e) so that every exponential is
// one exp2f; exp(z - m) = exp2(z2 - m2) and exp((z - m) / tau) =
// exp2((z2 - m2) / tau).
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math_constants.h>
#include <stdint.h>

#include "vp_internal.h"

namespace vp {
namespace {

constexpr int kWarps = 4;
constexpr int kThreads = 32 * kWarps;
constexpr int kSelThreads = 1024;
constexpr int kMaxHeads = 128;
constexpr int kGatherTile = 64;  // kept tokens staged per round in k_gather

// Budget modes (numbering of vp_budget_mode in include/vp.h).
enum { MODE_ADAPTIVE = 0, MODE_FIXED_RATIO = 1, MODE_FIXED_K = 2, MODE_DENSE = 3 };

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}
__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// exp2(a - m) with an empty term (a = -inf) giving exactly 0.
__device__ __forceinline__ float exp2_rel(float a, float m) {
  return a == -CUDART_INF_F ? 0.f : exp2f(a - m);
}
__device__ __forceinline__ float exp2_tau(float a, float m, float inv_tau) {
  return a == -CUDART_INF_F ? 0.f : exp2f((a - m) * inv_tau);
}

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// Loads N consecutive elements (N * sizeof(T) in {4, 8, 16} bytes) as floats.
template <int N>
__device__ __forceinline__ void load_f(const float* p, float (&f)[N]) {
  static_assert(N == 1 || N == 2 || N == 4, "fp32 vector width");
  if constexpr (N == 4) {
    float4 v = __ldg(reinterpret_cast<const float4*>(p));
    f[0] = v.x; f[1] = v.y; f[2] = v.z; f[3] = v.w;
  } else if constexpr (N == 2) {
    float2 v = __ldg(reinterpret_cast<const float2*>(p));
    f[0] = v.x; f[1] = v.y;
  } else {
    f[0] = __ldg(p);
  }
}
__device__ __forceinline__ void bf2(uint32_t u, float& lo, float& hi) {
  lo = __uint_as_float(u << 16);
  hi = __uint_as_float(u & 0xffff0000u);
}
template <int N>
__device__ __forceinline__ void load_f(const __nv_bfloat16* p, float (&f)[N]) {
  static_assert(N == 2 || N == 4 || N == 8, "bf16 vector width");
  if constexpr (N == 8) {
    uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
    bf2(v.x, f[0], f[1]); bf2(v.y, f[2], f[3]); bf2(v.z, f[4], f[5]); bf2(v.w, f[6], f[7]);
  } else if constexpr (N == 4) {
    uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
    bf2(v.x, f[0], f[1]); bf2(v.y, f[2], f[3]);
  } else {
    uint32_t v = __ldg(reinterpret_cast<const unsigned int*>(p));
    bf2(v, f[0], f[1]);
  }
}

struct Seq {
  int vs, nv, tl;
};

// Per-sequence span and length, clamped into the configured ranges; a value
// that needed clamping is recorded in the device error word.
__device__ __forceinline__ Seq load_seq(const StepParams& p, int b, bool report) {
  int vs = __ldg(p.vis_start + b), nv = __ldg(p.vis_len + b), tl = __ldg(p.text_len + b);
  unsigned e = 0;
  if (nv < 0 || nv > p.max_visual) { e |= ERR_SPAN; nv = min(max(nv, 0), p.max_visual); }
  if (tl < 1) { e |= ERR_TEXT; tl = 1; }
  if (nv + tl > p.max_seq) { e |= ERR_LEN; tl = max(1, p.max_seq - nv); }
  if (vs < 0 || vs > tl) { e |= ERR_SPAN; vs = min(max(vs, 0), tl); }
  if (e && report) atomicOr(p.err, e);
  return Seq{vs, nv, tl};
}

// Address of the D-element row of (sequence b, kv-head g, token pos); NULL if
// the paged block table does not map it to a page of the pool.
template <typename T>
__device__ __forceinline__ const T* kv_row(const KvView& kv, const StepParams& p, int b, int g, int pos) {
  const T* base = reinterpret_cast<const T*>(kv.data);
  if (!p.paged)
    return base + (int64_t)b * kv.sb + (int64_t)g * kv.sh + (int64_t)pos * kv.st;
  const int lp = pos >> p.page_shift;
  if (lp >= kv.max_pages) return nullptr;
  const int page = __ldg(kv.block_table + (int64_t)b * kv.max_pages + lp);
  if (page < 0 || page >= kv.num_pages) return nullptr;
  return base + (int64_t)page * kv.sb + (int64_t)g * kv.sh + (int64_t)(pos & (p.page_size - 1)) * kv.st;
}

// Raw dot products of one key row with the GM (padded) query heads in shared memory.
template <typename T, int D, int GM>
__device__ __forceinline__ void dot_row(const T* row, const float (*q_s)[D], float (&z)[GM]) {
  constexpr int CH = 16 / sizeof(T);
#pragma unroll
  for (int h = 0; h < GM; ++h) z[h] = 0.f;
#pragma unroll 4
  for (int d0 = 0; d0 < D; d0 += CH) {
    float kf[CH];
    load_f<CH>(row + d0, kf);
#pragma unroll
    for (int h = 0; h < GM; ++h) {
#pragma unroll
      for (int e = 0; e < CH; e += 4) {
        const float4 qv = *reinterpret_cast<const float4*>(&q_s[h][d0 + e]);
        z[h] = fmaf(qv.x, kf[e], z[h]);
        z[h] = fmaf(qv.y, kf[e + 1], z[h]);
        z[h] = fmaf(qv.z, kf[e + 2], z[h]);
        z[h] = fmaf(qv.w, kf[e + 3], z[h]);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// k_score: grid (ns, Hkv, B), 128 threads.  Each warp walks 32-token groups
// (lane = token) of the split; a split covers a slice of the sequence's work,
// visual tokens weighing 1 (K only) and text tokens 2 (K and V).
// ---------------------------------------------------------------------------
template <typename T, int D, int GM>
__global__ void __launch_bounds__(kThreads) k_score(const StepParams p) {
  constexpr int DPL = D / 32;  // dims per lane in the text P.V phase
  const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.G, H = p.H;

  __shared__ __align__(16) float q_s[GM][D];
  __shared__ float pr_s[kWarps][GM][32];
  __shared__ const T* vrow_s[kWarps][32];
  __shared__ float wst_s[kWarps][GM][ST_N];
  __shared__ float wsc_s[kWarps][GM];
  __shared__ __align__(16) float o_s[GM][D];

  const Seq sq = load_seq(p, b, s == 0 && g == 0);
  const T* qb = reinterpret_cast<const T*>(p.q) + ((int64_t)b * H + g * G) * D;
  for (int i = threadIdx.x; i < GM * D; i += kThreads) {
    const int h = i / D, d = i % D;
    q_s[h][d] = h < G ? to_f(qb[h * D + d]) : 0.f;
  }
  __syncthreads();

  const int W = sq.nv + 2 * sq.tl;
  const int per = (W + p.ns - 1) / p.ns;
  const int w0 = min(W, s * per), w1 = min(W, w0 + per);
  const int va = min(w0, sq.nv), vb = min(w1, sq.nv);
  const int ta = (max(w0, sq.nv) - sq.nv + 1) >> 1, tb = (max(w1, sq.nv) - sq.nv + 1) >> 1;

  float m_v[GM], l1v[GM], ltv[GM], m_t[GM], l1t[GM], ltt[GM], acc[GM][DPL];
#pragma unroll
  for (int h = 0; h < GM; ++h) {
    m_v[h] = m_t[h] = -CUDART_INF_F;
    l1v[h] = ltv[h] = l1t[h] = ltt[h] = 0.f;
#pragma unroll
    for (int j = 0; j < DPL; ++j) acc[h][j] = 0.f;
  }
  unsigned err = 0;

  // Visual tokens: logits to the workspace, visual statistics.
  for (int base = va + warp * 32; base < vb; base += kWarps * 32) {
    const int i = base + lane;
    bool valid = i < vb;
    float z[GM];
    if (valid) {
      const T* row = kv_row<T>(p.k, p, b, g, sq.vs + i);
      if (row) dot_row<T, D, GM>(row, q_s, z); else { valid = false; err |= ERR_PAGE; }
    }
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      if (h >= G) break;
      const float zz = valid ? z[h] * p.c_log2 : -CUDART_INF_F;
      if (i < vb) p.z_ws[((int64_t)b * H + g * G + h) * p.max_visual + i] = zz;
      const float mn = fmaxf(m_v[h], warp_max(zz));
      if (mn > m_v[h]) {
        l1v[h] *= exp2_rel(m_v[h], mn);
        ltv[h] *= exp2_tau(m_v[h], mn, p.inv_tau);
        m_v[h] = mn;
      }
      if (valid) {
        l1v[h] += exp2f(zz - mn);
        ltv[h] += exp2f((zz - mn) * p.inv_tau);
      }
    }
  }

  // Text tokens: text statistics and the unnormalised text output.
  for (int base = ta + warp * 32; base < tb; base += kWarps * 32) {
    const int ti = base + lane;
    bool valid = ti < tb;
    const int pos = ti < sq.vs ? ti : ti + sq.nv;
    float z[GM];
    const T* vrow = nullptr;
    if (valid) {
      const T* row = kv_row<T>(p.k, p, b, g, pos);
      vrow = kv_row<T>(p.v, p, b, g, pos);
      if (row && vrow) dot_row<T, D, GM>(row, q_s, z); else { valid = false; vrow = nullptr; err |= ERR_PAGE; }
    }
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      if (h >= G) break;
      const float zz = valid ? z[h] * p.c_log2 : -CUDART_INF_F;
      const float mn = fmaxf(m_t[h], warp_max(zz));
      if (mn > m_t[h]) {
        const float a = exp2_rel(m_t[h], mn);
        l1t[h] *= a;
        ltt[h] *= exp2_tau(m_t[h], mn, p.inv_tau);
#pragma unroll
        for (int j = 0; j < DPL; ++j) acc[h][j] *= a;
        m_t[h] = mn;
      }
      float pr = 0.f;
      if (valid) {
        pr = exp2f(zz - mn);
        l1t[h] += pr;
        ltt[h] += exp2f((zz - mn) * p.inv_tau);
      }
      pr_s[warp][h][lane] = pr;
    }
    vrow_s[warp][lane] = vrow;
    __syncwarp();
    const int nt = min(32, tb - base);
    for (int t0 = 0; t0 < nt; t0 += 4) {
      float vv[4][DPL];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const T* vr = t0 + u < nt ? vrow_s[warp][t0 + u] : nullptr;
        if (vr) load_f<DPL>(vr + lane * DPL, vv[u]);
        else {
#pragma unroll
          for (int j = 0; j < DPL; ++j) vv[u][j] = 0.f;
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
#pragma unroll
        for (int h = 0; h < GM; ++h) {
          if (h >= G) break;
          const float pr = t0 + u < nt ? pr_s[warp][h][t0 + u] : 0.f;
#pragma unroll
          for (int j = 0; j < DPL; ++j) acc[h][j] = fmaf(pr, vv[u][j], acc[h][j]);
        }
      }
    }
    __syncwarp();
  }
  if (err) atomicOr(p.err, err);

  // Merge the four warps: statistics, then the text outputs (fixed order).
#pragma unroll
  for (int h = 0; h < GM; ++h) {
    if (h >= G) break;
    const float a = warp_sum(l1v[h]), bb = warp_sum(ltv[h]);
    const float c = warp_sum(l1t[h]), d = warp_sum(ltt[h]);
    if (lane == 0) {
      wst_s[warp][h][ST_MV] = m_v[h]; wst_s[warp][h][ST_L1V] = a; wst_s[warp][h][ST_LTV] = bb;
      wst_s[warp][h][ST_MT] = m_t[h]; wst_s[warp][h][ST_L1T] = c; wst_s[warp][h][ST_LTT] = d;
    }
  }
  __syncthreads();
  if (threadIdx.x < G) {
    const int h = threadIdx.x;
    float Mv = -CUDART_INF_F, Mt = -CUDART_INF_F;
    for (int w = 0; w < kWarps; ++w) {
      Mv = fmaxf(Mv, wst_s[w][h][ST_MV]);
      Mt = fmaxf(Mt, wst_s[w][h][ST_MT]);
    }
    float r[ST_N] = {Mv, 0.f, 0.f, Mt, 0.f, 0.f};
    for (int w = 0; w < kWarps; ++w) {
      const float mv = wst_s[w][h][ST_MV], mt = wst_s[w][h][ST_MT];
      r[ST_L1V] += exp2_rel(mv, Mv) * wst_s[w][h][ST_L1V];
      r[ST_LTV] += exp2_tau(mv, Mv, p.inv_tau) * wst_s[w][h][ST_LTV];
      const float at = exp2_rel(mt, Mt);
      r[ST_L1T] += at * wst_s[w][h][ST_L1T];
      r[ST_LTT] += exp2_tau(mt, Mt, p.inv_tau) * wst_s[w][h][ST_LTT];
      wsc_s[w][h] = at;
    }
    float* dst = p.split_st + (((int64_t)b * H + g * G + h) * p.ns_max + s) * ST_N;
#pragma unroll
    for (int k = 0; k < ST_N; ++k) dst[k] = r[k];
  }
  __syncthreads();
  for (int w = 0; w < kWarps; ++w) {
    if (warp == w) {
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        if (h >= G) break;
#pragma unroll
        for (int j = 0; j < DPL; ++j) {
          const float prev = w == 0 ? 0.f : o_s[h][lane * DPL + j];
          o_s[h][lane * DPL + j] = fmaf(wsc_s[w][h], acc[h][j], prev);
        }
      }
    }
    __syncthreads();
  }
  for (int i = threadIdx.x; i < G * D; i += kThreads) {
    const int h = i / D, d = i % D;
    p.split_o[(((int64_t)b * H + g * G + h) * p.ns_max + s) * D + d] = o_s[h][d];
  }
}

// ---------------------------------------------------------------------------
// k_select: grid (granularity ? Hkv : 1, B), 1024 threads, dynamic shared
// memory holding the N_v score keys.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int budget_k(const StepParams& p, float m_max, int nv) {
  if (nv <= 0) return 0;
  switch (p.mode) {
    case MODE_DENSE: return nv;
    case MODE_FIXED_K: return max(0, min(p.fixed_k, nv));
    case MODE_FIXED_RATIO: {
      const long long k = ((long long)p.ratio_ppm * nv + 999999) / 1000000;
      return (int)min((long long)nv, max(k, 1LL));
    }
    default: {
      // Eq. 7 in float32: one rounded product, then the ceiling (exact: the
      // product is at most N_v <= 32768).
      const float prod = __fmul_rn(m_max, (float)nv);
      const long long raw = (long long)ceilf(prod);
      const long long k_lo = ((long long)p.r_lo_ppm * nv + 999999) / 1000000;
      const long long k_hi = max(k_lo, ((long long)p.r_hi_ppm * nv) / 1000000);
      return (int)min((long long)nv, min(max(raw, k_lo), k_hi));
    }
  }
}

// Exclusive prefix sum over the block (all threads must call).
__device__ __forceinline__ int block_excl_scan(int x, int* wsum_s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  if (lane == 31) wsum_s[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? wsum_s[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += n;
    }
    wsum_s[lane] = w;
  }
  __syncthreads();
  const int res = (warp ? wsum_s[warp - 1] : 0) + incl - x;
  __syncthreads();
  return res;
}

__global__ void __launch_bounds__(kSelThreads) k_select(const StepParams p) {
  extern __shared__ uint32_t key_s[];
  __shared__ float hM_s[kMaxHeads], hInv_s[kMaxHeads], hMass_s[kMaxHeads], hMass1_s[kMaxHeads];
  __shared__ unsigned hist_s[256];
  __shared__ int wsum_s[32];
  __shared__ int sh_i[4];

  const int gsel = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int H = p.H;
  const Seq sq = load_seq(p, b, false);
  const int nv = sq.nv;

  // 1. Split statistics -> per-head max, normalisers and masses (Eq. 5, Eq. 6).
  for (int h = tid; h < H; h += kSelThreads) {
    const float* st = p.split_st + ((int64_t)b * H + h) * p.ns_max * ST_N;
    float M = -CUDART_INF_F;
    for (int s = 0; s < p.ns; ++s) M = fmaxf(M, fmaxf(st[s * ST_N + ST_MV], st[s * ST_N + ST_MT]));
    float L1v = 0.f, L1t = 0.f, Ltv = 0.f, Ltt = 0.f;
    for (int s = 0; s < p.ns; ++s) {
      const float* r = st + s * ST_N;
      L1v += exp2_rel(r[ST_MV], M) * r[ST_L1V];
      Ltv += exp2_tau(r[ST_MV], M, p.inv_tau) * r[ST_LTV];
      L1t += exp2_rel(r[ST_MT], M) * r[ST_L1T];
      Ltt += exp2_tau(r[ST_MT], M, p.inv_tau) * r[ST_LTT];
    }
    const float L1 = L1v + L1t, Lt = Ltv + Ltt;
    hM_s[h] = M;
    hInv_s[h] = L1 > 0.f ? 1.f / L1 : 0.f;
    hMass_s[h] = Lt > 0.f ? Ltv / Lt : 0.f;
    hMass1_s[h] = L1 > 0.f ? L1v / L1 : 0.f;
  }
  __syncthreads();

  // 2. Head mean, head max (Sec. 4.3) and the budget (Eq. 7).
  if (tid < 32) {
    float sm = 0.f, mx = 0.f, s1 = 0.f;
    for (int h = tid; h < H; h += 32) {
      sm += hMass_s[h];
      mx = fmaxf(mx, hMass_s[h]);
      s1 += hMass1_s[h];
    }
    sm = warp_sum(sm);
    mx = warp_max(mx);
    s1 = warp_sum(s1);
    if (tid == 0) {
      const int K = min(budget_k(p, mx, nv), p.kept_cap);
      sh_i[0] = K;
      sh_i[1] = 0;
      sh_i[2] = 0;
      if (gsel == 0 && p.mass_stats) {
        float* ms = p.mass_stats + (int64_t)b * 4;
        ms[0] = sm / H; ms[1] = mx; ms[2] = s1 / H; ms[3] = (float)K;
      }
    }
  }
  if (gsel == 0)
    for (int h = tid; h < H; h += kSelThreads) p.mass[(int64_t)b * H + h] = hMass_s[h];

  // 3. Importance S_i (Eq. 2), kept as float bits (S >= 0 orders like its bits).
  const int hbeg = p.granularity ? gsel * p.G : 0;
  const int hcnt = p.granularity ? p.G : H;
  __syncthreads();
  const int K = sh_i[0];
  unsigned bad = 0;
  for (int i = tid; i < nv; i += kSelThreads) {
    float a = 0.f;
    for (int hh = 0; hh < hcnt; ++hh) {
      const int h = hbeg + hh;
      const float z = p.z_ws[((int64_t)b * H + h) * p.max_visual + i];
      a = fmaf(exp2_rel(z, hM_s[h]), hInv_s[h], a);
    }
    const float sc = a / (float)hcnt;
    if (!isfinite(sc)) bad = 1;
    key_s[i] = __float_as_uint(sc);
  }
  if (bad) atomicOr(p.err, ERR_NONFINITE);

  const int nsel = p.granularity ? p.Hkv : 1;
  int32_t* kept = p.kept_idx + ((int64_t)b * nsel + gsel) * p.kept_cap;
  if (tid == 0) p.kept_count[(int64_t)b * nsel + gsel] = K;
  __syncthreads();

  // 4. Radix select of the K-th largest key, 8 bits per pass from the top.
  const bool take_all = K >= nv;
  uint32_t theta = 0;
  unsigned krem = 0;
  if (K > 0 && !take_all) {
    uint32_t prefix = 0, mask = 0;
    krem = (unsigned)K;
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = tid; i < 256; i += kSelThreads) hist_s[i] = 0;
      __syncthreads();
      for (int i = tid; i < nv; i += kSelThreads) {
        const uint32_t k = key_s[i];
        if ((k & mask) == prefix) atomicAdd(&hist_s[(k >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (tid < 32) {
        // Lane L owns digits 255-8L ... 248-8L (descending).
        unsigned c[8], tot = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) { c[j] = hist_s[255 - 8 * tid - j]; tot += c[j]; }
        unsigned incl = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned n = __shfl_up_sync(0xffffffffu, incl, o);
          if (tid >= o) incl += n;
        }
        const unsigned excl = incl - tot;
        if (excl < krem && krem <= incl) {
          unsigned run = excl;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (run + c[j] >= krem) { sh_i[1] = 255 - 8 * tid - j; sh_i[2] = (int)run; break; }
            run += c[j];
          }
        }
      }
      __syncthreads();
      krem -= (unsigned)sh_i[2];
      prefix |= (uint32_t)sh_i[1] << shift;
      mask |= 255u << shift;
      __syncthreads();
    }
    theta = prefix;  // the K-th largest key; krem keys equal to it are kept
  }

  // 5. Ascending compaction: keys above theta, plus the first krem equal keys.
  if (K > 0) {
    const int per = (nv + kSelThreads - 1) / kSelThreads;
    const int i0 = min(nv, tid * per), i1 = min(nv, i0 + per);
    int n_eq = 0;
    if (!take_all)
      for (int i = i0; i < i1; ++i) n_eq += key_s[i] == theta;
    const int eq_before = block_excl_scan(n_eq, wsum_s);
    int n_sel = 0;
    {
      int r = eq_before;
      for (int i = i0; i < i1; ++i) {
        const uint32_t k = key_s[i];
        const bool sel = take_all || k > theta || (k == theta && (unsigned)r < krem);
        r += k == theta;
        n_sel += sel;
      }
    }
    int o = block_excl_scan(n_sel, wsum_s);
    int r = eq_before;
    for (int i = i0; i < i1; ++i) {
      const uint32_t k = key_s[i];
      const bool sel = take_all || k > theta || (k == theta && (unsigned)r < krem);
      r += k == theta;
      if (sel && o < K) kept[o++] = i;
    }
  }
  for (int i = max(K, 0) + tid; i < p.kept_cap; i += kSelThreads) kept[i] = -1;
}

// ---------------------------------------------------------------------------
// k_gather: grid (nk, Hkv, B), 128 threads.  Chunk c of the kept list is
// staged 64 tokens at a time: indices, V-row addresses and logits to shared
// memory, then every thread accumulates one 16-byte slice of the V rows of
// every (128 / slices-per-row)-th token.  The last chunk of (b, kv-head) to
// finish merges all partials and writes the output.
// ---------------------------------------------------------------------------
template <typename T, int D, int GM>
__global__ void __launch_bounds__(kThreads) k_gather(const StepParams p) {
  constexpr int CH = 16 / sizeof(T);          // elements per 16-byte slice
  constexpr int CPR = D / CH;                 // slices per row
  constexpr int SLOTS = kThreads / CPR;       // tokens processed side by side
  static_assert(kThreads % CPR == 0, "row slicing");
  const int c = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.G, H = p.H;
  const int slot = tid / CPR, ch = tid % CPR;

  __shared__ const T* vrow_s[kGatherTile];
  __shared__ float pz_s[GM][kGatherTile];
  __shared__ float run_s[GM][3];  // running max, running sum, rescale factor
  __shared__ __align__(16) float o_s[GM][D];
  __shared__ float fin_s[GM];
  __shared__ int last_s;

  const Seq sq = load_seq(p, b, false);
  const int sel = p.granularity ? b * p.Hkv + g : b;
  const int K = max(0, min(__ldg(p.kept_count + sel), min(sq.nv, p.kept_cap)));
  const int32_t* kept = p.kept_idx + (int64_t)sel * p.kept_cap;
  const int per = (K + p.nk - 1) / max(p.nk, 1);
  const int j0 = min(K, c * per), j1 = min(K, j0 + per);

  if (tid < GM) { run_s[tid][0] = -CUDART_INF_F; run_s[tid][1] = 0.f; run_s[tid][2] = 0.f; }
  float acc[GM][CH];
#pragma unroll
  for (int h = 0; h < GM; ++h)
#pragma unroll
    for (int e = 0; e < CH; ++e) acc[h][e] = 0.f;
  unsigned err = 0;
  __syncthreads();

  for (int jt = j0; jt < j1; jt += kGatherTile) {
    const int n = min(kGatherTile, j1 - jt);
    // A. stage indices, V rows and logits
    for (int t = tid; t < kGatherTile; t += kThreads) {
      const T* vr = nullptr;
      int i = -1;
      if (t < n) {
        i = kept[jt + t];
        if (i < 0 || i >= sq.nv) { err |= ERR_KEPT; i = -1; }
        else {
          vr = kv_row<T>(p.v, p, b, g, sq.vs + i);
          if (!vr) err |= ERR_PAGE;
        }
      }
      vrow_s[t] = vr;
      for (int h = 0; h < G; ++h)
        pz_s[h][t] = vr ? p.z_ws[((int64_t)b * H + g * G + h) * p.max_visual + i] : -CUDART_INF_F;
    }
    __syncthreads();
    // B. per-head tile max and running rescale (warp w handles heads w, w+4, ...)
    for (int h = warp; h < G; h += kWarps) {
      const float z0 = pz_s[h][lane], z1 = pz_s[h][lane + 32];
      const float mt = warp_max(fmaxf(z0, z1));
      const float mo = run_s[h][0];
      const float mn = fmaxf(mo, mt);
      const float e0 = exp2_rel(z0, mn), e1 = exp2_rel(z1, mn);
      const float ssum = warp_sum(e0 + e1);
      pz_s[h][lane] = e0;
      pz_s[h][lane + 32] = e1;
      if (lane == 0) {
        const float a = exp2_rel(mo, mn);
        run_s[h][0] = mn;
        run_s[h][1] = run_s[h][1] * a + ssum;
        run_s[h][2] = a;
      }
    }
    __syncthreads();
    // C. P.V over the staged rows
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      if (h >= G) break;
      const float a = run_s[h][2];
#pragma unroll
      for (int e = 0; e < CH; ++e) acc[h][e] *= a;
    }
#pragma unroll 4
    for (int t = slot; t < n; t += SLOTS) {
      const T* vr = vrow_s[t];
      if (!vr) continue;
      float vv[CH];
      load_f<CH>(vr + ch * CH, vv);
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        if (h >= G) break;
        const float pr = pz_s[h][t];
#pragma unroll
        for (int e = 0; e < CH; ++e) acc[h][e] = fmaf(pr, vv[e], acc[h][e]);
      }
    }
    __syncthreads();
  }
  if (err) atomicOr(p.err, err);

  // Reduce the token slots (fixed order) and publish this chunk's partial.
  for (int sl = 0; sl < SLOTS; ++sl) {
    if (slot == sl) {
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        if (h >= G) break;
#pragma unroll
        for (int e = 0; e < CH; ++e) {
          const float prev = sl == 0 ? 0.f : o_s[h][ch * CH + e];
          o_s[h][ch * CH + e] = prev + acc[h][e];
        }
      }
    }
    __syncthreads();
  }
  const int64_t pbase = ((int64_t)b * p.Hkv + g) * p.nk_max;
  for (int i = tid; i < G * D; i += kThreads)
    p.gpart_o[(pbase + c) * G * D + i] = o_s[i / D][i % D];
  if (tid < G) {
    p.gpart_st[((pbase + c) * G + tid) * 2 + 0] = run_s[tid][0];
    p.gpart_st[((pbase + c) * G + tid) * 2 + 1] = run_s[tid][1];
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const unsigned t = atomicAdd(p.tickets + (int64_t)b * p.Hkv + g, 1u);
    last_s = t == (unsigned)p.nk - 1u;
  }
  __syncthreads();
  if (!last_s) return;
  __threadfence();

  // Last chunk: merge text splits and kept chunks in log-sum-exp form.
  if (tid < G) {
    const int h = tid;
    float M = -CUDART_INF_F;
    const float* st = p.split_st + ((int64_t)b * H + g * G + h) * p.ns_max * ST_N;
    for (int s = 0; s < p.ns; ++s) M = fmaxf(M, st[s * ST_N + ST_MT]);
    for (int k = 0; k < p.nk; ++k) M = fmaxf(M, __ldcg(p.gpart_st + ((pbase + k) * G + h) * 2));
    fin_s[h] = M;
  }
  __syncthreads();
  for (int i = tid; i < G * D; i += kThreads) {
    const int h = i / D, d = i % D;
    const float M = fin_s[h];
    const int64_t hrow = (int64_t)b * H + g * G + h;
    const float* st = p.split_st + hrow * p.ns_max * ST_N;
    const float* so = p.split_o + hrow * p.ns_max * D + d;
    float num = 0.f, den = 0.f;
    for (int s = 0; s < p.ns; ++s) {
      const float w = exp2_rel(st[s * ST_N + ST_MT], M);
      num = fmaf(w, so[(int64_t)s * D], num);
      den = fmaf(w, st[s * ST_N + ST_L1T], den);
    }
    for (int k = 0; k < p.nk; ++k) {
      const float* gs = p.gpart_st + ((pbase + k) * G + h) * 2;
      const float w = exp2_rel(__ldcg(gs), M);
      num = fmaf(w, __ldcg(p.gpart_o + (pbase + k) * G * D + i), num);
      den = fmaf(w, __ldcg(gs + 1), den);
    }
    reinterpret_cast<T*>(p.out)[hrow * D + d] = from_f<T>(den > 0.f ? num / den : 0.f);
  }
  if (tid == 0) p.tickets[(int64_t)b * p.Hkv + g] = 0u;
}

template <typename T, int D>
cudaError_t launch_score_td(const StepParams& p, cudaStream_t st) {
  const dim3 grid(p.ns, p.Hkv, p.B);
  if (p.G <= 4) k_score<T, D, 4><<<grid, kThreads, 0, st>>>(p);
  else if (p.G <= 8) k_score<T, D, 8><<<grid, kThreads, 0, st>>>(p);
  else k_score<T, D, 16><<<grid, kThreads, 0, st>>>(p);
  return cudaGetLastError();
}

template <typename T, int D>
cudaError_t launch_gather_td(const StepParams& p, cudaStream_t st) {
  const dim3 grid(p.nk, p.Hkv, p.B);
  if (p.G <= 4) k_gather<T, D, 4><<<grid, kThreads, 0, st>>>(p);
  else if (p.G <= 8) k_gather<T, D, 8><<<grid, kThreads, 0, st>>>(p);
  else k_gather<T, D, 16><<<grid, kThreads, 0, st>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score(const StepParams& p, cudaStream_t st) {
  if (p.dtype == 0)
    return p.D == 128 ? launch_score_td<__nv_bfloat16, 128>(p, st) : launch_score_td<__nv_bfloat16, 64>(p, st);
  return p.D == 128 ? launch_score_td<float, 128>(p, st) : launch_score_td<float, 64>(p, st);
}

cudaError_t launch_gather(const StepParams& p, cudaStream_t st) {
  if (p.dtype == 0)
    return p.D == 128 ? launch_gather_td<__nv_bfloat16, 128>(p, st) : launch_gather_td<__nv_bfloat16, 64>(p, st);
  return p.D == 128 ? launch_gather_td<float, 128>(p, st) : launch_gather_td<float, 64>(p, st);
}

size_t select_smem_bytes(int max_visual) { return (size_t)(max_visual > 0 ? max_visual : 1) * sizeof(uint32_t); }

cudaError_t launch_select(const StepParams& p, cudaStream_t st) {
  const dim3 grid(p.granularity ? p.Hkv : 1, p.B);
  k_select<<<grid, kSelThreads, select_smem_bytes(p.max_visual), st>>>(p);
  return cudaGetLastError();
}

cudaError_t configure_kernels(int max_visual) {
  return cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)select_smem_bytes(max_visual));
}

cudaError_t raise_select_smem(int max_visual) {
  cudaFuncAttributes attr;
  cudaError_t e = cudaFuncGetAttributes(&attr, k_select);
  if (e != cudaSuccess) return e;
  const int need = (int)select_smem_bytes(max_visual);
  if (attr.maxDynamicSharedSizeBytes >= need) return cudaSuccess;
  return cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, need);
}

}  // namespace vp
