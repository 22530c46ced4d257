// CUDA kernels of one VisionPulse decode step (arxiv 2605.31457, Sec. 4.2-4.3).
//
//   k_score   per (sequence, kv-head, split): logits of the G query heads of the
//             kv-head against every key of the split (Eq. 6's Z).  Visual logits
//             go to the workspace; visual and text tokens keep separate online
//             softmax statistics at tau = 1 and at tau (the two sums of Eq. 6);
//             text tokens also accumulate their unnormalised attention output.
//   k_select  per sequence (or per kv-head), a cluster of up to 8 CTAs: merges
//             the split statistics into the visual mass per head (Eq. 5) and
//             its head-max (Sec. 4.3) and the budget K_t (Eq. 7 + clamp of
//             Sec. 5.2); every CTA computes the importance score S_i (Eq. 2) of
//             a slice of the visual tokens into rank 0's shared memory, which
//             then finds the Top-K_t set (Eq. 3) by radix select, ties to the
//             lower index, emitted in ascending order.
//   k_gather  per (sequence, kv-head): CTA c attends over chunk c of the kept
//             visual tokens, reading V only for them, and merges slice c of the
//             text partials; the last CTA to finish combines everything in
//             log-sum-exp form and writes the output (Sec. 4.2, Sec. 5.7).
//
// Logits are carried in log2 units (z * log2 e) so that every exponential is
// one exp2f: exp(z - m) = exp2(z2 - m2), exp((z - m) / tau) = exp2((z2 - m2) / tau).
//
// Every kernel may be launched as a programmatic dependent of the preceding
// kernel on the stream: it reads nothing that kernel writes before
// griddepcontrol.wait.  The slice gather kernel reads the call's inputs and
// the score kernel's partials before its wait: the select kernel between them
// lets its dependents start only after its own wait on the score kernel, so
// both are complete by then.  Each kernel also lets its own dependent start
// only after that wait, so the next call cannot overwrite the workspace early.
#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math_constants.h>
#include <stdint.h>

#include <type_traits>

#include "vp_internal.h"

namespace cg = cooperative_groups;

namespace vp {
namespace {

constexpr int kWarps = 8;                 // warps of a score CTA
constexpr int kThreads = 32 * kWarps;
constexpr int kStages = 3;                // TMA ring depth per warp
constexpr int kTile = 16;                 // tokens per tile
constexpr int kSelSliceSmall = 2048;  // longest slice per select rank for 512 threads
constexpr int kMaxHeads = 128;
constexpr int kGatherThreads = 256;
constexpr int kGatherWarps = kGatherThreads / 32;
constexpr int kGatherTile = 64;           // kept tokens staged per round in k_gather
constexpr unsigned long long kWaitLimitNs = 1000000000ull;  // an mbarrier wait gives up after 1 s

// Budget modes (numbering of vp_budget_mode in include/vp.h).
enum { MODE_ADAPTIVE = 0, MODE_FIXED_RATIO = 1, MODE_FIXED_K = 2, MODE_DENSE = 3, MODE_TOP_P = 4 };

// ------------------------------------------------------------------ helpers

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

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
// Reductions over the 8 lanes that share lane % 4 (the mma "group" axis).
__device__ __forceinline__ float group_max(float x) {
  x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 4));
  x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 8));
  return fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 16));
}
__device__ __forceinline__ float group_sum(float x) {
  x += __shfl_xor_sync(0xffffffffu, x, 4);
  x += __shfl_xor_sync(0xffffffffu, x, 8);
  return x + __shfl_xor_sync(0xffffffffu, x, 16);
}

// exp2 by the hardware approximation (ex2.approx: a few ulp, subnormal
// results flushed to 0), one instruction: the statistics merges run it on
// every split record, in kernels whose launches are latency-bound.
__device__ __forceinline__ float ex2_hw(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// exp2(a - m) with an empty term (a = -inf) giving exactly 0.
__device__ __forceinline__ float exp2_rel(float a, float m) {
  return a == -CUDART_INF_F ? 0.f : ex2_hw(a - m);
}
__device__ __forceinline__ float exp2_tau(float a, float m, float inv_tau) {
  return a == -CUDART_INF_F ? 0.f : ex2_hw((a - m) * inv_tau);
}

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
    const float4 v = __ldg(reinterpret_cast<const float4*>(p));
    f[0] = v.x; f[1] = v.y; f[2] = v.z; f[3] = v.w;
  } else if constexpr (N == 2) {
    const float2 v = __ldg(reinterpret_cast<const float2*>(p));
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
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
    bf2(v.x, f[0], f[1]); bf2(v.y, f[2], f[3]); bf2(v.z, f[4], f[5]); bf2(v.w, f[6], f[7]);
  } else if constexpr (N == 4) {
    const uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
    bf2(v.x, f[0], f[1]); bf2(v.y, f[2], f[3]);
  } else {
    bf2(__ldg(reinterpret_cast<const unsigned int*>(p)), f[0], f[1]);
  }
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t r;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
  return r;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}
// D = A * B + D, m16n8k16, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ unsigned smem_u32(const void* p) {
  return static_cast<unsigned>(__cvta_generic_to_shared(p));
}
// Four 8x8 b16 matrices from shared memory; lane l gives the row address of
// row l % 8 of matrix l / 8.
__device__ __forceinline__ void ldsm_x4(unsigned addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(unsigned addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}

// ---- mbarrier + bulk (TMA) copies
__device__ __forceinline__ void mbar_init(uint64_t* bar, unsigned count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() { asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory"); }
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, unsigned bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, unsigned parity) {
  unsigned ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}
__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait for a phase of an mbarrier; false if it did not complete
// within kWaitLimitNs.  try_wait itself suspends the thread until the phase
// completes or a hardware time slice ends, so the loop needs no sleep.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, unsigned parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (;;) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > kWaitLimitNs) return false;
  }
}
// A 4-byte load through L2 issued where it stands in the program (the
// compiler may not move it next to the value's first use), for prefetching.
__device__ __forceinline__ int ldcg_now(const int* ptr) {
  int v;
  asm volatile("ld.global.cg.s32 %0, [%1];\n" : "=r"(v) : "l"(ptr));
  return v;
}
// Orders this thread's earlier generic-proxy shared-memory accesses before
// later asynchronous-proxy (bulk copy) writes to the same memory.
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, unsigned bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n"
               ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}

// 16- and 4-byte asynchronous copies global -> shared (LSU path), and the
// arrive-on that completes an mbarrier phase once this thread's earlier such
// copies have landed; the barrier's pending count is raised first, so the
// arrival needs no room in the barrier's count (a normal arrival still
// completes the phase once the copies have landed).
__device__ __forceinline__ void cp_async16(unsigned dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(unsigned dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_arrive_counted(uint64_t* bar) {
  asm volatile("cp.async.mbarrier.arrive.shared::cta.b64 [%0];\n" ::"r"(smem_u32(bar)) : "memory");
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

// Token ranges of split s: the sequence's work (visual tokens weigh 1, text
// tokens 2) cut into ns equal parts.  Visual range [va, vb) is relative to the
// span start; text range [ta, tb) indexes the text tokens in cache order.
struct SplitRange {
  int va, vb, ta, tb;
};
__device__ __forceinline__ SplitRange split_range(const Seq& sq, int s, int ns) {
  const int W = sq.nv + 2 * sq.tl;
  const int per = (W + ns - 1) / ns;
  const int w0 = min(W, s * per), w1 = min(W, w0 + per);
  SplitRange r;
  r.va = min(w0, sq.nv);
  r.vb = min(w1, sq.nv);
  r.ta = (max(w0, sq.nv) - sq.nv + 1) >> 1;
  r.tb = (max(w1, sq.nv) - sq.nv + 1) >> 1;
  return r;
}
__device__ __forceinline__ int text_pos(const Seq& sq, int ti) { return ti < sq.vs ? ti : ti + sq.nv; }

// Merges n statistic records (`stride` floats apart); writes the text weight of
// each record to wt[k * wstride].
__device__ __forceinline__ void merge_stats(const float* recs, int n, int stride, float inv_tau, float* out,
                                            float* wt, int wstride) {
  float Mv = -CUDART_INF_F, Mt = -CUDART_INF_F;
  for (int k = 0; k < n; ++k) {
    Mv = fmaxf(Mv, recs[k * stride + ST_MV]);
    Mt = fmaxf(Mt, recs[k * stride + ST_MT]);
  }
  float l1v = 0.f, ltv = 0.f, l1t = 0.f, ltt = 0.f;
  for (int k = 0; k < n; ++k) {
    const float* r = recs + k * stride;
    l1v += exp2_rel(r[ST_MV], Mv) * r[ST_L1V];
    ltv += exp2_tau(r[ST_MV], Mv, inv_tau) * r[ST_LTV];
    const float at = exp2_rel(r[ST_MT], Mt);
    l1t += at * r[ST_L1T];
    ltt += exp2_tau(r[ST_MT], Mt, inv_tau) * r[ST_LTT];
    wt[k * wstride] = at;
  }
  out[ST_MT] = Mt; out[ST_L1T] = l1t; out[ST_LTT] = ltt; out[3] = 0.f;
  out[ST_MV] = Mv; out[ST_L1V] = l1v; out[ST_LTV] = ltv; out[7] = 0.f;
}

// ------------------------------------------------------- score epilogue
// Shared by the score kernels: per-warp statistics wst[w][h][ST_N] and text
// outputs (warp w at ow + w * ow_stride, [GM][D]) are merged into the CTA's
// partial and written to split slot s.
template <int GM, int D, int NW = kWarps>
struct ScoreTail {
  float cst[GM][ST_N];
  float wsc[NW][GM];
};

// NW warp records are merged; the kernel runs NTHR threads.
template <int GM, int D, int NW = kWarps, int NTHR = kThreads>
__device__ void score_epilogue(const StepParams& p, int b, int g, int s, const float (*wst)[GM][ST_N],
                               const float* ow, int ow_stride, ScoreTail<GM, D, NW>& tl) {
  const int tid = threadIdx.x, G = p.G;
  constexpr int D4 = D / 4;
  __syncthreads();
  if (tid < G) merge_stats(&wst[0][tid][0], NW, GM * ST_N, p.inv_tau, tl.cst[tid], &tl.wsc[0][tid], GM);
  __syncthreads();
  const int64_t rec0 = ((int64_t)b * p.H + g * G) * p.nsp_max + s;  // slot of head 0
  for (int i = tid; i < G * D4; i += NTHR) {
    const int h = i / D4, d = 4 * (i % D4);
    float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float a = tl.wsc[w][h];
      const float4 v = *reinterpret_cast<const float4*>(ow + w * ow_stride + h * D + d);
      o.x = fmaf(a, v.x, o.x); o.y = fmaf(a, v.y, o.y); o.z = fmaf(a, v.z, o.z); o.w = fmaf(a, v.w, o.w);
    }
    *reinterpret_cast<float4*>(p.split_o + (rec0 + (int64_t)h * p.nsp_max) * D + d) = o;
  }
  if (tid < 2 * G) {
    const int h = tid >> 1, half = tid & 1;
    *reinterpret_cast<float4*>(p.split_st + (rec0 + (int64_t)h * p.nsp_max) * ST_N + 4 * half) =
        *reinterpret_cast<const float4*>(&tl.cst[h][4 * half]);
  }
}

// ---------------------------------------------------------------------------
// k_score_mma (bf16).  Each warp streams 16-token tiles through a 3-stage ring
// in shared memory: one lane arms the stage's mbarrier with the tile's byte
// count, then lane r issues a bulk (TMA) copy of token row r of K (and of V
// for text tiles) into a row padded to 2D + 16 bytes, which makes the
// ldmatrix reads below free of bank conflicts.  Both contractions run on the
// tensor cores with mma.m16n8k16:
//   QK:  A = K tile (16 tokens x 16 dims, ldmatrix), B = q^T (16 dims x 8 heads).
//   PV:  A = V^T (16 dims x 16 tokens, ldmatrix.trans), B = P^T (16 tokens x
//        8 heads), taken from the QK accumulators with four shuffles.
// Lane (r = lane/4, c = lane%4) keeps the softmax statistics of heads 2c, 2c+1
// of each 8-head tile and accumulates the same heads' outputs, so rescaling
// the accumulators needs no communication.
// ---------------------------------------------------------------------------
template <int D, int NT>
struct MmaCfg {
  static constexpr int GM = 8 * NT;
  static constexpr int KS = D / 16;                    // QK k-steps
  static constexpr int MT = D / 16;                    // PV m-tiles (16 dims each)
  static constexpr int RP = 2 * D + 16;                // padded row pitch (bytes)
  static constexpr int TILE_BYTES = kTile * RP;
  static constexpr int STAGE = 2 * TILE_BYTES;         // K tile + V tile
  static constexpr int RING = kStages * STAGE;         // per warp
  static constexpr int OFF_BAR = kWarps * RING;
  static constexpr int OFF_TAIL = OFF_BAR + kWarps * kStages * 8;
  static constexpr int OFF_WST = OFF_TAIL + (int)sizeof(ScoreTail<GM, D>);
  static constexpr size_t SMEM = (size_t)OFF_WST + sizeof(float) * kWarps * GM * ST_N;
  static_assert(GM * D * 4 <= RING, "a warp's text partial must fit in its ring");
  static_assert(OFF_TAIL % 16 == 0 && OFF_WST % 16 == 0, "alignment");
};

template <int D, int NT>
__global__ void __launch_bounds__(kThreads) k_score_mma(const __grid_constant__ StepParams p) {
  using C = MmaCfg<D, NT>;
  constexpr int GM = C::GM;
  extern __shared__ __align__(128) unsigned char smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gr = lane >> 2, tg = lane & 3;  // mma group id / thread in group
  const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  unsigned char* ring = smem + warp * C::RING;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR) + warp * kStages;
  auto& tail = *reinterpret_cast<ScoreTail<GM, D>*>(smem + C::OFF_TAIL);
  auto wst = reinterpret_cast<float (*)[GM][ST_N]>(smem + C::OFF_WST);

  if (lane == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(bars + i, 1);
    mbar_fence_init();
  }
  __syncwarp();
  pdl_wait();
  const int G = p.G, H = p.H;
  const Seq sq = load_seq(p, b, s == 0 && g == 0);
  const SplitRange rg = split_range(sq, s, p.ns);
  const int n_vt = (rg.vb - rg.va + kTile - 1) / kTile;
  const int n_tt = (rg.tb - rg.ta + kTile - 1) / kTile;
  const int n_tiles = n_vt + n_tt;
  const int my_n = warp < n_tiles ? (n_tiles - warp + kWarps - 1) / kWarps : 0;

  unsigned err = 0;
  int issued = 0;  // tiles whose copies were issued
  // Arms stage k % kStages and issues the bulk copies of this warp's k-th tile.
  auto issue = [&](int k) {
    if (k >= my_n) return;
    issued = k + 1;
    const int j = warp + kWarps * k;
    const bool text = j >= n_vt;
    const int first = text ? rg.ta + (j - n_vt) * kTile : rg.va + j * kTile;
    const int cnt = min(kTile, (text ? rg.tb : rg.vb) - first);
    uint64_t* bar = bars + k % kStages;
    unsigned char* kt = ring + (k % kStages) * C::STAGE;
    const __nv_bfloat16* kr = nullptr;
    const __nv_bfloat16* vr = nullptr;
    if (lane < cnt) {
      const int pos = text ? text_pos(sq, first + lane) : sq.vs + first + lane;
      kr = kv_row<__nv_bfloat16>(p.k, p, b, g, pos);
      if (text) vr = kv_row<__nv_bfloat16>(p.v, p, b, g, pos);
      if (!kr || (text && !vr)) { err |= ERR_PAGE; kr = vr = nullptr; }
    }
    const unsigned nk = __popc(__ballot_sync(0xffffffffu, kr != nullptr));
    const unsigned nvr = __popc(__ballot_sync(0xffffffffu, vr != nullptr));
    fence_proxy_async();
    if (lane == 0) mbar_expect_tx(bar, (nk + nvr) * (2 * D));
    __syncwarp();
    if (kr) bulk_g2s(kt + lane * C::RP, kr, 2 * D, bar);
    if (vr) bulk_g2s(kt + C::TILE_BYTES + lane * C::RP, vr, 2 * D, bar);
  };
#pragma unroll
  for (int k = 0; k < kStages - 1; ++k) issue(k);

  // q^T fragments (natural dimension order): head 8n + gr, dims 16ks + 2tg (+8).
  uint32_t qf[NT][C::KS][2];
  const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(p.q) + ((int64_t)b * H + g * G) * D;
#pragma unroll
  for (int n = 0; n < NT; ++n) {
    const int h = 8 * n + gr;
    const uint32_t* qr = reinterpret_cast<const uint32_t*>(qb + h * D);
#pragma unroll
    for (int ks = 0; ks < C::KS; ++ks) {
      qf[n][ks][0] = h < G ? __ldg(qr + 8 * ks + tg) : 0u;
      qf[n][ks][1] = h < G ? __ldg(qr + 8 * ks + 4 + tg) : 0u;
    }
  }

  float m_v[NT][2], l1v[NT][2], ltv[NT][2], m_t[NT][2], l1t[NT][2], ltt[NT][2];
  float acc[NT][C::MT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      m_v[n][j] = m_t[n][j] = -CUDART_INF_F;
      l1v[n][j] = ltv[n][j] = l1t[n][j] = ltt[n][j] = 0.f;
    }
#pragma unroll
    for (int mi = 0; mi < C::MT; ++mi)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[n][mi][e] = 0.f;
  }

  // ldmatrix row addresses.  K (A operand, rows = tokens): matrix l / 8 covers
  // tokens 8 * ((l / 8) & 1) + (0..7) and dims 8 * (l / 16) + (0..7) of the 16 x 16
  // block.  V^T (A operand via .trans, rows = dims): matrix l / 8 covers
  // tokens 8 * (l / 16) + (0..7) and dims 8 * ((l / 8) & 1) + (0..7).
  const int krow = (lane & 7) + 8 * ((lane >> 3) & 1), kcol = 8 * (lane >> 4);
  const int vrow = (lane & 7) + 8 * (lane >> 4), vcol = 8 * ((lane >> 3) & 1);
  bool timed_out = false;
  int consumed = 0;  // tiles whose copies were waited for
  for (int k = 0; k < my_n; ++k) {
    // Tile k + 2 goes into the stage tile k - 1 used (consumed last iteration),
    // so all three stages are in flight while this warp waits for tile k.
    issue(k + kStages - 1);
    if (!mbar_wait(bars + k % kStages, (k / kStages) & 1)) { timed_out = true; break; }
    consumed = k + 1;
    const int j = warp + kWarps * k;
    const bool text = j >= n_vt;
    const int first = text ? rg.ta + (j - n_vt) * kTile : rg.va + j * kTile;
    const int cnt = min(kTile, (text ? rg.tb : rg.vb) - first);
    const unsigned kt = smem_u32(ring + (k % kStages) * C::STAGE);
    const unsigned vt = kt + C::TILE_BYTES;

    // ---- QK on the tensor cores
    float c[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) c[n][e] = 0.f;
#pragma unroll
    for (int ks = 0; ks < C::KS; ++ks) {
      uint32_t a0, a1, a2, a3;
      ldsm_x4(kt + krow * C::RP + (16 * ks + kcol) * 2, a0, a1, a2, a3);
#pragma unroll
      for (int n = 0; n < NT; ++n) mma_bf16(c[n], a0, a1, a2, a3, qf[n][ks][0], qf[n][ks][1]);
    }
    // c[n][e]: token row gr + 8 * (e >> 1), head 8n + 2tg + (e & 1).  Rows past
    // cnt were not copied (stale shared memory): they are masked here.
    const bool ok0 = gr < cnt, ok1 = gr + 8 < cnt;
    float zz[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const bool ok = (e < 2 ? ok0 : ok1) && (8 * n + 2 * tg + (e & 1)) < G;
        zz[n][e] = ok ? c[n][e] * p.c_log2 : -CUDART_INF_F;
      }

    if (!text) {
      float* zrow = p.z_ws + ((int64_t)b * p.max_visual + first) * p.hp + g * G;
#pragma unroll
      for (int n = 0; n < NT; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int h = 8 * n + 2 * tg + (e & 1), r = gr + 8 * (e >> 1);
          if (h < G && r < cnt) zrow[(int64_t)r * p.hp + h] = zz[n][e];
        }
#pragma unroll
      for (int n = 0; n < NT; ++n)
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const float mn = fmaxf(m_v[n][jj], group_max(fmaxf(zz[n][jj], zz[n][jj + 2])));
          if (mn > m_v[n][jj]) {
            l1v[n][jj] *= exp2_rel(m_v[n][jj], mn);
            ltv[n][jj] *= exp2_tau(m_v[n][jj], mn, p.inv_tau);
            m_v[n][jj] = mn;
          }
          if (mn != -CUDART_INF_F) {
            l1v[n][jj] += exp2f(zz[n][jj] - mn) + exp2f(zz[n][jj + 2] - mn);
            ltv[n][jj] += exp2f((zz[n][jj] - mn) * p.inv_tau) + exp2f((zz[n][jj + 2] - mn) * p.inv_tau);
          }
        }
    } else {
      uint32_t pb[NT][2];
#pragma unroll
      for (int n = 0; n < NT; ++n) {
        float pr[4];
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const float mn = fmaxf(m_t[n][jj], group_max(fmaxf(zz[n][jj], zz[n][jj + 2])));
          if (mn > m_t[n][jj]) {
            const float a = exp2_rel(m_t[n][jj], mn);
            l1t[n][jj] *= a;
            ltt[n][jj] *= exp2_tau(m_t[n][jj], mn, p.inv_tau);
#pragma unroll
            for (int mi = 0; mi < C::MT; ++mi) {
              acc[n][mi][jj] *= a;
              acc[n][mi][jj + 2] *= a;
            }
            m_t[n][jj] = mn;
          }
          pr[jj] = pr[jj + 2] = 0.f;
          if (mn != -CUDART_INF_F) {
            pr[jj] = exp2f(zz[n][jj] - mn);
            pr[jj + 2] = exp2f(zz[n][jj + 2] - mn);
            l1t[n][jj] += pr[jj] + pr[jj + 2];
            ltt[n][jj] += exp2f((zz[n][jj] - mn) * p.inv_tau) + exp2f((zz[n][jj + 2] - mn) * p.inv_tau);
          }
        }
        // P^T fragment for head 8n + gr: tokens 2tg, 2tg + 1 live in the first
        // halves of lanes 8tg + gr/2 and 8tg + 4 + gr/2, tokens 2tg + 8, 2tg + 9
        // in their second halves; the half is chosen by the head's parity.
        const uint32_t p01 = pack_bf16(pr[0], pr[1]), p23 = pack_bf16(pr[2], pr[3]);
        const int src0 = 8 * tg + (gr >> 1), src1 = src0 + 4;
        const uint32_t x0 = __shfl_sync(0xffffffffu, p01, src0), x1 = __shfl_sync(0xffffffffu, p01, src1);
        const uint32_t x2 = __shfl_sync(0xffffffffu, p23, src0), x3 = __shfl_sync(0xffffffffu, p23, src1);
        const uint32_t sel = (gr & 1) ? 0x7632u : 0x5410u;
        pb[n][0] = prmt(x0, x1, sel);
        pb[n][1] = prmt(x2, x3, sel);
      }
      // ---- PV on the tensor cores.  V rows past cnt hold stale data: their
      // probabilities are 0, but a stale NaN would still poison the product, so
      // the fragment words of those rows are zeroed.
      const bool vok_lo0 = 2 * tg < cnt, vok_lo1 = 2 * tg + 1 < cnt;
      const bool vok_hi0 = 2 * tg + 8 < cnt, vok_hi1 = 2 * tg + 9 < cnt;
      const bool full = cnt == kTile;
#pragma unroll
      for (int mi = 0; mi < C::MT; ++mi) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4_t(vt + vrow * C::RP + (16 * mi + vcol) * 2, a0, a1, a2, a3);
        if (!full) {
          // a0/a1: tokens 2tg (low half), 2tg + 1 (high half); a2/a3: tokens 2tg + 8, 2tg + 9.
          const uint32_t mlo = (vok_lo0 ? 0x0000ffffu : 0u) | (vok_lo1 ? 0xffff0000u : 0u);
          const uint32_t mhi = (vok_hi0 ? 0x0000ffffu : 0u) | (vok_hi1 ? 0xffff0000u : 0u);
          a0 &= mlo; a1 &= mlo; a2 &= mhi; a3 &= mhi;
        }
#pragma unroll
        for (int n = 0; n < NT; ++n) mma_bf16(acc[n][mi], a0, a1, a2, a3, pb[n][0], pb[n][1]);
      }
    }
    __syncwarp();
  }
  // After a timed-out wait, the copies still in flight must land (or time out
  // again) before the ring is reused for the partials or the CTA exits.
  for (int k = consumed; k < issued; ++k)
    if (!mbar_wait(bars + k % kStages, (k / kStages) & 1)) timed_out = true;
  pdl_trigger();
  if (timed_out) err |= ERR_TIMEOUT;
  if (err) atomicOr(p.err, err);

  // Warp partials: statistics to wst, text outputs into this warp's (now idle) ring.
#pragma unroll
  for (int n = 0; n < NT; ++n)
#pragma unroll
    for (int jj = 0; jj < 2; ++jj) {
      const float a = group_sum(l1v[n][jj]), bb = group_sum(ltv[n][jj]);
      const float cc = group_sum(l1t[n][jj]), dd = group_sum(ltt[n][jj]);
      const int h = 8 * n + 2 * tg + jj;
      if (gr == 0) {
        wst[warp][h][ST_MV] = m_v[n][jj]; wst[warp][h][ST_L1V] = a; wst[warp][h][ST_LTV] = bb;
        wst[warp][h][ST_MT] = m_t[n][jj]; wst[warp][h][ST_L1T] = cc; wst[warp][h][ST_LTT] = dd;
        wst[warp][h][3] = wst[warp][h][7] = 0.f;
      }
    }
  // acc[n][mi]: rows (dims) 16mi + gr and 16mi + gr + 8, heads 8n + 2tg, 8n + 2tg + 1.
  float* ow = reinterpret_cast<float*>(ring);
#pragma unroll
  for (int n = 0; n < NT; ++n)
#pragma unroll
    for (int mi = 0; mi < C::MT; ++mi) {
      const int h0 = 8 * n + 2 * tg, d0 = 16 * mi + gr;
      ow[h0 * D + d0] = acc[n][mi][0];
      ow[(h0 + 1) * D + d0] = acc[n][mi][1];
      ow[h0 * D + d0 + 8] = acc[n][mi][2];
      ow[(h0 + 1) * D + d0 + 8] = acc[n][mi][3];
    }
  score_epilogue<GM, D>(p, b, g, s, wst, reinterpret_cast<const float*>(smem), C::RING / 4, tail);
}

// ---------------------------------------------------------------------------
// k_score_tma (bf16).  The CTA's token range is cut into 32-token tiles
// aligned to absolute cache positions; warp w takes tiles w, w + NW, ...
// Every warp streams its own tiles through a private ring of S tile-sized
// slots in shared memory: lane 0 arms a slot's mbarrier with its byte count
// and loads the tile with 4-D bulk-tensor (TMA) copies -- boxes of 64
// dimensions x 32 rows (fewer when a page is shorter) with the 128-byte
// hardware swizzle, so the ldmatrix reads below are free of bank conflicts.
// A tile wholly inside the visual span takes one slot (K only); any other
// tile takes two consecutive slots (K, then V).  A warp refills a slot as soon
// as it has read it (K right after QK, V after PV), so up to S slots of its
// tiles are in flight.  Because each warp waits on its own slots strictly in
// the order it armed them, a barrier is never waited on more than one phase
// ahead.  QK and PV run on the tensor cores as in k_score_mma.  Rows past the
// live cache, or of an unmapped page, are masked by a row mask stored with
// the slot.  For paged caches the page ids of the CTA's boxes are read into
// shared memory once, before the first copy.
// ---------------------------------------------------------------------------
constexpr int kTmaTile = 32;
constexpr int kTmaMaxBoxes = 1024;  // page-id entries per cache a CTA may hold

template <int D, int NT, int NW, int S>
struct TmaCfg {
  static constexpr int GM = 8 * NT;
  static constexpr int THREADS = 32 * NW;
  static constexpr int KS = D / 16;                      // QK k-steps
  static constexpr int MT = D / 16;                      // PV m-tiles
  static constexpr int HALVES = D / 64;                  // 64-dimension boxes per row
  static constexpr int HALF_BYTES = kTmaTile * 128;      // one box: 32 rows x 128 bytes
  static constexpr int SLOT = HALVES * HALF_BYTES;       // one tile of K or of V
  static constexpr int RING = NW * S * SLOT;
  static constexpr int OFF_BAR = RING;                   // full[NW][S]
  static constexpr int OFF_MASK = OFF_BAR + NW * S * 8;  // row mask per slot
  static constexpr int OFF_PG = (OFF_MASK + NW * S * 4 + 15) / 16 * 16;  // page ids, K then V
  static constexpr int OFF_TAIL = OFF_PG + 2 * kTmaMaxBoxes * 4;
  static constexpr int OFF_WST = OFF_TAIL + (int)sizeof(ScoreTail<GM, D, NW>);
  static constexpr size_t SMEM = 1024 + (size_t)OFF_WST + sizeof(float) * NW * GM * ST_N;
  static_assert(S >= 2, "a text tile needs two slots");
  static_assert(NW * GM * D * 4 <= RING, "text partials must fit in the ring");
  static_assert(SLOT % 1024 == 0, "slots keep the swizzle atoms aligned");
};

// Byte offset of (row, element col) in a swizzled tile of 64-element boxes.
template <int HALF_BYTES>
__device__ __forceinline__ unsigned swz_off(int row, int col) {
  return (unsigned)((col >> 6) * HALF_BYTES + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4));
}
__device__ __forceinline__ float fexp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// exp2(a - m) by the hardware approximation, an empty term (a = -inf) giving 0.
__device__ __forceinline__ float fexp2_rel(float a, float m) { return a == -CUDART_INF_F ? 0.f : fexp2(a - m); }
// A tile of the K or V cache: every byte of it is read once per call, so it
// is marked evict-first in L2, which keeps the workspace (logits, split
// partials) and the kernels' other data resident while a step streams
// gigabytes of cache through the 129 MB L2.
__device__ __forceinline__ void tma_load_4d(unsigned dst, const CUtensorMap* map, int c0, int c1, int c2, int c3,
                                            uint64_t* bar) {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;\n"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(smem_u32(bar)),
        "l"(pol)
      : "memory");
}

// Page of the pool that holds cache position pos of sequence b; -1 if the
// block table maps it nowhere.
__device__ __forceinline__ int tma_page(const KvView& kv, const StepParams& p, int b, int pos) {
  const int lp = pos >> p.page_shift;
  if (lp >= kv.max_pages) return -1;
  const int page = __ldg(kv.block_table + (int64_t)b * kv.max_pages + lp);
  return (page < 0 || page >= kv.num_pages) ? -1 : page;
}

// The tiles of one split.  Tiles [v0, v1) lie wholly inside the visual span
// (K only); every other tile carries text rows (K and V).  Split s owns
// list entries [u0, u0 + n): a fixed weight per split (from the longest
// sequence), so that every working CTA moves about the same bytes.  For a
// layer after the anchor layer (ntext >= 0) the list is the cache tiles
// outside [v0, v1), then the kept visual tokens in tiles of 32, all
// attended with K and V.
struct TileRange {
  int u0, n, v0, v1, ntext;
  __device__ __forceinline__ bool text(int t) const {
    const int u = u0 + t;
    return ntext >= 0 || u < v0 || u >= v1;
  }
  __device__ __forceinline__ bool kept(int t) const { return ntext >= 0 && u0 + t >= ntext; }
  // Cache tile of entry t (not for kept entries).
  __device__ __forceinline__ int tile(int t) const {
    const int u = u0 + t;
    return (ntext >= 0 && u >= v0) ? u + (v1 - v0) : u;
  }
};
__device__ __forceinline__ TileRange tma_split(const Seq& sq, int s, int ns, int split_w, int n_kept) {
  const int T = sq.nv + sq.tl;
  const int NTl = (T + kTmaTile - 1) / kTmaTile;
  const int v0 = (sq.vs + kTmaTile - 1) / kTmaTile;
  const int v1 = max(v0, min(NTl, (sq.vs + sq.nv) / kTmaTile));
  TileRange r;
  r.v0 = v0;
  r.v1 = v1;
  if (n_kept >= 0) {  // after the anchor: every entry weighs 2
    r.ntext = NTl - (v1 - v0);
    const int L = r.ntext + (n_kept + kTmaTile - 1) / kTmaTile;
    const int per = max(split_w, (2 * L + ns - 1) / ns);
    r.u0 = (min(2 * L, s * per) + 1) / 2;
    r.n = (min(2 * L, (s + 1) * per) + 1) / 2 - r.u0;
    return r;
  }
  r.ntext = -1;
  const int W = 2 * NTl - (v1 - v0);  // text tiles weigh 2, visual tiles 1
  const int per = max(split_w, (W + ns - 1) / ns);  // splits past the sequence get nothing
  auto tile_of = [&](int w) {  // first tile whose weight prefix reaches w
    if (w <= 2 * v0) return (w + 1) / 2;
    if (w <= v0 + v1) return w - v0;
    return (w + (v1 - v0) + 1) / 2;
  };
  r.u0 = tile_of(min(W, s * per));
  r.n = tile_of(min(W, (s + 1) * per)) - r.u0;
  return r;
}

// ANCHOR: a layer after the anchor layer (text plus the given kept set).
template <int D, int NT, int NW, int S, bool ANCHOR>
__global__ void __launch_bounds__(32 * NW, 1) k_score_tma(const __grid_constant__ StepParams p) {
  using C = TmaCfg<D, NT, NW, S>;
  constexpr int GM = C::GM;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  // The 128-byte swizzle repeats every 1024 bytes: align the ring to that.
  unsigned char* smem = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gr = lane >> 2, tg = lane & 3;
  const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR) + warp * S;
  uint32_t* rowmask = reinterpret_cast<uint32_t*>(smem + C::OFF_MASK) + warp * S;
  int* kpg = reinterpret_cast<int*>(smem + C::OFF_PG);
  int* vpg = kpg + kTmaMaxBoxes;
  unsigned char* ring = smem + warp * S * C::SLOT;
  auto& tail = *reinterpret_cast<ScoreTail<GM, D, NW>*>(smem + C::OFF_TAIL);
  auto wst = reinterpret_cast<float (*)[GM][ST_N]>(smem + C::OFF_WST);

  if (tid < NW * S) mbar_init(reinterpret_cast<uint64_t*>(smem + C::OFF_BAR) + tid, 1);
  mbar_fence_init();
  // The descriptors are kernel parameters, not outputs of the previous kernel:
  // fetch them while that kernel finishes.
  if (tid == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmk)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmv)) : "memory");
  }
  // The decode step reads only the call's inputs (q, caches, spans, page
  // table) until its first workspace write, so its setup and first copies
  // run before griddepcontrol.wait, while the previous kernel of the stream
  // (which reads the workspace this kernel writes) finishes.  After the
  // anchor layer the kept sets come from that kernel: wait first.
  if (ANCHOR) pdl_wait();
  const int G = p.G, H = p.H;
  const Seq sq = load_seq(p, b, s == 0 && g == 0);
  const int T = sq.nv + sq.tl;
  unsigned err = 0;
  // After the anchor layer: the kept set of this sequence (or kv-head).
  int n_kept = -1;
  const int32_t* kept_rows = nullptr;
  if (ANCHOR) {
    const int sel = p.granularity ? b * p.Hkv + g : b;
    const int c = __ldcg(p.kept_count + sel);
    if (c < 0 || c > min(p.kept_cap, sq.nv)) err |= ERR_KEPT;
    n_kept = max(0, min(c, min(p.kept_cap, sq.nv)));
    kept_rows = p.kept_idx + (int64_t)sel * p.kept_cap;
  }
  const TileRange tr = tma_split(sq, s, p.ns, p.split_w, n_kept);
  // Entry kinds, constant-folded for the decode step.
  auto is_text = [&](int t) { return ANCHOR || tr.text(t); };
  auto is_kept = [&](int t) { return ANCHOR && tr.kept(t); };
  auto tile_at = [&](int t) { return ANCHOR ? tr.tile(t) : tr.u0 + t; };
  const int R = p.paged ? min(kTmaTile, p.page_size) : kTmaTile;  // rows per box
  const int nb = kTmaTile / R;                                     // boxes per tile (1..4)
  int n = tr.n;
  if (p.paged) {
    if (n * nb > kTmaMaxBoxes) {  // the host plan keeps every CTA below this
      err |= ERR_PAGE;
      n = 0;
    }
    for (int i = tid; i < n * nb; i += C::THREADS) {
      const int t = i / nb;
      if (is_kept(t)) continue;  // kept rows find their pages when issued
      const int pos = tile_at(t) * kTmaTile + (i % nb) * R;
      kpg[i] = pos < T ? tma_page(p.k, p, b, pos) : -2;
      vpg[i] = (pos < T && is_text(t)) ? tma_page(p.v, p, b, pos) : 0;
    }
  }
  __syncthreads();

  // ---------------------------------------------------------------- issue
  const int nj = warp < n ? (n - warp + NW - 1) / NW : 0;  // this warp's tiles
  int ji = 0, qi = 0, qf = 0;  // next tile to issue, its first slot, first slot not yet read
  const uint32_t boxmask = R >= 32 ? 0xffffffffu : ((1u << R) - 1u);
  auto issue = [&]() {
    while (ji < nj) {
      const int t = warp + NW * ji;
      const bool text = is_text(t);
      const int need = text ? 2 : 1;
      if (qi + need - qf > S) break;
      // The slots were last read by this warp's ldmatrix (generic proxy).
      fence_proxy_async();
      __syncwarp();
      if (is_kept(t)) {
        // Kept visual rows (after the anchor layer): each lane finds one row;
        // the warp copies K and V in 16-byte pieces, two rows per instruction,
        // into the swizzled layout of the tensor copies.
        const int r = (tr.u0 + t - tr.ntext) * kTmaTile + lane;
        int i = r < n_kept ? __ldcg(kept_rows + r) : -1;
        if (r < n_kept && (i < 0 || i >= sq.nv)) { err |= ERR_KEPT; i = -1; }
        const __nv_bfloat16* kr = nullptr;
        const __nv_bfloat16* vr = nullptr;
        if (i >= 0) {
          kr = kv_row<__nv_bfloat16>(p.k, p, b, g, sq.vs + i);
          vr = kv_row<__nv_bfloat16>(p.v, p, b, g, sq.vs + i);
          if (!kr || !vr) { err |= ERR_PAGE; kr = vr = nullptr; }
        }
        const unsigned m = __ballot_sync(0xffffffffu, kr != nullptr);
        const int ks = qi % S, vs = (qi + 1) % S;
        constexpr int PPR = 2 * D / 16, RPI = 32 / PPR;
        const unsigned kt = smem_u32(ring + ks * C::SLOT), vt = smem_u32(ring + vs * C::SLOT);
        const unsigned long long ka = reinterpret_cast<unsigned long long>(kr);
        const unsigned long long va = reinterpret_cast<unsigned long long>(vr);
#pragma unroll
        for (int jj = 0; jj < 32 / RPI; ++jj) {
          const int row = jj * RPI + lane / PPR;
          const unsigned off = swz_off<C::HALF_BYTES>(row, 8 * (lane % PPR));
          const unsigned long long a1 = __shfl_sync(0xffffffffu, ka, row);
          const unsigned long long a2 = __shfl_sync(0xffffffffu, va, row);
          if (a1) cp_async16(kt + off, reinterpret_cast<const char*>(a1) + (lane % PPR) * 16);
          if (a2) cp_async16(vt + off, reinterpret_cast<const char*>(a2) + (lane % PPR) * 16);
        }
        cp_async_arrive_counted(full + ks);
        cp_async_arrive_counted(full + vs);
        __syncwarp();
        if (lane == 0) {
          rowmask[ks] = m;
          mbar_expect_tx(full + ks, 0u);
          mbar_expect_tx(full + vs, 0u);
        }
      } else if (lane == 0) {
        const int p0 = tile_at(t) * kTmaTile;

        const int nvalid = min(kTmaTile, T - p0);
        uint32_t mask = nvalid >= 32 ? 0xffffffffu : ((1u << nvalid) - 1u);
        const int ks = qi % S, vs = (qi + 1) % S;
        unsigned bytes = 0;
        int kb[4], vb[4];
#pragma unroll
        for (int x = 0; x < 4; ++x) {
          kb[x] = -1;
          vb[x] = 0;
          if (x < nb && p0 + x * R < T) {
            if (p.paged) {
              kb[x] = kpg[t * nb + x];
              vb[x] = vpg[t * nb + x];
            } else {
              kb[x] = vb[x] = b;
            }
            if (kb[x] < 0 || vb[x] < 0) {
              err |= ERR_PAGE;
              mask &= ~(boxmask << (x * R));
              kb[x] = -1;
            } else {
              bytes += C::HALVES * R * 128u;
            }
          }
        }
        rowmask[ks] = mask;
        mbar_expect_tx(full + ks, bytes);
        if (text) mbar_expect_tx(full + vs, bytes);
        const unsigned kt = smem_u32(ring + ks * C::SLOT), vt = smem_u32(ring + vs * C::SLOT);
#pragma unroll
        for (int x = 0; x < 4; ++x) {
          if (kb[x] < 0) continue;
          const int row = p.paged ? ((p0 + x * R) & (p.page_size - 1)) : p0 + x * R;
          auto crd = [&](int axis, int base) { return axis == p.tpos ? row : axis == p.gpos ? g : base; };
#pragma unroll
          for (int hh = 0; hh < C::HALVES; ++hh) {
            const unsigned off = hh * C::HALF_BYTES + x * R * 128;
            tma_load_4d(kt + off, &p.tmk, 64 * hh, crd(1, kb[x]), crd(2, kb[x]), crd(3, kb[x]), full + ks);
            if (text) tma_load_4d(vt + off, &p.tmv, 64 * hh, crd(1, vb[x]), crd(2, vb[x]), crd(3, vb[x]), full + vs);
          }
        }
      }
      qi += need;
      ++ji;
    }
  };
  issue();

  // -------------------------------------------------------------- consume
  uint32_t qfr[NT][C::KS][2];
  const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(p.q) + ((int64_t)b * H + g * G) * D;
#pragma unroll
  for (int nn = 0; nn < NT; ++nn) {
    const int h = 8 * nn + gr;
    const uint32_t* qr = reinterpret_cast<const uint32_t*>(qb + h * D);
#pragma unroll
    for (int ks = 0; ks < C::KS; ++ks) {
      qfr[nn][ks][0] = h < G ? __ldg(qr + 8 * ks + tg) : 0u;
      qfr[nn][ks][1] = h < G ? __ldg(qr + 8 * ks + 4 + tg) : 0u;
    }
  }
  float m_v[NT][2], l1v[NT][2], ltv[NT][2], m_t[NT][2], l1t[NT][2], ltt[NT][2];
  float acc[NT][C::MT][4];
#pragma unroll
  for (int nn = 0; nn < NT; ++nn) {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      m_v[nn][j] = m_t[nn][j] = -CUDART_INF_F;
      l1v[nn][j] = ltv[nn][j] = l1t[nn][j] = ltt[nn][j] = 0.f;
    }
#pragma unroll
    for (int mi = 0; mi < C::MT; ++mi)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[nn][mi][e] = 0.f;
  }
  // ldmatrix lane roles: K as the A operand (rows = tokens), V^T via .trans.
  const int krow = (lane & 7) + 8 * ((lane >> 3) & 1), kcol = 8 * (lane >> 4);
  const int vrow = (lane & 7) + 8 * (lane >> 4), vcol = 8 * ((lane >> 3) & 1);
  const float ctau = p.inv_tau;
  bool timed_out = false;
  int qc = 0;  // first slot of the tile being read
  // The workspace (logits, partials) may still be read by the previous
  // kernel: each thread waits for it only before its first workspace write,
  // so splits of text tiles stream their whole range meanwhile.
  bool ws_ok = ANCHOR;

  for (int j = 0; j < nj; ++j) {
    const int t = warp + NW * j;
    const bool text = is_text(t);
    const int ks_ = qc % S;
    if (!mbar_wait(full + ks_, (qc / S) & 1)) { timed_out = true; break; }
    const uint32_t mask = rowmask[ks_];
    const bool kept_tile = is_kept(t);
    const int p0 = kept_tile ? 0 : tile_at(t) * kTmaTile;
    const unsigned kt = smem_u32(ring + ks_ * C::SLOT);

    // ---- QK for both 16-row halves of the tile, then refill the K slot
    // Even and odd k-steps accumulate separately: two short dependency chains
    // per 16-row half instead of one long one.
    float c[2][NT][4], c2[2][NT][4];
#pragma unroll
    for (int sb = 0; sb < 2; ++sb) {
#pragma unroll
      for (int nn = 0; nn < NT; ++nn)
#pragma unroll
        for (int e = 0; e < 4; ++e) c[sb][nn][e] = c2[sb][nn][e] = 0.f;
#pragma unroll
      for (int ks = 0; ks < C::KS; ++ks) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(kt + swz_off<C::HALF_BYTES>(16 * sb + krow, 16 * ks + kcol), a0, a1, a2, a3);
#pragma unroll
        for (int nn = 0; nn < NT; ++nn)
          mma_bf16((ks & 1) ? c2[sb][nn] : c[sb][nn], a0, a1, a2, a3, qfr[nn][ks][0], qfr[nn][ks][1]);
      }
#pragma unroll
      for (int nn = 0; nn < NT; ++nn)
#pragma unroll
        for (int e = 0; e < 4; ++e) c[sb][nn][e] += c2[sb][nn][e];
    }
    qf = qc + 1;
    issue();

    // c[sb][n][e]: row 16sb + gr + 8(e >> 1), head 8n + 2tg + (e & 1).
    float zv[2][NT][4], zt[2][NT][4];
    bool any_vis = false;
    // A tile with visual rows writes logits: wait for the workspace first (warp-uniform).
    if (!ws_ok && !kept_tile && p0 < sq.vs + sq.nv && p0 + kTmaTile > sq.vs) {
      pdl_wait();
      ws_ok = true;
    }
#pragma unroll
    for (int sb = 0; sb < 2; ++sb)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int row = 16 * sb + gr + 8 * (e >> 1);
        const int pos = p0 + row;
        const bool valid = (mask >> row) & 1u;
        // A cache row inside the visual span is visual; after the anchor
        // layer it is left out (its kept tokens come as kept rows).
        const bool inspan = !kept_tile && (unsigned)(pos - sq.vs) < (unsigned)sq.nv;
        const bool vis = !ANCHOR && valid && inspan;
        const bool txt = valid && !inspan;
        any_vis |= vis;
#pragma unroll
        for (int nn = 0; nn < NT; ++nn) {
          const bool hv = (8 * nn + 2 * tg + (e & 1)) < G;
          const float z = c[sb][nn][e] * p.c_log2;
          zv[sb][nn][e] = (vis && hv) ? z : -CUDART_INF_F;
          zt[sb][nn][e] = (txt && hv) ? z : -CUDART_INF_F;
        }
        if (vis) {
          float* zrow = p.z_ws + ((int64_t)b * p.max_visual + (pos - sq.vs)) * p.hp + g * G;
#pragma unroll
          for (int nn = 0; nn < NT; ++nn) {
            const int h = 8 * nn + 2 * tg + (e & 1);
            if (h < G) zrow[h] = zv[sb][nn][e];
          }
        }
      }
    // ---- visual statistics
    if (__any_sync(0xffffffffu, any_vis)) {
#pragma unroll
      for (int nn = 0; nn < NT; ++nn)
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const float mx = fmaxf(fmaxf(zv[0][nn][jj], zv[0][nn][jj + 2]), fmaxf(zv[1][nn][jj], zv[1][nn][jj + 2]));
          const float mn = fmaxf(m_v[nn][jj], group_max(mx));
          if (mn > m_v[nn][jj]) {
            l1v[nn][jj] *= exp2_rel(m_v[nn][jj], mn);
            ltv[nn][jj] *= exp2_tau(m_v[nn][jj], mn, ctau);
            m_v[nn][jj] = mn;
          }
          if (mn != -CUDART_INF_F) {
#pragma unroll
            for (int sb = 0; sb < 2; ++sb)
#pragma unroll
              for (int e = jj; e < 4; e += 2) {
                l1v[nn][jj] += fexp2(zv[sb][nn][e] - mn);
                ltv[nn][jj] += fexp2((zv[sb][nn][e] - mn) * ctau);
              }
          }
        }
    }
    // ---- text statistics, probabilities and P.V from the V slot
    if (text) {
      uint32_t pb[2][NT][2];
#pragma unroll
      for (int nn = 0; nn < NT; ++nn) {
        float pr[2][4];
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const float mx = fmaxf(fmaxf(zt[0][nn][jj], zt[0][nn][jj + 2]), fmaxf(zt[1][nn][jj], zt[1][nn][jj + 2]));
          const float mn = fmaxf(m_t[nn][jj], group_max(mx));
          if (mn > m_t[nn][jj]) {
            const float a = exp2_rel(m_t[nn][jj], mn);
            l1t[nn][jj] *= a;
            ltt[nn][jj] *= exp2_tau(m_t[nn][jj], mn, ctau);
#pragma unroll
            for (int mi = 0; mi < C::MT; ++mi) {
              acc[nn][mi][jj] *= a;
              acc[nn][mi][jj + 2] *= a;
            }
            m_t[nn][jj] = mn;
          }
#pragma unroll
          for (int sb = 0; sb < 2; ++sb)
#pragma unroll
            for (int e = jj; e < 4; e += 2) {
              const float pe = mn != -CUDART_INF_F ? fexp2(zt[sb][nn][e] - mn) : 0.f;
              pr[sb][e] = pe;
              l1t[nn][jj] += pe;
              if (mn != -CUDART_INF_F) ltt[nn][jj] += fexp2((zt[sb][nn][e] - mn) * ctau);
            }
        }
#pragma unroll
        for (int sb = 0; sb < 2; ++sb) {
          const uint32_t p01 = pack_bf16(pr[sb][0], pr[sb][1]), p23 = pack_bf16(pr[sb][2], pr[sb][3]);
          const int src0 = 8 * tg + (gr >> 1), src1 = src0 + 4;
          const uint32_t x0 = __shfl_sync(0xffffffffu, p01, src0), x1 = __shfl_sync(0xffffffffu, p01, src1);
          const uint32_t x2 = __shfl_sync(0xffffffffu, p23, src0), x3 = __shfl_sync(0xffffffffu, p23, src1);
          const uint32_t sel = (gr & 1) ? 0x7632u : 0x5410u;
          pb[sb][nn][0] = prmt(x0, x1, sel);
          pb[sb][nn][1] = prmt(x2, x3, sel);
        }
      }
      const int vq = qc + 1, vs_ = vq % S;
      if (!mbar_wait(full + vs_, (vq / S) & 1)) { timed_out = true; break; }
      const unsigned vt = smem_u32(ring + vs_ * C::SLOT);
#pragma unroll
      for (int sb = 0; sb < 2; ++sb) {
        // Words of rows outside the mask (past the cache, unmapped pages) are
        // zeroed: their probabilities are 0 but their bytes may not be finite.
        const uint32_t rb = mask >> (16 * sb);
        const uint32_t mlo = (((rb >> (2 * tg)) & 1u) ? 0x0000ffffu : 0u) | (((rb >> (2 * tg + 1)) & 1u) ? 0xffff0000u : 0u);
        const uint32_t mhi = (((rb >> (2 * tg + 8)) & 1u) ? 0x0000ffffu : 0u) | (((rb >> (2 * tg + 9)) & 1u) ? 0xffff0000u : 0u);
#pragma unroll
        for (int mi = 0; mi < C::MT; ++mi) {
          uint32_t a0, a1, a2, a3;
          ldsm_x4_t(vt + swz_off<C::HALF_BYTES>(16 * sb + vrow, 16 * mi + vcol), a0, a1, a2, a3);
          a0 &= mlo; a1 &= mlo; a2 &= mhi; a3 &= mhi;
#pragma unroll
          for (int nn = 0; nn < NT; ++nn) mma_bf16(acc[nn][mi], a0, a1, a2, a3, pb[sb][nn][0], pb[sb][nn][1]);
        }
      }
      qf = qc + 2;
      issue();
    }
    qc += text ? 2 : 1;
  }
  // After a timeout, let this warp's copies still in flight land (bounded)
  // before the ring is reused below.
  if (timed_out && lane == 0)
    for (int q = max(qc, qi - S); q < qi; ++q) mbar_wait(full + q % S, (q / S) & 1);
  __syncwarp();

  // Warp statistics now; text outputs once every warp is done with the ring.
#pragma unroll
  for (int nn = 0; nn < NT; ++nn)
#pragma unroll
    for (int jj = 0; jj < 2; ++jj) {
      const float a = group_sum(l1v[nn][jj]), bb = group_sum(ltv[nn][jj]);
      const float cc = group_sum(l1t[nn][jj]), dd = group_sum(ltt[nn][jj]);
      const int h = 8 * nn + 2 * tg + jj;
      if (gr == 0) {
        wst[warp][h][ST_MV] = m_v[nn][jj]; wst[warp][h][ST_L1V] = a; wst[warp][h][ST_LTV] = bb;
        wst[warp][h][ST_MT] = m_t[nn][jj]; wst[warp][h][ST_L1T] = cc; wst[warp][h][ST_LTT] = dd;
        wst[warp][h][3] = wst[warp][h][7] = 0.f;
      }
    }
  pdl_trigger();
  __syncthreads();
  float* ow = reinterpret_cast<float*>(smem) + warp * GM * D;
#pragma unroll
  for (int nn = 0; nn < NT; ++nn)
#pragma unroll
    for (int mi = 0; mi < C::MT; ++mi) {
      const int h0 = 8 * nn + 2 * tg, d0 = 16 * mi + gr;
      ow[h0 * D + d0] = acc[nn][mi][0];
      ow[(h0 + 1) * D + d0] = acc[nn][mi][1];
      ow[h0 * D + d0 + 8] = acc[nn][mi][2];
      ow[(h0 + 1) * D + d0 + 8] = acc[nn][mi][3];
    }
  if (timed_out) err |= ERR_TIMEOUT;
  if (err) atomicOr(p.err, err);
  if (!ws_ok) pdl_wait();
  score_epilogue<GM, D, NW, C::THREADS>(p, b, g, s, wst, reinterpret_cast<const float*>(smem), GM * D, tail);
}

// ---------------------------------------------------------------------------
// k_score_tc (bf16, D = 128, up to 16 query heads per kv-head): the decode
// step's score kernel on the fifth-generation tensor cores.  Grid (splits,
// Hkv, B) with the splits cut in 128-row tiles; 192 threads in three roles:
//   warp 0     (one lane) copies each tile's K, and its V where the tile holds
//              rows outside the visual span, with 4-D bulk-tensor copies into
//              a ring of three 32 KB slots (128-byte swizzle);
//   warp 1     holds 64 TMEM columns and (one lane) issues tcgen05.mma:
//              S = K q^T (M = 128 tokens, N = 16 heads, K = 128 dimensions)
//              into one of two S buffers, and O += V^T P^T (M = 128
//              dimensions, N = 16 heads, K = 128 tokens) into the O buffer,
//              each completion signalled by tcgen05.commit on an mbarrier;
//   warps 2-5  (one thread per token row; for O, per dimension) read S with
//              tcgen05.ld, write the visual logits, keep the visual
//              statistics per thread and turn text logits into probabilities
//              P = exp2(z - M_ref) for the P.V product.
// M_ref, a head's text reference maximum, is raised only when a logit passes
// it by more than theta = min(8, 64 tau) (log2 units), so that P and the
// tempered sums stay finite; the O accumulator and the sums are then
// rescaled.  Most tiles need no exchange between the threads.  The split's
// partial has the meaning of the other score kernels' partials.
// Waits are bounded: a thread whose wait gives up stops its work, still
// passes every barrier of its group, and the error word reports the timeout.
// ---------------------------------------------------------------------------
constexpr int kTcSlots = 3;  // ring slots of the kernel as launched (two CTAs per SM)
constexpr int kTcThreads = 192;

template <int NS>
struct TcCfgT {
  static constexpr int HALF = kTcRows * 128;           // 128 rows x 64 dimensions, swizzled
  static constexpr int SLOT = 2 * HALF;                // a 128 x 128 tile of K or of V
  static constexpr int QHALF = 16 * 128;               // 16 rows x 64 elements
  static constexpr int OFF_Q = NS * SLOT;              // q: 16 heads x 128 dimensions
  static constexpr int OFF_P = OFF_Q + 2 * QHALF;      // P^T: 2 buffers of 16 heads x 128 tokens
  static constexpr int PBUF = 2 * QHALF;
  static constexpr int OFF_BAR = OFF_P + 2 * PBUF;
  static constexpr int NBAR = 2 * NS + 9;              // full, empty, s_full, s_free, p_full, pv_done, mma_done
  static constexpr int OFF_PG = OFF_BAR + (NBAR * 8 + 15) / 16 * 16;
  static constexpr int OFF_RED = OFF_PG + 2 * kTcMaxBoxes * 4;  // float [4][16]: new text maxima
  static constexpr int OFF_TMEM = OFF_RED + 4 * 16 * 4;
  // The partial's reductions, float [4][16][6], take the P buffers once every
  // P.V product is complete.
  static_assert(4 * 16 * 6 * 4 <= 2 * PBUF, "reduction buffer fits the P buffers");
  static constexpr size_t SMEM = 1024 + (size_t)OFF_TMEM + 16;
  static_assert(SLOT % 1024 == 0 && OFF_Q % 1024 == 0 && OFF_P % 1024 == 0, "swizzle atoms stay aligned");
};
using TcCfg = TcCfgT<kTcSlots>;

// Shared-memory matrix descriptor of a 128-byte-swizzled operand (sm_100
// layout: start, leading and stride byte offsets in 16-byte units, version 1).
__device__ __forceinline__ uint64_t umma_desc(unsigned addr, unsigned lbo, unsigned sbo) {
  return (uint64_t)((addr >> 4) & 0x3fffu) | ((uint64_t)((lbo >> 4) & 0x3fffu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3fffu) << 32) | (1ull << 46) | (2ull << 61);
}
// Instruction descriptor: bf16 x bf16 -> f32, M = 128, N = 16; A K-major or
// MN-major, B K-major.
__host__ __device__ constexpr uint32_t umma_idesc(int a_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn << 15) | ((uint32_t)(16 >> 3) << 17) |
         ((uint32_t)(128 >> 4) << 24);
}
__device__ __forceinline__ void umma(unsigned d, uint64_t a, uint64_t b, uint32_t id, bool acc) {
  asm volatile("{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
               ::"r"(d), "l"(a), "l"(b), "r"(id), "r"((int)acc) : "memory");
}
// Arrives on the mbarrier once this thread's earlier tensor-core operations are complete.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tmem_ld16(unsigned taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_st16(unsigned taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n"
      ::"r"(taddr), "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_u32(bar)) : "memory");
}
// Barrier of the four softmax warps (named barrier 1); the second form also
// counts the threads whose predicate is true.
__device__ __forceinline__ void wg_sync() { asm volatile("barrier.cta.sync 1, 128;\n" ::: "memory"); }
__device__ __forceinline__ int wg_sync_count(bool pred) {
  int n;
  asm volatile("{\n .reg .pred p;\n setp.ne.b32 p, %1, 0;\n barrier.cta.red.popc.u32 %0, 1, 128, p;\n}\n"
               : "=r"(n) : "r"((int)pred) : "memory");
  return n;
}

template <int GM, int NS = kTcSlots>
__global__ void __launch_bounds__(kTcThreads, NS <= 3 ? 2 : 1) k_score_tc(const __grid_constant__ StepParams p) {
  using C = TcCfgT<NS>;
  constexpr int D = 128, S = NS;
  constexpr uint32_t kIdQK = umma_idesc(0), kIdPV = umma_idesc(1);
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char* smem = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);  // [S] a slot's copies landed
  uint64_t* empty = full + S;                                        // [S] a slot's tile was read
  uint64_t* s_full = full + 2 * S;                                   // [2] S buffer written
  uint64_t* s_free = s_full + 2;                                     // [2] S buffer read (128 arrivals)
  uint64_t* p_full = s_full + 4;                                     // [2] P buffer written (128 arrivals)
  uint64_t* pv_done = s_full + 6;                                    // [2] P.V of that P buffer complete
  uint64_t* mma_done = s_full + 8;                                   // every tensor-core operation complete
  int* kpg = reinterpret_cast<int*>(smem + C::OFF_PG);
  int* vpg = kpg + kTcMaxBoxes;
  float (*red)[16] = reinterpret_cast<float (*)[16]>(smem + C::OFF_RED);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_TMEM);

  if (tid == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(full + i, 1);
      mbar_init(empty + i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full + i, 1);
      mbar_init(s_free + i, 128);
      mbar_init(p_full + i, 128);
      mbar_init(pv_done + i, 1);
    }
    mbar_init(mma_done, 1);
    mbar_fence_init();
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmk2)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmv2)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 64;\n" ::"r"(smem_u32(tmem_slot))
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  // Everything up to the first workspace write reads only the call's inputs,
  // so it runs before griddepcontrol.wait (see k_score_tma).
  const int G = p.G, H = p.H;
  const Seq sq = load_seq(p, b, s == 0 && g == 0);
  const int T = sq.nv + sq.tl;
  const TcRange tr = tc_split(sq.vs, sq.nv, sq.tl, s, p.ns, p.split_w);
  const int R = p.paged ? min(kTcRows, p.page_size) : kTcRows;  // rows per copied box
  const int nb = kTcRows / R;
  int n = tr.n;
  unsigned err = 0;
  if (p.paged) {
    if (n * nb > kTcMaxBoxes) {  // the host plan keeps every split below this
      err |= ERR_PAGE;
      n = 0;
    }
    for (int i = tid; i < n * nb; i += kTcThreads) {
      const int t = i / nb, pos = (tr.u0 + t) * kTcRows + (i % nb) * R;
      kpg[i] = pos < T ? tma_page(p.k, p, b, pos) : -2;
      vpg[i] = (pos < T && !tr.pure(t)) ? tma_page(p.v, p, b, pos) : -2;
    }
  }
  // ---------------------------------------------------------------- copies
  // Warp 0 issues the pieces in the order the tensor cores read them: K of
  // tile i, then V of the text tile before it (its P.V follows tile i's QK);
  // iteration n issues only the last V.  Lane 0 arms the slot's barrier;
  // lane 2x + hh copies half hh of box x.
  int qc = 0;              // pieces issued
  int pi = 0, ppend = -1;  // next iteration; text tile whose V is due
  auto issue = [&](int i, int part) {
    const int sl = qc % S;
    if (!__all_sync(0xffffffffu, mbar_wait(empty + sl, ((qc / S) & 1) ^ 1))) return false;
    const int u = tr.u0 + i;
    const int* pg = part ? vpg : kpg;
    bool live = false, bad = false;
    int base = b, row = 0;
    const int x = lane >> 1, hh = lane & 1;
    if (x < nb) {
      const int pos = u * kTcRows + x * R;
      if (pos < T) {
        if (p.paged) {
          base = pg[i * nb + x];
          bad = base < 0;
          row = pos & (p.page_size - 1);
        } else {
          row = pos;
        }
        live = !bad;
      }
    }
    if (bad) err |= ERR_PAGE;
    const unsigned n_live = __popc(__ballot_sync(0xffffffffu, live));  // live halves
    if (lane == 0) mbar_expect_tx(full + sl, n_live * (unsigned)R * 128u);
    __syncwarp();
    if (live) {
      auto crd = [&](int axis) { return axis == p.tpos ? row : axis == p.gpos ? g : base; };
      tma_load_4d(smem_u32(smem + sl * C::SLOT) + hh * C::HALF + x * R * 128, part ? &p.tmv2 : &p.tmk2, 64 * hh,
                  crd(1), crd(2), crd(3), full + sl);
    }
    ++qc;
    return true;
  };
  // false when a wait gave up; with ring_only it stops before the first
  // piece that would wait for a slot to be read.
  auto produce = [&](bool ring_only) {
    for (; pi <= n; ++pi) {
      if (ring_only && qc + (pi < n ? 1 : 0) + (ppend >= 0 ? 1 : 0) > S) return true;
      if (pi < n && !issue(pi, 0)) return false;
      if (ppend >= 0 && !issue(ppend, 1)) return false;
      ppend = (pi < n && !tr.pure(pi)) ? pi : -1;
    }
    return true;
  };
  bool timed_out = false;
  // Contiguous caches: the first slots' copies start before the CTA-wide
  // barrier; they need only the barriers that lane 0 initialised.
  if (warp == 0 && !p.paged) {
    __syncwarp();
    timed_out = !produce(true);
  }
  if (warp >= 2) {  // q of the kv-head's query heads, rows past G zero, K-major and swizzled
    const uint32_t* qb = reinterpret_cast<const uint32_t*>(reinterpret_cast<const __nv_bfloat16*>(p.q) +
                                                           ((int64_t)b * H + g * G) * D);
    for (int i = tid - 64; i < 16 * (D / 8); i += 128) {
      const int h = i / (D / 8), c = i % (D / 8);  // 16-byte piece c (dimensions 8c .. 8c + 7)
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (h < G) {
        const uint32_t* src = qb + h * (D / 2) + 4 * c;
        v = make_uint4(__ldg(src), __ldg(src + 1), __ldg(src + 2), __ldg(src + 3));
      }
      *reinterpret_cast<uint4*>(smem + C::OFF_Q + (c >> 3) * C::QHALF + h * 128 + (((c & 7) ^ (h & 7)) << 4)) = v;
    }
    fence_proxy_async();  // read by the tensor core
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const unsigned tmem = *tmem_slot;  // columns [0,16) and [16,32): S buffers; [32,48): O

  if (warp == 0) {
    if (!timed_out && !produce(false)) timed_out = true;
    // Copies still in flight (only after a timeout can any be unread) land
    // before the CTA's shared memory is released.
    for (int k = max(0, qc - S); k < qc; ++k) mbar_wait(full + k % S, (k / S) & 1);
  } else if (warp == 1) {
    // ------------------------------------------------------ tensor cores
    // Tile i's QK is issued before the P.V of the previous text tile, so that
    // the softmax threads find S(i) ready when they finish that tile's P.
    // Every lane waits (and zeroes stale V rows); the warp leaves the loop
    // together when any lane's wait gives up.
    auto wait_all = [&](uint64_t* bar, unsigned parity) { return __all_sync(0xffffffffu, mbar_wait(bar, parity)); };
    int q = 0, j = 0;        // pieces read, text tiles multiplied
    int pend = -1, pq = 0;   // text tile whose P.V is due, and its V piece (read after K of the next tile)
    auto pv = [&]() {        // the P.V product of text tile `pend`
      const int sv = pq % S, pb = j & 1;
      if (!wait_all(full + sv, (pq / S) & 1)) return false;
      // V rows past the cache or of an unmapped page hold stale bytes: zero
      // them (their probabilities are 0, but 0 x NaN is not).
      const int p0 = (tr.u0 + pend) * kTcRows;
      bool stale = p0 + kTcRows > T;
      if (p.paged)
        for (int x = 0; x < nb; ++x) stale |= vpg[pend * nb + x] < 0;
      if (stale) {
        unsigned char* vt = smem + sv * C::SLOT;
        for (int r = lane; r < kTcRows; r += 32) {
          if (p0 + r < T && !(p.paged && vpg[pend * nb + r / R] < 0)) continue;
#pragma unroll
          for (int c = 0; c < 16; ++c)
            *reinterpret_cast<uint4*>(vt + (c >> 3) * C::HALF + r * 128 + (c & 7) * 16) = make_uint4(0u, 0u, 0u, 0u);
        }
        fence_proxy_async();
      }
      __syncwarp();
      if (!wait_all(p_full + pb, (j >> 1) & 1)) return false;
      tc_fence_after();
      if (lane == 0) {
        const unsigned vb = smem_u32(smem + sv * C::SLOT), pbs = smem_u32(smem + C::OFF_P + pb * C::PBUF);
#pragma unroll
        for (int ks = 0; ks < kTcRows / 16; ++ks)
          umma(tmem + 32, umma_desc(vb + ks * 2048, C::HALF, 1024),
               umma_desc(pbs + (ks >> 2) * C::QHALF + (ks & 3) * 32, 16, 1024), kIdPV, j > 0 || ks > 0);
        umma_commit(pv_done + pb);
        umma_commit(empty + sv);
      }
      __syncwarp();
      ++j;
      pend = -1;
      return true;
    };
    // Iteration n only multiplies the last text tile's P.V.
    for (int i = 0; i <= n; ++i) {
      if (i < n) {
        const int sb = i & 1, sk = q % S;
        if (!wait_all(full + sk, (q / S) & 1) || !wait_all(s_free + sb, ((i >> 1) & 1) ^ 1)) {
          timed_out = true;
          break;
        }
        tc_fence_after();
        if (lane == 0) {
          const unsigned kb = smem_u32(smem + sk * C::SLOT), qs = smem_u32(smem + C::OFF_Q);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks)
            umma(tmem + 16 * sb, umma_desc(kb + (ks >> 2) * C::HALF + (ks & 3) * 32, 16, 1024),
                 umma_desc(qs + (ks >> 2) * C::QHALF + (ks & 3) * 32, 16, 1024), kIdQK, ks > 0);
          umma_commit(s_full + sb);
          umma_commit(empty + sk);
        }
        __syncwarp();
        ++q;
      }
      if (pend >= 0) {
        pq = q++;
        if (!pv()) { timed_out = true; break; }
      }
      if (i < n && !tr.pure(i)) pend = i;
    }
    if (lane == 0) umma_commit(mma_done);  // after every operation issued above
    __syncwarp();
    if (!mbar_wait(mma_done, 0)) timed_out = true;
  } else {
    // -------------------------------------------- softmax (one row each)
    const int wq = warp & 3;                     // TMEM lanes [32 wq, 32 wq + 32)
    const int r = wq * 32 + lane;                // token row of a tile; dimension of O
    const unsigned taddr = tmem + ((unsigned)(wq * 32) << 16);
    const float inv_tau = p.inv_tau, theta = fminf(8.f, 64.f / inv_tau);
    float mv[GM], l1v[GM], ltv[GM], mref[GM], l1t[GM], ltt[GM];
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      mv[h] = mref[h] = -CUDART_INF_F;
      l1v[h] = ltv[h] = l1t[h] = ltt[h] = 0.f;
    }
    float* zbase = p.z_ws + (int64_t)b * p.max_visual * p.hp + g * G;
    const bool zvec = (G & 3) == 0;
    bool dead = false;  // a wait of this thread gave up: skip the work, keep the barriers
    // The workspace may still be read by the previous kernel: a thread waits
    // for it only before its first workspace write (visual logits, or the
    // split's partial), so splits of text tiles stream their whole range
    // meanwhile.
    bool ws_ok = false;
    int j = 0;          // text tiles seen
    for (int i = 0; i < n; ++i) {
      const int u = tr.u0 + i, sb = i & 1;
      float sv[16];
      if (__all_sync(0xffffffffu, !dead && mbar_wait(s_full + sb, (i >> 1) & 1))) {
        tc_fence_after();
        tmem_ld16(taddr + 16 * sb, sv);
      } else {
        dead = true;
#pragma unroll
        for (int h = 0; h < 16; ++h) sv[h] = 0.f;
      }
      tc_fence_before();
      mbar_arrive(s_free + sb);
      // A tile with visual rows writes logits: wait for the workspace first
      // (the same decision for every softmax thread).
      if (!ws_ok && u * kTcRows < sq.vs + sq.nv && u * kTcRows + kTcRows > sq.vs) {
        pdl_wait();
        ws_ok = true;
      }
      const int pos = u * kTcRows + r;
      bool valid = !dead && pos < T;
      if (valid && p.paged) valid = kpg[i * nb + r / R] >= 0;
      const bool vis = valid && (unsigned)(pos - sq.vs) < (unsigned)sq.nv;
      const bool txt = valid && !vis;
#pragma unroll
      for (int h = 0; h < GM; ++h) sv[h] *= p.c_log2;
      if (vis) {
        float* zr = zbase + (int64_t)(pos - sq.vs) * p.hp;
        if (zvec) {
#pragma unroll
          for (int h = 0; h < GM; h += 4)
            if (h < G) *reinterpret_cast<float4*>(zr + h) = make_float4(sv[h], sv[h + 1], sv[h + 2], sv[h + 3]);
        } else {
#pragma unroll
          for (int h = 0; h < GM; ++h)
            if (h < G) zr[h] = sv[h];
        }
#pragma unroll
        for (int h = 0; h < GM; ++h) {
          if (h >= G) continue;
          const float z = sv[h];
          if (z > mv[h]) {
            l1v[h] = fmaf(l1v[h], exp2_rel(mv[h], z), 1.f);
            ltv[h] = fmaf(ltv[h], exp2_tau(mv[h], z, inv_tau), 1.f);
            mv[h] = z;
          } else {
            l1v[h] += fexp2(z - mv[h]);
            ltv[h] += fexp2((z - mv[h]) * inv_tau);
          }
        }
      }
      if (tr.pure(i)) continue;
      // ---- text rows: raise M_ref where a logit passes it by more than theta
      bool need = false;
#pragma unroll
      for (int h = 0; h < GM; ++h) need |= txt && h < G && sv[h] > mref[h] + theta;
      if (wg_sync_count(need)) {
#pragma unroll
        for (int h = 0; h < GM; ++h) {
          const float m = warp_max(txt && h < G ? sv[h] : -CUDART_INF_F);
          if (lane == 0) red[wq][h] = m;
        }
        wg_sync();
        float f[GM];
#pragma unroll
        for (int h = 0; h < GM; ++h) {
          const float mn = fmaxf(mref[h], fmaxf(fmaxf(red[0][h], red[1][h]), fmaxf(red[2][h], red[3][h])));
          f[h] = exp2_rel(mref[h], mn);
          l1t[h] *= f[h];
          ltt[h] *= exp2_tau(mref[h], mn, inv_tau);
          mref[h] = mn;
        }
        wg_sync();  // red is read before its next use
        if (j > 0 && __any_sync(0xffffffffu, !dead)) {
          // O holds the products of text tiles 0 .. j - 1: rescale it once the last is complete.
          if (__all_sync(0xffffffffu, !dead && mbar_wait(pv_done + ((j - 1) & 1), ((j - 1) >> 1) & 1))) {
            tc_fence_after();
            float o[16];
            tmem_ld16(taddr + 32, o);
#pragma unroll
            for (int h = 0; h < GM; ++h) o[h] *= f[h];
            tmem_st16(taddr + 32, o);
          } else {
            dead = true;
          }
        }
      }
      // ---- probabilities, into P^T (K-major, swizzled) for the P.V product
      __nv_bfloat16 pr[16];
#pragma unroll
      for (int h = 0; h < 16; ++h) {
        float pe = 0.f;
        if (h < GM && h < G && txt) {
          pe = fexp2(sv[h] - mref[h]);
          l1t[h] += pe;
          ltt[h] += fexp2((sv[h] - mref[h]) * inv_tau);
        }
        pr[h] = __float2bfloat16_rn(pe);
      }
      const int pb = j & 1;
      if (j >= 2 && !dead && !mbar_wait(pv_done + pb, ((j >> 1) & 1) ^ 1)) dead = true;  // buffer free
      unsigned char* pt = smem + C::OFF_P + pb * C::PBUF + (r >> 6) * C::QHALF + (r & 7) * 2;
#pragma unroll
      for (int h = 0; h < 16; ++h)
        *reinterpret_cast<__nv_bfloat16*>(pt + h * 128 + ((((r & 63) >> 3) ^ (h & 7)) << 4)) = pr[h];
      fence_proxy_async();
      tc_fence_before();
      mbar_arrive(p_full + pb);
      ++j;
    }
    // ---- the split's partial: text output, then statistics
    float o[16];
#pragma unroll
    for (int h = 0; h < 16; ++h) o[h] = 0.f;
    if (j > 0 && __any_sync(0xffffffffu, !dead)) {
      if (__all_sync(0xffffffffu, !dead && mbar_wait(pv_done + ((j - 1) & 1), ((j - 1) >> 1) & 1))) {
        tc_fence_after();
        tmem_ld16(taddr + 32, o);
      } else {
        dead = true;
      }
    }
    pdl_trigger();
    float (*red6)[16][6] = reinterpret_cast<float (*)[16][6]>(smem + C::OFF_P);
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      const float M = warp_max(mv[h]);
      const float a1 = warp_sum(l1v[h] * exp2_rel(mv[h], M)), at = warp_sum(ltv[h] * exp2_tau(mv[h], M, inv_tau));
      const float c1 = warp_sum(l1t[h]), ct = warp_sum(ltt[h]);
      if (lane == 0) {
        red6[wq][h][0] = M; red6[wq][h][1] = a1; red6[wq][h][2] = at;
        red6[wq][h][3] = c1; red6[wq][h][4] = ct;
      }
    }
    wg_sync();
    if (!ws_ok) pdl_wait();
    const int64_t rec0 = ((int64_t)b * H + g * G) * p.nsp_max + s;  // split slot of head 0
    if (r < G) {
      const int h = r;
      float M = -CUDART_INF_F;
#pragma unroll
      for (int w = 0; w < 4; ++w) M = fmaxf(M, red6[w][h][0]);
      float a1 = 0.f, at = 0.f, c1 = 0.f, ct = 0.f;
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        a1 = fmaf(red6[w][h][1], exp2_rel(red6[w][h][0], M), a1);
        at = fmaf(red6[w][h][2], exp2_tau(red6[w][h][0], M, inv_tau), at);
        c1 += red6[w][h][3];
        ct += red6[w][h][4];
      }
      float mt = -CUDART_INF_F;
#pragma unroll
      for (int hh = 0; hh < GM; ++hh)
        if (hh == h) mt = mref[hh];
      float4* rec = reinterpret_cast<float4*>(p.split_st + (rec0 + (int64_t)h * p.nsp_max) * ST_N);
      rec[0] = make_float4(mt, c1, ct, 0.f);  // ST_MT, ST_L1T, ST_LTT
      rec[1] = make_float4(M, a1, at, 0.f);   // ST_MV, ST_L1V, ST_LTV
    }
#pragma unroll
    for (int h = 0; h < GM; ++h)
      if (h < G) p.split_o[(rec0 + (int64_t)h * p.nsp_max) * D + r] = o[h];
    if (dead) timed_out = true;
  }
  if (timed_out) err |= ERR_TIMEOUT;
  if (err) atomicOr(p.err, err);
  // Teardown: every copy has landed and every tensor-core operation is
  // complete (warps 0 and 1 waited for them, bounded); free the columns.
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 64;\n" ::"r"(tmem) : "memory");
  }
}

// ---------------------------------------------------------------------------
// k_compact: grid (row chunks, Hkv, B), 256 threads.  Writes the compacted
// cache of one (sequence, kv-head): the rows before the visual span, the kept
// visual rows in their order, then the rows after the span (vp_compact_kv).
// Each thread copies 16-byte pieces; a warp covers whole rows, so the reads
// of consecutive kept rows and of the text rows are coalesced per row.
// ---------------------------------------------------------------------------
constexpr int kCompactRows = 128;  // destination rows per CTA

__global__ void __launch_bounds__(256) k_compact(const __grid_constant__ CompactParams c) {
  // kept_idx / kept_count may come from the previous kernel.  No early
  // trigger: the next call may read the caches written here before its own
  // wait, so it starts only once this grid has completed.
  pdl_wait();
  const int g = blockIdx.y, b = blockIdx.z;
  int vs = __ldg(c.vis_start + b), nv = __ldg(c.vis_len + b), tl = __ldg(c.text_len + b);
  unsigned e = 0;
  if (nv < 0 || nv > c.max_visual) { e |= ERR_SPAN; nv = min(max(nv, 0), c.max_visual); }
  if (tl < 1) { e |= ERR_TEXT; tl = 1; }
  if (nv + tl > c.max_seq) { e |= ERR_LEN; tl = max(1, c.max_seq - nv); }
  if (vs < 0 || vs > tl) { e |= ERR_SPAN; vs = min(max(vs, 0), tl); }
  int K = __ldcg(c.kept_count + b);
  if (K < 0 || K > min(c.kept_cap, nv)) { e |= ERR_KEPT; K = max(0, min(K, min(c.kept_cap, nv))); }
  const int Tn = K + tl;  // rows of the compacted sequence
  const int ppr = c.D * c.esz / 16;  // 16-byte pieces per row
  const int rpi = 256 / ppr;         // rows per pass of the CTA
  const int r0 = blockIdx.x * kCompactRows, r1 = min(Tn, r0 + kCompactRows);
  const char* src = static_cast<const char*>(c.src.data);
  char* dst = static_cast<char*>(c.dst);
  for (int t = r0 + threadIdx.x / ppr; t < r1; t += rpi) {
    const int piece = threadIdx.x % ppr;
    int pos;  // source row
    if (t < vs) {
      pos = t;
    } else if (t < vs + K) {
      const int i = __ldcg(c.kept_idx + (int64_t)b * c.kept_cap + (t - vs));
      pos = (i >= 0 && i < nv) ? vs + i : -1;
      if (pos < 0) e |= ERR_KEPT;
    } else {
      pos = t - K + nv;
    }
    const char* row = nullptr;
    if (pos >= 0) {
      if (c.paged) {
        const int lp = pos >> c.page_shift;
        const int page = lp < c.src.max_pages ? __ldg(c.src.block_table + (int64_t)b * c.src.max_pages + lp) : -1;
        if (page >= 0 && page < c.src.num_pages)
          row = src + ((int64_t)page * c.src.sb + (int64_t)g * c.src.sh + (int64_t)(pos & (c.page_size - 1)) * c.src.st) * c.esz;
        else
          e |= ERR_PAGE;
      } else {
        row = src + ((int64_t)b * c.src.sb + (int64_t)g * c.src.sh + (int64_t)pos * c.src.st) * c.esz;
      }
    }
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (row) v = __ldg(reinterpret_cast<const uint4*>(row) + piece);
    reinterpret_cast<uint4*>(dst + ((int64_t)b * c.dsb + (int64_t)g * c.dsh + (int64_t)t * c.dst_t) * c.esz)[piece] = v;
  }
  if (e) atomicOr(c.err, e);
}

// ---------------------------------------------------------------------------
// k_score_f32 (fp32 caches): lane-per-token dot products on the FMA pipes,
// lane-per-dimension P.V; the same partials as k_score_mma.
// ---------------------------------------------------------------------------
template <int D, int GM>
struct F32Smem {
  float q[GM][D];
  float pr[kWarps][GM][32];
  const float* vrow[kWarps][32];
  float wst[kWarps][GM][ST_N];
  float ow[kWarps][GM][D];
  ScoreTail<GM, D> tail;
};

template <int D, int GM>
__device__ __forceinline__ void dot_row_f32(const float* row, const float (*q_s)[D], float (&z)[GM]) {
#pragma unroll
  for (int h = 0; h < GM; ++h) z[h] = 0.f;
#pragma unroll 4
  for (int d0 = 0; d0 < D; d0 += 4) {
    float kf[4];
    load_f<4>(row + d0, kf);
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      const float4 qv = *reinterpret_cast<const float4*>(&q_s[h][d0]);
      z[h] = fmaf(qv.x, kf[0], z[h]);
      z[h] = fmaf(qv.y, kf[1], z[h]);
      z[h] = fmaf(qv.z, kf[2], z[h]);
      z[h] = fmaf(qv.w, kf[3], z[h]);
    }
  }
}

template <int D, int GM>
__global__ void __launch_bounds__(kThreads) k_score_f32(const __grid_constant__ StepParams p) {
  constexpr int DPL = D / 32;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  auto& sm = *reinterpret_cast<F32Smem<D, GM>*>(smem_raw);
  const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait();
  const int G = p.G, H = p.H;
  const Seq sq = load_seq(p, b, s == 0 && g == 0);
  const float* qb = reinterpret_cast<const float*>(p.q) + ((int64_t)b * H + g * G) * D;
  for (int i = threadIdx.x; i < GM * D; i += kThreads) {
    const int h = i / D, d = i % D;
    sm.q[h][d] = h < G ? qb[h * D + d] : 0.f;
  }
  __syncthreads();
  const SplitRange rg = split_range(sq, s, p.ns);

  float m_v[GM], l1v[GM], ltv[GM], m_t[GM], l1t[GM], ltt[GM], acc[GM][DPL];
#pragma unroll
  for (int h = 0; h < GM; ++h) {
    m_v[h] = m_t[h] = -CUDART_INF_F;
    l1v[h] = ltv[h] = l1t[h] = ltt[h] = 0.f;
#pragma unroll
    for (int j = 0; j < DPL; ++j) acc[h][j] = 0.f;
  }
  unsigned err = 0;

  for (int base = rg.va + warp * 32; base < rg.vb; base += kWarps * 32) {
    const int i = base + lane;
    bool valid = i < rg.vb;
    float z[GM];
    if (valid) {
      const float* row = kv_row<float>(p.k, p, b, g, sq.vs + i);
      if (row) dot_row_f32<D, GM>(row, sm.q, z); else { valid = false; err |= ERR_PAGE; }
    }
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      if (h >= G) break;
      const float zz = valid ? z[h] * p.c_log2 : -CUDART_INF_F;
      if (i < rg.vb) p.z_ws[((int64_t)b * p.max_visual + i) * p.hp + g * G + h] = zz;
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

  for (int base = rg.ta + warp * 32; base < rg.tb; base += kWarps * 32) {
    const int ti = base + lane;
    bool valid = ti < rg.tb;
    const int pos = text_pos(sq, ti);
    float z[GM];
    const float* vrow = nullptr;
    if (valid) {
      const float* row = kv_row<float>(p.k, p, b, g, pos);
      vrow = kv_row<float>(p.v, p, b, g, pos);
      if (row && vrow) dot_row_f32<D, GM>(row, sm.q, z); else { valid = false; vrow = nullptr; err |= ERR_PAGE; }
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
      sm.pr[warp][h][lane] = pr;
    }
    sm.vrow[warp][lane] = vrow;
    __syncwarp();
    const int nt = min(32, rg.tb - base);
    for (int t0 = 0; t0 < nt; t0 += 4) {
      float vv[4][DPL];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float* vr = t0 + u < nt ? sm.vrow[warp][t0 + u] : nullptr;
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
          const float pr = t0 + u < nt ? sm.pr[warp][h][t0 + u] : 0.f;
#pragma unroll
          for (int j = 0; j < DPL; ++j) acc[h][j] = fmaf(pr, vv[u][j], acc[h][j]);
        }
      }
    }
    __syncwarp();
  }
  pdl_trigger();
  if (err) atomicOr(p.err, err);

#pragma unroll
  for (int h = 0; h < GM; ++h) {
    const float a = warp_sum(l1v[h]), bb = warp_sum(ltv[h]);
    const float c = warp_sum(l1t[h]), d = warp_sum(ltt[h]);
    if (lane == 0) {
      sm.wst[warp][h][ST_MV] = m_v[h]; sm.wst[warp][h][ST_L1V] = a; sm.wst[warp][h][ST_LTV] = bb;
      sm.wst[warp][h][ST_MT] = m_t[h]; sm.wst[warp][h][ST_L1T] = c; sm.wst[warp][h][ST_LTT] = d;
      sm.wst[warp][h][3] = sm.wst[warp][h][7] = 0.f;
    }
#pragma unroll
    for (int j = 0; j < DPL; ++j) sm.ow[warp][h][lane * DPL + j] = acc[h][j];
  }
  score_epilogue<GM, D>(p, b, g, s, sm.wst, &sm.ow[0][0][0], GM * D, sm.tail);
}

// ---------------------------------------------------------------------------
// k_select: grid (cl, granularity ? Hkv : 1, B) in clusters of cl CTAs of
// 512 threads (1024 when a rank's slice of the visual tokens is long).
// Dynamic shared memory: the N_v score keys, of which rank 0's copy is used.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int budget_k(const StepParams& p, float m_max, int nv) {
  if (nv <= 0) return 0;
  switch (p.mode) {
    case MODE_DENSE: return nv;
    case MODE_TOP_P: return 0;  // decided by the radix select over the score sums
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

// The cut of the Top-K set (Eq. 3) found by a radix select over score keys
// (float bits of non-negative scores, which order like the scores).
struct RadixCut {
  uint32_t theta;    // keys above theta are kept
  unsigned krem;     // keys equal to theta to keep (the lowest-index ones)
  unsigned n_theta;  // keys equal to theta (last pass only)
  bool whole;        // the cut fell on a bucket boundary: keep every key >= theta + 1
};

template <int NTH>
__global__ void __launch_bounds__(NTH) k_select(const __grid_constant__ StepParams p) {
  constexpr int NW = NTH / 32;
  extern __shared__ __align__(16) uint32_t key_s[];  // [max_visual] score keys (rank 0's copy is used)
  __shared__ float hM_s[kMaxHeads], hInv_s[kMaxHeads], hMass_s[kMaxHeads], hMass1_s[kMaxHeads];
  __shared__ unsigned hist_s[3][256];  // one per radix pass, used in turn
  __shared__ int wsum_s[32];
  __shared__ int sh_i[4];
  __shared__ int act_s, act_rank_s[8];  // active-token counts (diagnostics)
  __shared__ float hsum_s[3][256];      // top-p: score sums per digit
  __shared__ float vsum_s, vsum_rank_s[8];

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank(), ncl = (int)cluster.num_blocks();
  const int gsel = blockIdx.y, b = blockIdx.z, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < 3 * 256; i += NTH) (&hist_s[0][0])[i] = 0;
  if (tid == 0) { act_s = 0; vsum_s = 0.f; }
  const bool topp = p.mode == MODE_TOP_P;
  if (topp)
    for (int i = tid; i < 3 * 256; i += NTH) (&hsum_s[0][0])[i] = 0.f;
  const Seq sq = load_seq(p, b, false);  // an input: read before the wait
  pdl_wait();
  pdl_trigger();
  const int H = p.H, ns = p.ns;
  const float inv_tau = p.inv_tau;

  // 1. Split statistics -> per-head max, normalisers and masses (Eq. 5, Eq. 6).
  //    Warp w merges heads w, w + NW, ...; lane l folds splits l, l + 32, ...
  //    in a running (max, sums) state and the warp merges the lanes.  The
  //    first records are requested together with the sequence lengths, and
  //    each head's records while the previous head is being merged.
  const float* stb = p.split_st + (int64_t)b * H * p.nsp_max * ST_N;
  auto fetch = [&](int h, int s, float4& x, float4& y) {  // x: text (M, L1, Ltau), y: visual
    if (h < H && s < ns) {
      const float4* r = reinterpret_cast<const float4*>(stb + ((int64_t)h * p.nsp_max + s) * ST_N);
      x = __ldcg(r);
      y = __ldcg(r + 1);
    } else {
      x = y = make_float4(-CUDART_INF_F, 0.f, 0.f, 0.f);
    }
  };
  float4 cx0, cy0, cx1, cy1;
  fetch(warp, lane, cx0, cy0);
  fetch(warp, lane + 32, cx1, cy1);
  const int nv = sq.nv;
  // This rank's slice of the visual tokens; its first logit row is requested
  // now so that it arrives while the statistics are merged (heads up to 32;
  // at 1024 threads the registers are too few for it).
  const int per = (nv + ncl - 1) / ncl;
  const int i0 = min(nv, rank * per), i1 = min(nv, i0 + per);
  const int hbeg = p.granularity ? gsel * p.G : 0;
  const int hcnt = p.granularity ? p.G : H;
  const bool vec = (hbeg & 3) == 0 && (hcnt & 3) == 0;
  // Long slices (the 1024-thread form, slices above kSelSliceSmall) take the
  // row-shared importance loop below; short ones (the B = 1 decode) request
  // each thread's first row now.  The 512-thread form is compiled without the
  // row-shared loop: its launches are latency-bound, and the larger code
  // measured slower there.
  const bool wide = NTH >= 1024 && vec && hcnt >= 4 && hcnt <= 32 && (i1 - i0) > 2 * NTH;
  const bool pre = !wide && NTH <= 512 && vec && hcnt <= 32 && i0 + tid < i1;
  float4 zpre[8];
  if (pre) {
    const float4* zr = reinterpret_cast<const float4*>(p.z_ws + ((int64_t)b * p.max_visual + i0 + tid) * p.hp + hbeg);
#pragma unroll
    for (int q = 0; q < 8; ++q) zpre[q] = 4 * q < hcnt ? __ldcg(zr + q) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  for (int h = warp; h < H; h += NW) {
    float4 nx0, ny0, nx1, ny1;
    fetch(h + NW, lane, nx0, ny0);
    fetch(h + NW, lane + 32, nx1, ny1);
    float m = -CUDART_INF_F, a1v = 0.f, atv = 0.f, a1t = 0.f, att = 0.f;
    auto fold = [&](const float4& x, const float4& y) {
      const float mn = fmaxf(m, fmaxf(x.x, y.x));
      if (mn > m) {
        const float f1 = exp2_rel(m, mn), ft = exp2_tau(m, mn, inv_tau);
        a1v *= f1; a1t *= f1; atv *= ft; att *= ft;
        m = mn;
      }
      a1v = fmaf(exp2_rel(y.x, m), y.y, a1v);
      atv = fmaf(exp2_tau(y.x, m, inv_tau), y.z, atv);
      a1t = fmaf(exp2_rel(x.x, m), x.y, a1t);
      att = fmaf(exp2_tau(x.x, m, inv_tau), x.z, att);
    };
    fold(cx0, cy0);
    fold(cx1, cy1);
    for (int s = lane + 64; s < ns; s += 32) {
      float4 x, y;
      fetch(h, s, x, y);
      fold(x, y);
    }
    const float M = warp_max(m);
    const float f1 = exp2_rel(m, M), ft = exp2_tau(m, M, inv_tau);
    const float L1v = warp_sum(a1v * f1), Ltv = warp_sum(atv * ft);
    const float L1t = warp_sum(a1t * f1), Ltt = warp_sum(att * ft);
    if (lane == 0) {
      const float L1 = L1v + L1t, Lt = Ltv + Ltt;
      hM_s[h] = M;
      hInv_s[h] = L1 > 0.f ? 1.f / L1 : 0.f;
      hMass_s[h] = Lt > 0.f ? Ltv / Lt : 0.f;
      hMass1_s[h] = L1 > 0.f ? L1v / L1 : 0.f;
    }
    cx0 = nx0; cy0 = ny0; cx1 = nx1; cy1 = ny1;
  }
  __syncthreads();

  // 2. Rank 0: head mean, head max (Sec. 4.3) and the budget (Eq. 7).
  const int nsel = p.granularity ? p.Hkv : 1;
  if (rank == 0) {
    if (warp == 0) {
      float sm = 0.f, mx = 0.f, s1 = 0.f;
      for (int h = lane; h < H; h += 32) {
        sm += hMass_s[h];
        mx = fmaxf(mx, hMass_s[h]);
        s1 += hMass1_s[h];
      }
      sm = warp_sum(sm);
      mx = warp_max(mx);
      s1 = warp_sum(s1);
      if (lane == 0) {
        const int K = min(budget_k(p, mx, nv), p.kept_cap);
        sh_i[0] = K;
        if (!topp) p.kept_count[(int64_t)b * nsel + gsel] = K;  // top-p: after the select
        if (gsel == 0 && p.mass_stats) {
          float* ms = p.mass_stats + (int64_t)b * 4;
          ms[0] = sm / H; ms[1] = mx; ms[2] = s1 / H;
          if (!topp) ms[3] = (float)K;
        }
      }
    } else if (gsel == 0) {
      for (int h = tid - 32; h < H; h += NTH - 32) {
        p.mass[(int64_t)b * H + h] = hMass_s[h];
        p.hmax[(int64_t)b * H + h] = hM_s[h];
      }
    }
  }

  // 3. Importance S_i (Eq. 2) of this rank's slice of the visual tokens, as
  //    float bits (S >= 0 orders like its bits), into rank 0's key array.
  const float inv_cnt = 1.f / (float)hcnt;
  uint32_t* key0 = ncl > 1 ? cluster.map_shared_rank(key_s, 0) : key_s;
  unsigned bad = 0;
  const bool diag = p.n_act || p.act_bits;
  int n_on = 0;
  float vsum = 0.f;  // top-p: this thread's share of the visual score total
  auto emit = [&](int i, float a) {  // a: sum over the heads of exp2(z - M_h) / L_h
    const float sc = a * inv_cnt;
    if (!isfinite(sc)) bad = 1;
    key0[i] = __float_as_uint(sc);
    vsum += sc;
    if (diag && __float_as_uint(sc) > p.act_delta_bits) {  // S_i > delta (Sec. 4.3)
      ++n_on;
      if (p.act_bits) atomicOr(p.act_bits + ((int64_t)b * nsel + gsel) * p.act_words + (i >> 5), 1u << (i & 31));
    }
  };
  // Long slices: LPT lanes share a token row, each reading one float4 of its
  // heads, so that a warp's load covers consecutive rows; eight loads per
  // lane are in flight, and a reduce-scatter over the LPT lanes leaves every
  // lane whole-token sums to emit.
  auto wide_loop = [&](auto lpt_tag) {
    constexpr int LPT = decltype(lpt_tag)::value, TPI = 32 / LPT, V = 8;
    const int Q = hcnt / 4, lq = lane % LPT;
    const bool qok = lq < Q;
    float m4[4], i4[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int h = hbeg + 4 * lq + c;
      m4[c] = qok ? hM_s[h] : 0.f;
      i4[c] = qok ? hInv_s[h] : 0.f;
    }
    const float* zb = p.z_ws + (int64_t)b * p.max_visual * p.hp + hbeg + 4 * lq;
    int off = 0;  // first of this lane's V / LPT values after the reduce-scatter
#pragma unroll
    for (int s_ = 0; s_ < 3; ++s_)
      if ((LPT >> (s_ + 1)) > 0 && (lane & (LPT >> (s_ + 1)))) off += V >> (s_ + 1);
    for (int base = i0 + warp * V * TPI; base < i1; base += NW * V * TPI) {
      float4 zz[V];
#pragma unroll
      for (int j = 0; j < V; ++j) {
        const int tok = base + j * TPI + lane / LPT;
        zz[j] = (qok && tok < i1) ? __ldcg(reinterpret_cast<const float4*>(zb + (int64_t)tok * p.hp))
                                  : make_float4(-CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F, -CUDART_INF_F);
      }
      float v[V];
#pragma unroll
      for (int j = 0; j < V; ++j) {
        float a = fexp2_rel(zz[j].x, m4[0]) * i4[0];
        a = fmaf(fexp2_rel(zz[j].y, m4[1]), i4[1], a);
        a = fmaf(fexp2_rel(zz[j].z, m4[2]), i4[2], a);
        v[j] = fmaf(fexp2_rel(zz[j].w, m4[3]), i4[3], a);
      }
#pragma unroll
      for (int s_ = 0; s_ < 3; ++s_) {
        const int o = LPT >> (s_ + 1), half = V >> (s_ + 1);
        if (o == 0) break;
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int k = 0; k < half; ++k) {
          const float send = up ? v[k] : v[k + half];
          const float keep = up ? v[k + half] : v[k];
          v[k] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
      }
#pragma unroll
      for (int k = 0; k < V / LPT; ++k) {
        const int tok = base + (k + off) * TPI + lane / LPT;
        if (tok < i1) emit(tok, v[k]);
      }
    }
  };
  bool done = false;
  if constexpr (NTH >= 1024) {
    if (wide) {
      const int Q = hcnt / 4;
      if (Q <= 1) wide_loop(std::integral_constant<int, 1>{});
      else if (Q <= 2) wide_loop(std::integral_constant<int, 2>{});
      else if (Q <= 4) wide_loop(std::integral_constant<int, 4>{});
      else wide_loop(std::integral_constant<int, 8>{});
      done = true;
    }
  }
  if (!done) {
    for (int i = i0 + tid; i < i1; i += NTH) {
      const float* zr = p.z_ws + ((int64_t)b * p.max_visual + i) * p.hp + hbeg;
      float a = 0.f;
      if (pre && i == i0 + tid) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (4 * q < hcnt) {
            const int h = hbeg + 4 * q;
            a = fmaf(fexp2_rel(zpre[q].x, hM_s[h]), hInv_s[h], a);
            a = fmaf(fexp2_rel(zpre[q].y, hM_s[h + 1]), hInv_s[h + 1], a);
            a = fmaf(fexp2_rel(zpre[q].z, hM_s[h + 2]), hInv_s[h + 2], a);
            a = fmaf(fexp2_rel(zpre[q].w, hM_s[h + 3]), hInv_s[h + 3], a);
          }
        }
      } else if (vec) {
        for (int hh = 0; hh < hcnt; hh += 4) {
          const float4 z4 = __ldcg(reinterpret_cast<const float4*>(zr + hh));
          const int h = hbeg + hh;
          a = fmaf(fexp2_rel(z4.x, hM_s[h]), hInv_s[h], a);
          a = fmaf(fexp2_rel(z4.y, hM_s[h + 1]), hInv_s[h + 1], a);
          a = fmaf(fexp2_rel(z4.z, hM_s[h + 2]), hInv_s[h + 2], a);
          a = fmaf(fexp2_rel(z4.w, hM_s[h + 3]), hInv_s[h + 3], a);
        }
      } else {
        for (int hh = 0; hh < hcnt; ++hh)
          a = fmaf(fexp2_rel(__ldcg(zr + hh), hM_s[hbeg + hh]), hInv_s[hbeg + hh], a);
      }
      emit(i, a);
    }
  }
  if (bad) atomicOr(p.err, ERR_NONFINITE);
  if (p.n_act || topp) {  // this rank's count and score total, into rank 0's slots
    n_on = __reduce_add_sync(0xffffffffu, n_on);
    vsum = warp_sum(vsum);
    if (lane == 0 && n_on) atomicAdd(&act_s, n_on);
    if (lane == 0 && topp) atomicAdd(&vsum_s, vsum);
    __syncthreads();
    if (tid == 0) {
      (ncl > 1 ? cluster.map_shared_rank(act_rank_s, 0) : act_rank_s)[rank] = act_s;
      (ncl > 1 ? cluster.map_shared_rank(vsum_rank_s, 0) : vsum_rank_s)[rank] = vsum_s;
    }
  }
  if (ncl > 1) cluster.sync();  // rank 0 now sees every key (and its own K)
  else __syncthreads();
  if (rank != 0) return;

  if (p.n_act && tid == 0) {
    int n = 0;
    for (int r = 0; r < ncl; ++r) n += act_rank_s[r];
    p.n_act[(int64_t)b * nsel + gsel] = n;
  }
  int K = sh_i[0];
  int32_t* kept = p.kept_idx + ((int64_t)b * nsel + gsel) * p.kept_cap;

  // 4. Radix select of the K-th largest key, 8 bits per pass from the top;
  //    lanes holding the same digit add to the histogram once per warp.  One
  //    barrier per pass: every warp scans the finished histogram itself, and
  //    pass p clears the buffer of pass p - 2 for pass p + 1.  (The same cut
  //    as radix_cut, written out here: at 1024 threads this kernel runs at the
  //    64-register limit, and with the shared routine it spilled more.)
  uint32_t theta = 0;
  unsigned krem = 0, n_theta = 0;  // keys equal to theta: to keep, in total
  if (topp) {
    // Top-p budget (App. A.2): the fewest top keys whose scores reach a share
    // p of the visual total.  Radix select over the score mass: each pass
    // keeps every digit above the one where the remaining mass is reached.
    float total = 0.f;
    for (int r = 0; r < ncl; ++r) total += vsum_rank_s[r];
    K = 0;
    if (nv > 0 && p.ratio_ppm >= 1000000) {
      K = nv;
    } else if (nv > 0 && p.ratio_ppm > 0) {
      float need = (float)p.ratio_ppm * 1e-6f * total;  // score mass still to cover
      unsigned above = 0;                                // keys above the current bucket
      uint32_t prefix = 0, mask = 0;
      bool all = false;
      for (int pass = 0; pass < 4 && !all; ++pass) {
        const int shift = 24 - 8 * pass;
        unsigned* hist = hist_s[pass % 3];
        float* hsum = hsum_s[pass % 3];
        if (pass >= 2)
          for (int i = tid; i < 256; i += NTH) { hist_s[(pass + 1) % 3][i] = 0; hsum_s[(pass + 1) % 3][i] = 0.f; }
        for (int base = 0; base < nv; base += NTH) {
          const int i = base + tid;
          const uint32_t kk = i < nv ? key_s[i] : 0u;
          const bool m = i < nv && (kk & mask) == prefix;
          const unsigned dg = (kk >> shift) & 255u;
          const unsigned act = __ballot_sync(0xffffffffu, m);
          if (act) {
            const int leader = __ffs(act) - 1;
            const unsigned d0 = __shfl_sync(0xffffffffu, dg, leader);
            if (__all_sync(0xffffffffu, !m || dg == d0)) {
              const float ws = warp_sum(m ? __uint_as_float(kk) : 0.f);
              if (lane == leader) { atomicAdd(&hist[d0], (unsigned)__popc(act)); atomicAdd(&hsum[d0], ws); }
            } else if (m) {
              atomicAdd(&hist[dg], 1u);
              atomicAdd(&hsum[dg], __uint_as_float(kk));
            }
          }
        }
        __syncthreads();
        unsigned cc[8], ctot = 0;
        float cs[8], stot = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          cc[j] = hist[255 - 8 * lane - j]; ctot += cc[j];
          cs[j] = hsum[255 - 8 * lane - j]; stot += cs[j];
        }
        unsigned cin = ctot;
        float sin_ = stot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned nc = __shfl_up_sync(0xffffffffu, cin, o);
          const float ns_ = __shfl_up_sync(0xffffffffu, sin_, o);
          if (lane >= o) { cin += nc; sin_ += ns_; }
        }
        const unsigned cex = cin - ctot;
        const float sex = sin_ - stot;
        const bool mine = sex < need && need <= sin_ && ctot > 0;
        unsigned dsel = 0, cnt_before = 0, cnt = 0;
        float sum_before = 0.f;
        if (mine) {
          // The lane's own running sum may round differently from the scan:
          // without a digit reaching the mass, its last non-empty digit holds it.
          unsigned cr = cex;
          float sr = sex;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (cc[j] > 0) { dsel = 255 - 8 * lane - j; cnt_before = cr; sum_before = sr; cnt = cc[j]; }
            if (cc[j] > 0 && sr + cs[j] >= need) break;
            cr += cc[j];
            sr += cs[j];
          }
        }
        const unsigned found = __ballot_sync(0xffffffffu, mine && cnt > 0);
        if (!found) { all = true; break; }  // rounding left the mass short: keep every candidate
        const int src = __ffs(found) - 1;
        dsel = __shfl_sync(0xffffffffu, dsel, src);
        cnt_before = __shfl_sync(0xffffffffu, cnt_before, src);
        sum_before = __shfl_sync(0xffffffffu, sum_before, src);
        cnt = __shfl_sync(0xffffffffu, cnt, src);
        above += cnt_before;
        need -= sum_before;
        prefix |= dsel << shift;
        mask |= 255u << shift;
        if (shift == 0) n_theta = cnt;
      }
      if (all) {
        K = nv;
      } else {
        theta = prefix;
        const float tv = __uint_as_float(theta);
        unsigned m_eq = tv > 0.f ? (unsigned)ceilf(need / tv) : n_theta;
        m_eq = max(1u, min(m_eq, n_theta));
        krem = m_eq;
        K = (int)(above + m_eq);
      }
    }
    K = min(K, p.kept_cap);
    if (tid == 0) {
      p.kept_count[(int64_t)b * nsel + gsel] = K;
      if (gsel == 0 && p.mass_stats) p.mass_stats[(int64_t)b * 4 + 3] = (float)K;
    }
    if (K >= nv) krem = 0;
  }
  bool take_all = K >= nv;
  bool whole = false;  // the radix select stopped at a bucket kept whole (no tie to split)
  if (!topp && K > 0 && !take_all) {
    uint32_t prefix = 0, mask = 0;
    krem = (unsigned)K;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      unsigned* hist = hist_s[pass % 3];
      if (pass >= 2)  // the buffer of pass - 2, scanned by every warp before the last barrier
        for (int i = tid; i < 256; i += NTH) hist_s[(pass + 1) % 3][i] = 0;
      for (int base = 0; base < nv; base += NTH) {
        const int i = base + tid;
        const uint32_t k = i < nv ? key_s[i] : 0u;
        const bool m = i < nv && (k & mask) == prefix;
        const unsigned dg = (k >> shift) & 255u;
        const unsigned act = __ballot_sync(0xffffffffu, m);
        if (act) {
          const int leader = __ffs(act) - 1;
          const unsigned d0 = __shfl_sync(0xffffffffu, dg, leader);
          if (__all_sync(0xffffffffu, !m || dg == d0)) {
            if (lane == leader) atomicAdd(&hist[d0], (unsigned)__popc(act));
          } else if (m) {
            atomicAdd(&hist[dg], 1u);
          }
        }
      }
      __syncthreads();
      // Lane L owns digits 255-8L ... 248-8L (descending).
      unsigned c[8], tot = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) { c[j] = hist[255 - 8 * lane - j]; tot += c[j]; }
      unsigned incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      const unsigned excl = incl - tot;
      const bool mine = excl < krem && krem <= incl;
      unsigned dsel = 0, before = 0, cnt = 0;
      if (mine) {
        unsigned run = excl;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (run + c[j] >= krem) { dsel = 255 - 8 * lane - j; before = run; cnt = c[j]; break; }
          run += c[j];
        }
      }
      const int src = max(__ffs(__ballot_sync(0xffffffffu, mine)) - 1, 0);
      dsel = __shfl_sync(0xffffffffu, dsel, src);
      before = __shfl_sync(0xffffffffu, before, src);
      cnt = __shfl_sync(0xffffffffu, cnt, src);
      krem -= before;
      prefix |= dsel << shift;
      mask |= 255u << shift;
      if (shift == 0) n_theta = cnt;
      if (shift > 0 && krem == cnt) {  // the whole bucket is kept: the threshold is its lowest key
        whole = true;
        break;
      }
    }
    // The K-th largest key (krem keys equal to it are kept), or, when a
    // bucket is kept whole, every key from its lowest possible value up.
    theta = whole ? prefix - 1u : prefix;
  }

  // 5. Ascending compaction: keys above theta, plus the first krem equal keys
  //    (every equal key when there is no tie to break: one scan less).
  if (K > 0) {
    // An odd chunk length keeps the threads' reads in distinct banks.
    const int per_t = ((nv + NTH - 1) / NTH) | 1;
    const int j0 = min(nv, tid * per_t), j1 = min(nv, j0 + per_t);
    const bool ties = !take_all && !whole && krem < n_theta;
    int n_eq = 0;
    if (ties)
      for (int i = j0; i < j1; ++i) n_eq += key_s[i] == theta;
    const int eq_before = ties ? block_excl_scan(n_eq, wsum_s) : 0;
    if (!ties) krem = 0xffffffffu;
    int n_sel = 0;
    {
      int r = eq_before;
      for (int i = j0; i < j1; ++i) {
        const uint32_t k = key_s[i];
        const bool sel = take_all || k > theta || (!whole && k == theta && (unsigned)r < krem);
        r += k == theta;
        n_sel += sel;
      }
    }
    int o = block_excl_scan(n_sel, wsum_s);
    int r = eq_before;
    for (int i = j0; i < j1; ++i) {
      const uint32_t k = key_s[i];
      const bool sel = take_all || k > theta || (!whole && k == theta && (unsigned)r < krem);
      r += k == theta;
      if (sel && o < K) kept[o++] = i;
    }
  }
  for (int i = max(K, 0) + tid; i < p.kept_cap; i += NTH) kept[i] = -1;
}

// Chunk gather, part (b): dimension slice c of the text partials of the
// score splits, merged (c < nm) into mt_o / mt_st.
template <int D, int GM, int NTHR>
__device__ void gather_text_slice(const StepParams& p, int c, int64_t hrow0, float (*tw)[kNsMax], float (*tl)[kNsMax]) {
  constexpr int D4 = D / 4;
  const int tid = threadIdx.x, G = p.G, ns = p.ns;
  for (int i = tid; i < G * ns; i += NTHR) {
    const int h = i / ns, s = i % ns;
    const float2 r = __ldcg(reinterpret_cast<const float2*>(p.split_st + ((hrow0 + h) * p.nsp_max + s) * ST_N));
    tw[h][s] = r.x;  // ST_MT
    tl[h][s] = r.y;  // ST_L1T
  }
  __syncthreads();
  if (tid < G) {
    const int h = tid;
    float M = -CUDART_INF_F;
    for (int s = 0; s < ns; ++s) M = fmaxf(M, tw[h][s]);
    float L = 0.f;
    for (int s = 0; s < ns; ++s) {
      const float w = exp2_rel(tw[h][s], M);
      tw[h][s] = w;
      L = fmaf(w, tl[h][s], L);
    }
    if (c == 0) {
      p.mt_st[(hrow0 + h) * 2 + 0] = M;
      p.mt_st[(hrow0 + h) * 2 + 1] = L;
    }
  }
  __syncthreads();
  const int s4 = D4 / p.nm;  // float4s of this CTA's slice, per head
  for (int i = tid; i < G * s4; i += NTHR) {
    const int h = i / s4, d = 4 * (c * s4 + i % s4);
    const float* so = p.split_o + (hrow0 + h) * p.nsp_max * D + d;
    float4 num = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
    for (int s = 0; s < ns; ++s) {
      const float4 v = __ldcg(reinterpret_cast<const float4*>(so + (int64_t)s * D));
      const float w = tw[h][s];
      num.x = fmaf(w, v.x, num.x); num.y = fmaf(w, v.y, num.y); num.z = fmaf(w, v.z, num.z); num.w = fmaf(w, v.w, num.w);
    }
    *reinterpret_cast<float4*>(p.mt_o + (hrow0 + h) * D + d) = num;
  }
}

// Chunk gather, finish: the last CTA of (sequence, kv-head) to arrive combines
// the text output with the kept chunks (log-sum-exp form) and writes out.
// The text part is the merged slice output, or the single split partial.
template <typename T, int D, int GM, int NTHR>
__device__ void gather_finish(const StepParams& p, int b, int g, int64_t hrow0, int64_t pbase,
                              float (*tw)[kNsMax], float (*fin)[4], int* last) {
  constexpr int D4 = D / 4;
  const int tid = threadIdx.x, G = p.G;
  __threadfence();
  __syncthreads();
  if (tid == 0) *last = atomicAdd(p.tickets + (int64_t)b * p.Hkv + g, 1u) == (unsigned)p.nc - 1u;
  __syncthreads();
  if (!*last) return;
  __threadfence();
  const float* t_o = p.nm ? p.mt_o + hrow0 * D : p.split_o + hrow0 * p.nsp_max * D;
  const int t_ostride = p.nm ? D : p.nsp_max * D;
  if (tid < G) {
    const int h = tid;
    float mt, lt;
    if (p.nm) {
      mt = __ldcg(p.mt_st + (hrow0 + h) * 2);
      lt = __ldcg(p.mt_st + (hrow0 + h) * 2 + 1);
    } else {
      mt = __ldcg(p.split_st + (hrow0 + h) * p.nsp_max * ST_N + ST_MT);
      lt = __ldcg(p.split_st + (hrow0 + h) * p.nsp_max * ST_N + ST_L1T);
    }
    float M = mt;
    for (int k = 0; k < p.nk; ++k) M = fmaxf(M, __ldcg(p.gpart_st + ((pbase + k) * G + h) * 2));
    const float wt = exp2_rel(mt, M);
    float den = wt * lt;
    for (int k = 0; k < p.nk; ++k) {
      const float w = exp2_rel(__ldcg(p.gpart_st + ((pbase + k) * G + h) * 2), M);
      tw[h][k] = w;
      den = fmaf(w, __ldcg(p.gpart_st + ((pbase + k) * G + h) * 2 + 1), den);
    }
    fin[h][0] = wt;
    fin[h][1] = den > 0.f ? 1.f / den : 0.f;
  }
  __syncthreads();
  for (int i = tid; i < G * D4; i += NTHR) {
    const int h = i / D4, d = 4 * (i % D4);
    const float wt = fin[h][0];
    const float4 tv = __ldcg(reinterpret_cast<const float4*>(t_o + (int64_t)h * t_ostride + d));
    float4 num = make_float4(wt * tv.x, wt * tv.y, wt * tv.z, wt * tv.w);
#pragma unroll 4
    for (int k = 0; k < p.nk; ++k) {
      const float4 v = __ldcg(reinterpret_cast<const float4*>(p.gpart_o + ((pbase + k) * G + h) * D + d));
      const float w = tw[h][k];
      num.x = fmaf(w, v.x, num.x); num.y = fmaf(w, v.y, num.y); num.z = fmaf(w, v.z, num.z); num.w = fmaf(w, v.w, num.w);
    }
    const float inv = fin[h][1];
    T* o = reinterpret_cast<T*>(p.out) + (hrow0 + h) * D + d;
    o[0] = from_f<T>(num.x * inv); o[1] = from_f<T>(num.y * inv);
    o[2] = from_f<T>(num.z * inv); o[3] = from_f<T>(num.w * inv);
  }
  if (tid == 0) p.tickets[(int64_t)b * p.Hkv + g] = 0u;
}

// ---------------------------------------------------------------------------
// k_gather: grid (nc, Hkv, B), 256 threads.  CTA c (a) attends over chunk c of
// the kept list (c < nk), staged 64 tokens at a time -- indices, V-row
// addresses and logits to shared memory, then each thread accumulates a
// 16-byte slice of the V rows of every (256 / slices-per-row)-th token -- and
// (b) merges dimension slice c of the text partials of the score splits
// (c < nm).  The last CTA of (sequence, kv-head) to finish combines the merged
// text output with the kept chunks and writes out.
// ---------------------------------------------------------------------------
template <typename T, int D, int GM>
struct GatherSmem {
  const T* vrow[kGatherTile];
  float pz[GM][kGatherTile];
  float run[GM][4];                         // running max, sum, rescale factor
  float red[kGatherWarps / 2][GM][D];       // warp-tree reduction buffer
  float tw[GM][kNsMax];                     // text-split maxima, then weights
  float tl[GM][kNsMax];                     // text-split sums
  float fin[GM][4];
  int last;
};

template <typename T, int D, int GM>
__global__ void __launch_bounds__(kGatherThreads) k_gather(const __grid_constant__ StepParams p) {
  constexpr int CH = 16 / sizeof(T);          // elements per 16-byte slice
  constexpr int CPR = D / CH;                 // slices per row
  constexpr int SLOTS = kGatherThreads / CPR; // tokens processed side by side
  static_assert(kGatherThreads % CPR == 0 && CPR <= 32, "row slicing");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  auto& sm = *reinterpret_cast<GatherSmem<T, D, GM>*>(smem_raw);
  const int c = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int slot = tid / CPR, ch = tid % CPR;

  pdl_wait();
  pdl_trigger();
  const int G = p.G, H = p.H;
  const int64_t hrow0 = (int64_t)b * H + g * G;
  const int64_t pbase = ((int64_t)b * p.Hkv + g) * p.nk_max;
  unsigned err = 0;

  // (a) kept chunk c
  if (c < p.nk) {
    const Seq sq = load_seq(p, b, false);
    const int sel = p.granularity ? b * p.Hkv + g : b;
    const int K = max(0, min(__ldcg(p.kept_count + sel), min(sq.nv, p.kept_cap)));
    const int32_t* kept = p.kept_idx + (int64_t)sel * p.kept_cap;
    const int per = (K + p.nk - 1) / p.nk;
    const int j0 = min(K, c * per), j1 = min(K, j0 + per);
    if (tid < GM) { sm.run[tid][0] = -CUDART_INF_F; sm.run[tid][1] = 0.f; sm.run[tid][2] = 0.f; }
    float acc[GM][CH];
#pragma unroll
    for (int h = 0; h < GM; ++h)
#pragma unroll
      for (int e = 0; e < CH; ++e) acc[h][e] = 0.f;
    __syncthreads();
    for (int jt = j0; jt < j1; jt += kGatherTile) {
      const int n = min(kGatherTile, j1 - jt);
      if (tid < kGatherTile) {
        const int t = tid;
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
        sm.vrow[t] = vr;
        const float* zr = p.z_ws + ((int64_t)b * p.max_visual + (i < 0 ? 0 : i)) * p.hp + g * G;
        float zv[GM];
#pragma unroll
        for (int h = 0; h < GM; ++h) zv[h] = (vr && h < G) ? __ldcg(zr + h) : -CUDART_INF_F;
#pragma unroll
        for (int h = 0; h < GM; ++h) sm.pz[h][t] = zv[h];
      }
      __syncthreads();
      // per-head tile max and running rescale (warp w handles heads w, w + 8)
      for (int h = warp; h < G; h += kGatherWarps) {
        const float z0 = sm.pz[h][lane], z1 = sm.pz[h][lane + 32];
        const float mo = sm.run[h][0];
        const float mn = fmaxf(mo, warp_max(fmaxf(z0, z1)));
        const float e0 = exp2_rel(z0, mn), e1 = exp2_rel(z1, mn);
        const float ssum = warp_sum(e0 + e1);
        sm.pz[h][lane] = e0;
        sm.pz[h][lane + 32] = e1;
        if (lane == 0) {
          const float a = exp2_rel(mo, mn);
          sm.run[h][0] = mn;
          sm.run[h][1] = sm.run[h][1] * a + ssum;
          sm.run[h][2] = a;
        }
      }
      __syncthreads();
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        if (h >= G) break;
        const float a = sm.run[h][2];
#pragma unroll
        for (int e = 0; e < CH; ++e) acc[h][e] *= a;
      }
#pragma unroll 4
      for (int t = slot; t < n; t += SLOTS) {
        const T* vr = sm.vrow[t];
        if (!vr) continue;
        float vv[CH];
        load_f<CH>(vr + ch * CH, vv);
#pragma unroll
        for (int h = 0; h < GM; ++h) {
          if (h >= G) break;
          const float pr = sm.pz[h][t];
#pragma unroll
          for (int e = 0; e < CH; ++e) acc[h][e] = fmaf(pr, vv[e], acc[h][e]);
        }
      }
      __syncthreads();
    }
    // Reduce the token slots: lanes of one warp first, then a warp tree.
#pragma unroll
    for (int o = CPR; o < 32; o <<= 1)
#pragma unroll
      for (int h = 0; h < GM; ++h)
#pragma unroll
        for (int e = 0; e < CH; ++e) acc[h][e] += __shfl_xor_sync(0xffffffffu, acc[h][e], o);
    for (int half = kGatherWarps / 2; half >= 1; half >>= 1) {
      if (warp >= half && warp < 2 * half && lane < CPR) {
#pragma unroll
        for (int h = 0; h < GM; ++h)
#pragma unroll
          for (int e = 0; e < CH; ++e) sm.red[warp - half][h][ch * CH + e] = acc[h][e];
      }
      __syncthreads();
      if (warp < half && lane < CPR) {
#pragma unroll
        for (int h = 0; h < GM; ++h)
#pragma unroll
          for (int e = 0; e < CH; ++e) acc[h][e] += sm.red[warp][h][ch * CH + e];
      }
      __syncthreads();
    }
    if (warp == 0 && lane < CPR) {
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        if (h < G) {
          float* dst = p.gpart_o + ((pbase + c) * G + h) * D + ch * CH;
#pragma unroll
          for (int e = 0; e < CH; ++e) dst[e] = acc[h][e];
        }
      }
    }
    if (tid < G) {
      p.gpart_st[((pbase + c) * G + tid) * 2 + 0] = sm.run[tid][0];
      p.gpart_st[((pbase + c) * G + tid) * 2 + 1] = sm.run[tid][1];
    }
  }

  if (c < p.nm) gather_text_slice<D, GM, kGatherThreads>(p, c, hrow0, sm.tw, sm.tl);
  if (err) atomicOr(p.err, err);
  gather_finish<T, D, GM, kGatherThreads>(p, b, g, hrow0, pbase, sm.tw, sm.fin, &sm.last);
}

// ---------------------------------------------------------------------------
// k_gather_mma (bf16): grid (nc, Hkv, B), 4 warps.  CTA c (a) attends over
// chunk c of the kept list (c < nk).  Warp w takes 32-token tiles w, w + 4,
// ... of the chunk and streams the kept V rows through a private ring of
// S slots: lane j copies row j of a tile with one bulk copy into a slot of
// padded rows (a 16-byte shift per row: conflict-free ldmatrix), and the
// token's logits with 4-byte cp.async (heads 0-3 into the row's pad bytes);
// the slot's mbarrier completes once the row bytes and every lane's logits
// have landed.  The kept-list entries are read three tiles ahead of their
// copies (the first ones in the same round trip as the kept count).  S is 1
// when no chunk holds more than one tile per warp (four CTAs share an SM);
// otherwise 3 (two CTAs per SM) or 2 (three CTAs per SM, the same bytes in
// flight per SM over more warps), whichever runs the grid in fewer waves, 3
// on a tie (a lone CTA in a short last wave keeps more copies in flight).
// The tile's logits give per-head probabilities; P.V runs on the tensor
// cores as in the score kernel (A = V^T by ldmatrix.trans, B = P^T from a
// per-warp bf16 buffer).  The warps' partials are merged in shared memory:
// the only CTA of its (sequence, kv-head) combines them with the text part
// and writes the output; otherwise they form the chunk's partial, and (b)
// and the final combine are shared with k_gather.
// ---------------------------------------------------------------------------
constexpr int kGmWarps = 4;
constexpr int kGmSlots = 3;  // ring slots of the deeper form (the other has 2)

template <int D, int NT, int S>
struct GmCfg {
  static constexpr int GM = 8 * NT;
  static constexpr int THREADS = 32 * kGmWarps;
  static constexpr int MT = D / 16;
  // 32 V rows at a pitch of 2D + 16 bytes; the pad of row j holds token j's
  // logits of heads 0-3, the other heads' logits sit in a separate array.
  static constexpr int RP = 2 * D + 16;
  static constexpr int SLOT = 32 * RP;
  static constexpr int ZX = GM - 4;
  // Kept rows per CTA: a single slot serves one tile per warp.
  static constexpr int MAX_CHUNK = S == 1 ? 32 * kGmWarps : kGmMaxChunk;
  // After part (a) the ring holds the warps' outputs, then the split weights;
  // before it, the split weights of part (b).
  static constexpr int OFF_TW = kGmWarps * GM * D * 4;
  static constexpr int RING_BYTES = kGmWarps * S * SLOT;
  static constexpr int REUSE_BYTES = OFF_TW + 2 * GM * kNsMax * 4;
  static constexpr int RING = RING_BYTES > REUSE_BYTES ? RING_BYTES : REUSE_BYTES;
  static constexpr int OFF_BAR = RING;                          // full[warps][slots]
  static constexpr int OFF_P = OFF_BAR + kGmWarps * S * 8;      // bf16 [warps][GM][32] probabilities
  static constexpr int OFF_ZX = OFF_P + kGmWarps * GM * 32 * 2; // float [warps][slots][ZX][32] logits
  static constexpr int OFF_MASK = OFF_ZX + kGmWarps * S * ZX * 32 * 4;  // copied rows per slot
  static constexpr int OFF_WST = OFF_MASK + kGmWarps * S * 4;           // float [warps][GM][2]
  static constexpr int OFF_FIN = OFF_WST + kGmWarps * GM * 2 * 4;       // float [GM][4]
  static constexpr int OFF_LAST = OFF_FIN + GM * 4 * 4;
  static constexpr size_t SMEM = (size_t)OFF_LAST + 16;
  static_assert(RP % 16 == 0 && (RP / 16) % 8 == 1, "row pitch: 16-byte aligned rows, one bank group apart");
  static_assert(OFF_BAR % 8 == 0 && OFF_P % 16 == 0 && OFF_ZX % 16 == 0 && OFF_WST % 16 == 0, "alignment");
};

template <int D, int NT, int S>
__global__ void __launch_bounds__(32 * kGmWarps) k_gather_mma(const __grid_constant__ StepParams p) {
  using C = GmCfg<D, NT, S>;
  constexpr int GM = C::GM;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned char* smem = smem_raw;
  const int c = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gr = lane >> 2, tg = lane & 3;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR) + warp * S;
  __nv_bfloat16* P = reinterpret_cast<__nv_bfloat16*>(smem + C::OFF_P) + warp * GM * 32;
  float* zx = reinterpret_cast<float*>(smem + C::OFF_ZX) + warp * S * C::ZX * 32;
  uint32_t* mask_s = reinterpret_cast<uint32_t*>(smem + C::OFF_MASK) + warp * S;
  float (*wst)[GM][2] = reinterpret_cast<float (*)[GM][2]>(smem + C::OFF_WST);
  float (*fin)[4] = reinterpret_cast<float (*)[4]>(smem + C::OFF_FIN);
  int* last = reinterpret_cast<int*>(smem + C::OFF_LAST);
  unsigned char* ring = smem + warp * S * C::SLOT;

  // A slot's phase completes on lane 0's arrival (with the row bytes as its
  // transaction count) once the rows and every lane's logits have landed.
  if (tid < kGmWarps * S) mbar_init(reinterpret_cast<uint64_t*>(smem + C::OFF_BAR) + tid, 1);
  mbar_fence_init();
  __syncthreads();
  const int G = p.G, H = p.H;
  const int64_t hrow0 = (int64_t)b * H + g * G;
  float (*tw)[kNsMax] = reinterpret_cast<float (*)[kNsMax]>(smem + C::OFF_TW);
  float (*tl)[kNsMax] = tw + GM;
  // The sequence's record is a caller input: read it before the wait.
  const Seq sq = load_seq(p, b, false);
  // (b) first: it reads only the score kernel's partials, complete before the
  // select kernel lets this grid start.  Its shared memory is the ring's.
  // After the anchor layer no select kernel runs in between: there (b)
  // waits for the score kernel like everything else.
  if (c < p.nm && !p.anchor) {
    gather_text_slice<D, GM, C::THREADS>(p, c, hrow0, tw, tl);
    fence_proxy_async();
    __syncthreads();
  }
  pdl_wait();
  pdl_trigger();
  if (c < p.nm && p.anchor) {
    gather_text_slice<D, GM, C::THREADS>(p, c, hrow0, tw, tl);
    fence_proxy_async();
    __syncthreads();
  }
  const int64_t pbase = ((int64_t)b * p.Hkv + g) * p.nk_max;
  unsigned err = 0;
  bool timed_out = false;
  // The only CTA of its (sequence, kv-head) combines the text part with its
  // chunk itself: no partial round trip through global memory, no ticket.
  const bool lone = p.nc == 1 && p.nk == 1;

  // (a) kept chunk c
  if (c < p.nk) {
    const int sel = p.granularity ? b * p.Hkv + g : b;
    const int32_t* kept = p.kept_idx + (int64_t)sel * p.kept_cap;
    // Kept-list entry of row `lane` of this warp's tile k for a chunk
    // starting at j, read now (entries past the chunk are read in bounds
    // and masked at use; with no kept capacity the list may be absent and
    // nothing is read).  The copies of tile k are issued S tiles before it
    // is consumed and its entry QD tiles before that: an iteration can take
    // less than a round trip to L2.
    constexpr int QD = 3;
    auto raw_entry = [&](int j, int k) {
      return p.kept_cap > 0 ? ldcg_now(kept + min(j + 32 * (warp + kGmWarps * k) + lane, p.kept_cap - 1)) : -1;
    };
    // The first S + QD tiles' entries are read in the same round trip as the
    // count, at the chunk start a full list would give (exact for chunk 0
    // and whenever the count is the cap); a different start reloads them.
    const int j0s = min(p.kept_cap, c * ((p.kept_cap + p.nk - 1) / p.nk));
    int raw[S + QD];
#pragma unroll
    for (int k = 0; k < S + QD; ++k) raw[k] = raw_entry(j0s, k);
    const int K = max(0, min(__ldcg(p.kept_count + sel), min(sq.nv, p.kept_cap)));
    const int per = (K + p.nk - 1) / p.nk;
    const int j0 = min(K, c * per), j1 = min(K, min(j0 + per, j0 + C::MAX_CHUNK));
    if (per > C::MAX_CHUNK) err |= ERR_KEPT;  // the plan keeps every chunk within the limit
    const int ntile = (j1 - j0 + 31) / 32;
    const int nj = warp < ntile ? (ntile - warp + kGmWarps - 1) / kGmWarps : 0;  // this warp's tiles
    const float* zb = p.z_ws + (int64_t)b * p.max_visual * p.hp + g * G;
    int issued = 0;  // tiles of this warp whose copies were issued

    // Kept index of row `lane` of this warp's tile k from its entry, or -1
    // (past the chunk; an out-of-range index is flagged and skipped).
    auto row_index = [&](int k, int e) {
      const int j = 32 * (warp + kGmWarps * k) + lane;
      int i = -1;
      if (k < nj && j0 + j < j1) {
        i = e;
        if (i < 0 || i >= sq.nv) { err |= ERR_KEPT; i = -1; }
      }
      return i;
    };
    if (j0 != j0s) {  // CTA-uniform
#pragma unroll
      for (int k = 0; k < S + QD; ++k) raw[k] = raw_entry(j0, k);
    }
    auto issue = [&](int k, int i) {  // all lanes; i = this lane's kept index
      if (k >= nj) return;
      const int slot = k % S;
      const __nv_bfloat16* vr = nullptr;
      if (i >= 0) {
        vr = kv_row<__nv_bfloat16>(p.v, p, b, g, sq.vs + i);
        if (!vr) { err |= ERR_PAGE; i = -1; }
      }
      const unsigned m = __ballot_sync(0xffffffffu, vr != nullptr);
      unsigned char* row = ring + slot * C::SLOT + lane * C::RP;
      // The slot was last read by this warp's ldmatrix and loads (generic
      // proxy); its rows are next written by bulk copies (async proxy).
      fence_proxy_async();
      __syncwarp();  // every lane is done reading this slot
      if (lane == 0) mask_s[slot] = m;
      // Logits of this lane's token: heads 0-3 into its row's pad.
      if (vr) {
        const float* zr = zb + (int64_t)i * p.hp;
        for (int h = 0; h < G; ++h)
          cp_async4(h < 4 ? smem_u32(row + 2 * D + 4 * h) : smem_u32(zx + (slot * C::ZX + h - 4) * 32 + lane), zr + h);
      }
      cp_async_arrive_counted(full + slot);
      __syncwarp();  // every lane's arrival is counted before lane 0's
      if (lane == 0) mbar_expect_tx(full + slot, (unsigned)__popc(m) * (2 * D));
      __syncwarp();
      if (vr) bulk_g2s(row, vr, 2 * D, full + slot);
      issued = k + 1;
    };
    // Prologue: the first S tiles; the next QD tiles' entries stay queued.
#pragma unroll
    for (int k = 0; k < S; ++k) issue(k, row_index(k, raw[k]));
    int q[QD];
#pragma unroll
    for (int t = 0; t < QD; ++t) q[t] = raw[S + t];

    // Probabilities are taken relative to each head's largest logit over all
    // tokens (from the select kernel), so no running maximum is needed.
    float mh[GM], lsum[GM];
    float acc[NT][C::MT][4];
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      mh[h] = h < G ? __ldcg(p.hmax + hrow0 + h) : -CUDART_INF_F;
      lsum[h] = 0.f;
    }
#pragma unroll
    for (int nn = 0; nn < NT; ++nn)
#pragma unroll
      for (int mi = 0; mi < C::MT; ++mi)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[nn][mi][e] = 0.f;
    // ldmatrix.trans lane roles for V^T (A operand, rows = dimensions).
    const int vrow = (lane & 7) + 8 * (lane >> 4), vcol = 8 * ((lane >> 3) & 1);

    for (int k = 0; k < nj; ++k) {
      const int slot = k % S;
      if (!mbar_wait(full + slot, (k / S) & 1)) { timed_out = true; break; }
      const uint32_t mask = mask_s[slot];
      const bool live = (mask >> lane) & 1u;
      const float4 z4 = *reinterpret_cast<const float4*>(ring + slot * C::SLOT + lane * C::RP + 2 * D);
      float z[GM];
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        z[h] = -CUDART_INF_F;
        if (live && h < G) {
          if (h < 4) z[h] = h == 0 ? z4.x : h == 1 ? z4.y : h == 2 ? z4.z : z4.w;
          else z[h] = zx[(slot * C::ZX + (h >= 4 ? h - 4 : 0)) * 32 + lane];
        }
      }

      // Probabilities of this tile (the warp's buffer was last read by the
      // previous tile's P.V, before the loop's closing __syncwarp).
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        if (h >= G) continue;
        const float pe = exp2_rel(z[h], mh[h]);
        lsum[h] += pe;
        P[h * 32 + lane] = __float2bfloat16_rn(pe);
      }
      __syncwarp();
      const unsigned vt = smem_u32(ring + slot * C::SLOT);
#pragma unroll
      for (int sb = 0; sb < 2; ++sb) {
        uint32_t pb[NT][2];
#pragma unroll
        for (int nn = 0; nn < NT; ++nn) {
          const __nv_bfloat16* pr = P + (8 * nn + gr) * 32 + 16 * sb + 2 * tg;
          pb[nn][0] = *reinterpret_cast<const uint32_t*>(pr);
          pb[nn][1] = *reinterpret_cast<const uint32_t*>(pr + 8);
        }
        // Rows that were not copied hold stale bytes: zero their words.  (B
        // columns of heads past G hold stale bytes too; those heads' sums
        // are never read.)
        const uint32_t rb = mask >> (16 * sb);
        if ((rb & 0xffffu) == 0xffffu) {  // all 16 rows copied (warp-uniform)
#pragma unroll
          for (int mi = 0; mi < C::MT; ++mi) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4_t(vt + (16 * sb + vrow) * C::RP + (16 * mi + vcol) * 2, a0, a1, a2, a3);
#pragma unroll
            for (int nn = 0; nn < NT; ++nn) mma_bf16(acc[nn][mi], a0, a1, a2, a3, pb[nn][0], pb[nn][1]);
          }
          continue;
        }
        const uint32_t mlo = (((rb >> (2 * tg)) & 1u) ? 0x0000ffffu : 0u) | (((rb >> (2 * tg + 1)) & 1u) ? 0xffff0000u : 0u);
        const uint32_t mhi = (((rb >> (2 * tg + 8)) & 1u) ? 0x0000ffffu : 0u) | (((rb >> (2 * tg + 9)) & 1u) ? 0xffff0000u : 0u);
#pragma unroll
        for (int mi = 0; mi < C::MT; ++mi) {
          uint32_t a0, a1, a2, a3;
          ldsm_x4_t(vt + (16 * sb + vrow) * C::RP + (16 * mi + vcol) * 2, a0, a1, a2, a3);
          a0 &= mlo; a1 &= mlo; a2 &= mhi; a3 &= mhi;
#pragma unroll
          for (int nn = 0; nn < NT; ++nn) mma_bf16(acc[nn][mi], a0, a1, a2, a3, pb[nn][0], pb[nn][1]);
        }
      }
      __syncwarp();
      // Refill this slot with tile k + S; queue the entry of tile k + S + QD.
      const int icur = row_index(k + S, q[0]);
#pragma unroll
      for (int t = 0; t + 1 < QD; ++t) q[t] = q[t + 1];
      q[QD - 1] = raw_entry(j0, k + S + QD);
      issue(k + S, icur);
    }
    // After a timeout, let this warp's copies still in flight land (bounded)
    // before the ring is reused below.
    if (timed_out && lane == 0)
      for (int k = max(0, issued - S); k < issued; ++k) mbar_wait(full + k % S, (k / S) & 1);
    __syncwarp();

    // Warp partials -> chunk partial (log-sum-exp over the warps).
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      const float l = warp_sum(lsum[h]);
      if (lane == 0) { wst[warp][h][0] = mh[h]; wst[warp][h][1] = l; }
    }
    // Lone CTA: request the text output and statistics (the merged slice this
    // CTA wrote in part (b), or the single split partial) before the sums.
    constexpr int D4 = D / 4, IT = (GM * D4 + C::THREADS - 1) / C::THREADS;
    float4 tv[IT];
    float2 ts[IT];
    if (lone) {
      const float* t_o = p.nm ? p.mt_o + hrow0 * D : p.split_o + hrow0 * p.nsp_max * D;
      const int t_ostride = p.nm ? D : p.nsp_max * D;
#pragma unroll
      for (int it = 0; it < IT; ++it) {
        const int i = tid + it * C::THREADS;
        if (i < G * D4) {
          const int h = i / D4, d = 4 * (i % D4);
          tv[it] = __ldcg(reinterpret_cast<const float4*>(t_o + (int64_t)h * t_ostride + d));
          const float* st = p.nm ? p.mt_st + (hrow0 + h) * 2 : p.split_st + (hrow0 + h) * p.nsp_max * ST_N;
          ts[it] = p.nm ? make_float2(__ldcg(st), __ldcg(st + 1)) : make_float2(__ldcg(st + ST_MT), __ldcg(st + ST_L1T));
        }
      }
    }
    __syncthreads();  // every warp is done with its ring
    float* ow = reinterpret_cast<float*>(smem) + warp * GM * D;
#pragma unroll
    for (int nn = 0; nn < NT; ++nn)
#pragma unroll
      for (int mi = 0; mi < C::MT; ++mi) {
        const int h0 = 8 * nn + 2 * tg, d0 = 16 * mi + gr;
        ow[h0 * D + d0] = acc[nn][mi][0];
        ow[(h0 + 1) * D + d0] = acc[nn][mi][1];
        ow[h0 * D + d0 + 8] = acc[nn][mi][2];
        ow[(h0 + 1) * D + d0 + 8] = acc[nn][mi][3];
      }
    __syncthreads();
    if (lone) {
      // Same arithmetic as the combine of gather_finish with one chunk.
#pragma unroll
      for (int it = 0; it < IT; ++it) {
        const int i = tid + it * C::THREADS;
        if (i >= G * D4) continue;
        const int h = i / D4, d = 4 * (i % D4);
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
        float l = 0.f;
#pragma unroll
        for (int w = 0; w < kGmWarps; ++w) {
          const float4 v = *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(smem) + (w * GM + h) * D + d);
          o.x += v.x; o.y += v.y; o.z += v.z; o.w += v.w;
          l += wst[w][h][1];
        }
        const float mk = wst[0][h][0], mt = ts[it].x;
        const float M = fmaxf(mt, mk);
        const float wt = exp2_rel(mt, M), wk = exp2_rel(mk, M);
        const float den = fmaf(wk, l, wt * ts[it].y);
        const float inv = den > 0.f ? 1.f / den : 0.f;
        float4 num = make_float4(wt * tv[it].x, wt * tv[it].y, wt * tv[it].z, wt * tv[it].w);
        num.x = fmaf(wk, o.x, num.x); num.y = fmaf(wk, o.y, num.y); num.z = fmaf(wk, o.z, num.z); num.w = fmaf(wk, o.w, num.w);
        __nv_bfloat16* op = reinterpret_cast<__nv_bfloat16*>(p.out) + (hrow0 + h) * D + d;
        op[0] = from_f<__nv_bfloat16>(num.x * inv); op[1] = from_f<__nv_bfloat16>(num.y * inv);
        op[2] = from_f<__nv_bfloat16>(num.z * inv); op[3] = from_f<__nv_bfloat16>(num.w * inv);
      }
    }
    for (int i = tid; !lone && i < G * D; i += C::THREADS) {
      const int h = i / D, d = i % D;
      float o = 0.f, l = 0.f;
#pragma unroll
      for (int w = 0; w < kGmWarps; ++w) {
        o += reinterpret_cast<const float*>(smem)[(w * GM + h) * D + d];
        l += wst[w][h][1];
      }
      p.gpart_o[((pbase + c) * G + h) * D + d] = o;
      if (d == 0) {
        p.gpart_st[((pbase + c) * G + h) * 2 + 0] = wst[0][h][0];
        p.gpart_st[((pbase + c) * G + h) * 2 + 1] = l;
      }
    }
    __syncthreads();  // the ring is reused below
  }

  if (timed_out) err |= ERR_TIMEOUT;
  if (err) atomicOr(p.err, err);
  if (!lone) gather_finish<__nv_bfloat16, D, GM, C::THREADS>(p, b, g, hrow0, pbase, tw, fin, last);
}

// ---------------------------------------------------------------------------
// k_gather_slice: grid (D / 16, Hkv, B), 256 threads, for kept sets of at most
// kSliceMaxKept tokens per (sequence, kv-head).  CTA c owns output dimensions
// [16c, 16c + 16) of the G heads.  It first merges the same slice of the
// score splits' text partials -- they come from the score kernel, which has
// completed before any select CTA lets this grid start, so this part runs
// before griddepcontrol.wait and overlaps the select kernel.  After the wait
// it attends over every kept visual token (reading only its 16-dimension
// slice of V, fetched in the same round trip as the token's logits) and
// combines both parts in log-sum-exp form.  No partial leaves the CTA.
// ---------------------------------------------------------------------------
constexpr int kSliceDims = 16;

template <int GM>
struct SliceSmem {
  float pz[GM][kSliceMaxKept];            // kept logits, then probabilities
  float tm[GM][kNsMax];                   // text split maxima, then weights
  float tl[GM][kNsMax];                   // text split sums
  float red[kGatherWarps][GM][kSliceDims];  // kept-part warp partials
  float4 tred[kGatherThreads];            // text-part thread partials
  float fin[GM][4];                       // m_k, l_k, M_t, L_t
};

template <typename T, int D, int GM>
__global__ void __launch_bounds__(kGatherThreads) k_gather_slice(const __grid_constant__ StepParams p) {
  constexpr int SD = kSliceDims;
  constexpr int CH = 16 / sizeof(T);      // elements per 16-byte chunk
  constexpr int CPS = SD / CH;            // chunks per row slice (2 bf16, 4 fp32)
  constexpr int TSTRIDE = kGatherThreads / CPS;  // kept tokens handled side by side
  constexpr int TPT = kSliceMaxKept / TSTRIDE;   // kept tokens per thread
  extern __shared__ __align__(16) unsigned char smem_raw[];
  auto& sm = *reinterpret_cast<SliceSmem<GM>*>(smem_raw);
  const int cd = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.G, H = p.H, ns = p.ns;
  const int64_t hrow0 = (int64_t)b * H + g * G;
  const Seq sq = load_seq(p, b, false);

  // 1. Text split statistics, then per head: text max, split weights, sum.
  for (int i = tid; i < G * ns; i += kGatherThreads) {
    const int h = i / ns, s = i % ns;
    const float2 r = __ldcg(reinterpret_cast<const float2*>(p.split_st + ((hrow0 + h) * p.nsp_max + s) * ST_N));
    sm.tm[h][s] = r.x;  // ST_MT
    sm.tl[h][s] = r.y;  // ST_L1T
  }
  __syncthreads();
  for (int h = warp; h < G; h += kGatherWarps) {
    float mt = -CUDART_INF_F;
    for (int s = lane; s < ns; s += 32) mt = fmaxf(mt, sm.tm[h][s]);
    mt = warp_max(mt);
    float lt = 0.f;
    for (int s = lane; s < ns; s += 32) {
      const float w = exp2_rel(sm.tm[h][s], mt);
      sm.tm[h][s] = w;
      lt = fmaf(w, sm.tl[h][s], lt);
    }
    lt = warp_sum(lt);
    if (lane == 0) { sm.fin[h][2] = mt; sm.fin[h][3] = lt; }
  }
  __syncthreads();
  // 2. Text partials of the slice: thread (element e = (head, float4), split group sg).
  {
    const int NE = G * (SD / 4);
    const int nsg = kGatherThreads / NE;
    const int e = tid % NE, sg = tid / NE;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (sg < nsg) {
      const int h = e / (SD / 4), d = cd * SD + 4 * (e % (SD / 4));
      const float* so = p.split_o + (hrow0 + h) * p.nsp_max * D + d;
#pragma unroll 4
      for (int s = sg; s < ns; s += nsg) {
        const float4 v = __ldcg(reinterpret_cast<const float4*>(so + (int64_t)s * D));
        const float w = sm.tm[h][s];
        acc.x = fmaf(w, v.x, acc.x); acc.y = fmaf(w, v.y, acc.y); acc.z = fmaf(w, v.z, acc.z); acc.w = fmaf(w, v.w, acc.w);
      }
    }
    sm.tred[tid] = acc;
  }

  pdl_wait();
  pdl_trigger();
  const int sel = p.granularity ? b * p.Hkv + g : b;
  const int K = max(0, min(__ldcg(p.kept_count + sel), min(sq.nv, min(p.kept_cap, kSliceMaxKept))));
  const int32_t* kept = p.kept_idx + (int64_t)sel * p.kept_cap;
  unsigned err = 0;

  // 3. Kept tokens: thread (token slot j0, chunk q) takes tokens j0 + TSTRIDE t;
  //    their V slices and (chunk 0) their logits are fetched together.
  const int j0 = tid / CPS, q = tid % CPS;
  int idx[TPT];
#pragma unroll
  for (int t = 0; t < TPT; ++t) {
    const int j = j0 + TSTRIDE * t;
    idx[t] = j < K ? __ldcg(kept + j) : -1;
    if (j < K && (idx[t] < 0 || idx[t] >= sq.nv)) { err |= ERR_KEPT; idx[t] = -1; }
  }
  float vv[TPT][CH];
#pragma unroll
  for (int t = 0; t < TPT; ++t) {
#pragma unroll
    for (int e = 0; e < CH; ++e) vv[t][e] = 0.f;
    if (idx[t] >= 0) {
      const T* vr = kv_row<T>(p.v, p, b, g, sq.vs + idx[t]);
      if (vr) load_f<CH>(vr + cd * SD + q * CH, vv[t]);
      else err |= ERR_PAGE;
    }
  }
  if (q == 0) {
#pragma unroll
    for (int t = 0; t < TPT; ++t) {
      const int j = j0 + TSTRIDE * t;
      if (j >= K) break;
      const float* zr = p.z_ws + ((int64_t)b * p.max_visual + (idx[t] < 0 ? 0 : idx[t])) * p.hp + g * G;
      float zv[GM];
#pragma unroll
      for (int h = 0; h < GM; ++h) zv[h] = (idx[t] >= 0 && h < G) ? __ldcg(zr + h) : -CUDART_INF_F;
#pragma unroll
      for (int h = 0; h < GM; ++h) sm.pz[h][j] = zv[h];
    }
  }
  __syncthreads();
  // 4. Per head: kept max, probabilities, sum.
  for (int h = warp; h < G; h += kGatherWarps) {
    float m = -CUDART_INF_F;
    for (int t = lane; t < K; t += 32) m = fmaxf(m, sm.pz[h][t]);
    m = warp_max(m);
    float l = 0.f;
    for (int t = lane; t < K; t += 32) {
      const float e = exp2_rel(sm.pz[h][t], m);
      sm.pz[h][t] = e;
      l += e;
    }
    l = warp_sum(l);
    if (lane == 0) { sm.fin[h][0] = m; sm.fin[h][1] = l; }
  }
  __syncthreads();
  // 5. P.V over the kept tokens from registers, reduced over the warp's token lanes.
  {
    float ko[GM][CH];
#pragma unroll
    for (int h = 0; h < GM; ++h)
#pragma unroll
      for (int e = 0; e < CH; ++e) ko[h][e] = 0.f;
#pragma unroll
    for (int t = 0; t < TPT; ++t) {
      const int j = j0 + TSTRIDE * t;
      if (j >= K) break;
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        if (h >= G) break;
        const float pr = sm.pz[h][j];
#pragma unroll
        for (int e = 0; e < CH; ++e) ko[h][e] = fmaf(pr, vv[t][e], ko[h][e]);
      }
    }
#pragma unroll
    for (int o = CPS; o < 32; o <<= 1)
#pragma unroll
      for (int h = 0; h < GM; ++h)
#pragma unroll
        for (int e = 0; e < CH; ++e) ko[h][e] += __shfl_xor_sync(0xffffffffu, ko[h][e], o);
    if (lane < CPS) {
#pragma unroll
      for (int h = 0; h < GM; ++h)
#pragma unroll
        for (int e = 0; e < CH; ++e) sm.red[warp][h][lane * CH + e] = ko[h][e];
    }
  }
  if (err) atomicOr(p.err, err);
  __syncthreads();

  // 6. Combine (thread per (head, dimension) of the slice).
  if (tid < G * SD) {
    const int h = tid / SD, d = tid % SD;
    float kv = 0.f;
#pragma unroll
    for (int w = 0; w < kGatherWarps; ++w) kv += sm.red[w][h][d];
    const int NE = G * (SD / 4), nsg = kGatherThreads / NE;
    const int e = h * (SD / 4) + d / 4;
    float tv = 0.f;
    for (int sg = 0; sg < nsg; ++sg) {
      const float4 v = sm.tred[sg * NE + e];
      tv += (d & 3) == 0 ? v.x : (d & 3) == 1 ? v.y : (d & 3) == 2 ? v.z : v.w;
    }
    const float mk = sm.fin[h][0], lk = sm.fin[h][1], mt = sm.fin[h][2], lt = sm.fin[h][3];
    const float M = fmaxf(mk, mt);
    const float ak = exp2_rel(mk, M), at = exp2_rel(mt, M);
    const float den = ak * lk + at * lt;
    const float o = den > 0.f ? (ak * kv + at * tv) / den : 0.f;
    reinterpret_cast<T*>(p.out)[(hrow0 + h) * D + cd * SD + d] = from_f<T>(o);
  }
}

// ---------------------------------------------------------------------------
// k_selgat: the select kernel and the slice gather in one launch, for the
// calls the slice gather serves (few sequences, kept sets of at most
// kSliceMaxKept rows, at most 8 query heads per kv-head, a budget known in
// advance).  Grid (cl, nsel, B) in clusters of cl CTAs of 512 threads, one
// cluster per selection unit (a sequence, or a (sequence, kv-head) when
// granularity = 1); CTA r of the cluster owns the output dimensions
// [d0, d0 + W) of one kv-head g.
//   1. Every CTA merges the split statistics of every head into M_h, L1_h
//      and the masses (Eq. 5, Eq. 6); rank 0 also takes the head mean, the
//      head max (Sec. 4.3) and the budget K_t (Eq. 7 + clamp).
//   2. Every CTA requests the text partials of the score splits for its
//      dimensions, scores its slice of the visual tokens (S_i of Eq. 2) into
//      rank 0's shared memory meanwhile, then sums the text part.
//   3. Rank 0 cuts the Top-K_t set (Eq. 3) by a radix select over the keys
//      held in registers and compacts it, ascending, into the output and its
//      shared memory; the other CTAs copy it over distributed shared memory.
//   4. Every CTA stages the V slices and logits of the kept tokens in shared
//      memory in one round trip, attends over them for its dimensions (P.V on
//      the tensor cores for bf16 caches) and combines the result with the
//      text part in log-sum-exp form.  Nothing but the results leaves the
//      cluster; one launch and one dependency replace two, and only the
//      selection itself lies between the score kernel and the kept rows'
//      loads.
// ---------------------------------------------------------------------------
constexpr int kSgThreads = 512;
constexpr int kSgWarps = kSgThreads / 32;
constexpr int kSgMaxW = 128;  // output dimensions of one CTA, at most (64 with fp32 caches)

// Register-resident Top-K cut of the fused kernel (Eq. 3) over n <= 8 * NTH
// score keys: thread t holds keys [8t, 8t + 8), valid while below n.  Keys
// are float bits of scores in [0, 1] (clamped below 2^30 by the producer), so
// the digits skip the two top bits: passes on bits 29-22, 21-14, 13-6, 5-0.
// The first digits of the scores concentrate in few buckets, so every warp
// counts into its own histogram (hist: two sets of NTH / 32 histograms of 256
// bins in shared memory, alternating between passes; each warp clears its
// own histogram of a set before counting into it); thread d < 256 then adds
// up digit d over the warps into tot, and lane L of every warp owns digits
// 255-8L ... 248-8L of the sums.
constexpr int kCutKeys = 8;
template <int NTH>
__device__ __forceinline__ RadixCut radix_cut_regs(const uint32_t (&k)[kCutKeys], int nvalid, int K, unsigned* hist,
                                                   unsigned* tot) {
  constexpr int NW = NTH / 32;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  unsigned krem = (unsigned)K, n_theta = 0;
  bool whole = false;
  uint32_t prefix = 0, mask = 0;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = pass < 3 ? 22 - 8 * pass : 0;
    const uint32_t dmask = pass < 3 ? 255u : 63u;
    unsigned* h = hist + ((pass & 1) * NW + warp) * 256;
    // This warp's histogram of the set: last read before the previous pass's
    // second barrier, so it may be cleared now.
    reinterpret_cast<uint4*>(h)[2 * lane] = make_uint4(0u, 0u, 0u, 0u);
    reinterpret_cast<uint4*>(h)[2 * lane + 1] = make_uint4(0u, 0u, 0u, 0u);
    __syncwarp();
#pragma unroll
    for (int j = 0; j < kCutKeys; ++j)
      if (j < nvalid && (k[j] & mask) == prefix) atomicAdd(&h[(k[j] >> shift) & dmask], 1u);
    __syncthreads();
    if (tid < 256) {
      unsigned c = 0;
#pragma unroll
      for (int w = 0; w < NW; ++w) c += hist[((pass & 1) * NW + w) * 256 + tid];
      tot[tid] = c;
    }
    __syncthreads();
    unsigned cnt8[8], sum8 = 0;
    {
      const uint4* tp = reinterpret_cast<const uint4*>(tot + 248 - 8 * lane);
      const uint4 lo = tp[0], hi = tp[1];  // digits 248-8L .. 251-8L, 252-8L .. 255-8L
      cnt8[0] = hi.w; cnt8[1] = hi.z; cnt8[2] = hi.y; cnt8[3] = hi.x;
      cnt8[4] = lo.w; cnt8[5] = lo.z; cnt8[6] = lo.y; cnt8[7] = lo.x;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) sum8 += cnt8[j];
    unsigned incl = sum8;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned nn = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += nn;
    }
    const unsigned excl = incl - sum8;
    const bool mine = excl < krem && krem <= incl;
    unsigned dsel = 0, before = 0, cnt = 0;
    if (mine) {
      unsigned run = excl;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (run + cnt8[j] >= krem) { dsel = 255 - 8 * lane - j; before = run; cnt = cnt8[j]; break; }
        run += cnt8[j];
      }
    }
    const int src = max(__ffs(__ballot_sync(0xffffffffu, mine)) - 1, 0);
    dsel = __shfl_sync(0xffffffffu, dsel, src);
    before = __shfl_sync(0xffffffffu, before, src);
    cnt = __shfl_sync(0xffffffffu, cnt, src);
    krem -= before;
    prefix |= dsel << shift;
    mask |= dmask << shift;
    if (pass == 3) n_theta = cnt;
    if (pass < 3 && krem == cnt) {  // the whole bucket is kept
      whole = true;
      break;
    }
  }
  return RadixCut{whole ? prefix - 1u : prefix, krem, n_theta, whole};
}

// Exclusive prefix sum over the block with one barrier: wsum_s[NTH / 32]
// must not be written again before the next barrier.
template <int NTH>
__device__ __forceinline__ int block_excl_scan_1b(int x, int* wsum_s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  if (lane == 31) wsum_s[warp] = incl;
  __syncthreads();
  int before = 0;
  for (int w = 0; w < warp; ++w) before += wsum_s[w];
  return before + incl - x;
}

// Ascending compaction of the register-resident keys (see radix_cut_regs):
// keys above c.theta plus the first c.krem keys equal to it (every key when
// take_all), written to kept (global) and, with TO_SMEM, to kept_s (shared
// memory).  wsum_s holds 2 * NTH / 32 ints.
template <int NTH, bool TO_SMEM>
__device__ __forceinline__ void compact_kept_regs(const uint32_t (&k)[kCutKeys], int nvalid, int K, bool take_all,
                                                  const RadixCut& c, int* wsum_s, int32_t* kept, int* kept_s) {
  const int i0 = kCutKeys * (int)threadIdx.x;
  const bool ties = !take_all && !c.whole && c.krem < c.n_theta;
  int n_eq = 0;
  if (ties)
#pragma unroll
    for (int j = 0; j < kCutKeys; ++j) n_eq += j < nvalid && k[j] == c.theta;
  const int eq_before = ties ? block_excl_scan_1b<NTH>(n_eq, wsum_s + NTH / 32) : 0;
  const unsigned krem = ties ? c.krem : 0xffffffffu;
  unsigned selm = 0;
  {
    int r = eq_before;
#pragma unroll
    for (int j = 0; j < kCutKeys; ++j) {
      const bool v = j < nvalid;
      const bool sel = v && (take_all || k[j] > c.theta || (!c.whole && k[j] == c.theta && (unsigned)r < krem));
      r += v && k[j] == c.theta;
      selm |= (unsigned)sel << j;
    }
  }
  int o = block_excl_scan_1b<NTH>(__popc(selm), wsum_s);
#pragma unroll
  for (int j = 0; j < kCutKeys; ++j)
    if (((selm >> j) & 1u) && o < K) {
      kept[o] = i0 + j;
      if constexpr (TO_SMEM) kept_s[o] = i0 + j;
      ++o;
    }
}

constexpr int kSgKP = kSliceMaxKept + 1;  // float row pitch of the kept logits (rows in distinct banks)
constexpr int kSgPB = kSliceMaxKept + 8;  // bf16 row pitch of the kept probabilities (likewise)

template <int GM>
struct SgSmem {
  float hM[kMaxHeads], hInv[kMaxHeads], hMass[kMaxHeads], hMass1[kMaxHeads];
  float hMt[GM], hLt[GM];        // text-only max and sum of this CTA's heads
  alignas(16) unsigned tot[256];  // radix: digit counts summed over the warps
  int wsum[32];
  int K;                         // the budget K_t (rank 0; the others copy it)
  int kept[kSliceMaxKept];       // the kept list (rank 0; the others copy it)
  float pz[GM][kSgKP];           // kept logits, then (fp32 caches) probabilities
  __nv_bfloat16 pb[8][kSgPB];    // bf16 caches: probabilities, B operand of the tensor-core P.V
  float red[kSgWarps][128];      // P.V partials of every warp
  float4 to[GM * kSgMaxW / 4];   // text part of the output
  float fin[GM][2];              // kept max, kept sum
};

constexpr int kSgTextSplits = 10;  // text split partials a thread requests ahead

// Byte offset of 16-byte piece c of row j in a stage of 128-byte rows, the
// pieces XOR-swizzled by the row so that ldmatrix reads hit distinct banks.
__device__ __forceinline__ unsigned sg_swz(int j, int c) { return (unsigned)(j * 128 + ((c ^ (j & 7)) << 4)); }
// 16-byte piece c of kept row j of a bf16 V stage: rows of up to 64
// dimensions (128 bytes, swizzled) per half, the second 64 dimensions of a
// row in a second half of kSliceMaxKept rows.
__device__ __forceinline__ unsigned sg_voff(int j, int c) {
  return (unsigned)((c >> 3) * (kSliceMaxKept * 128)) + sg_swz(j, c & 7);
}

// GATHER = false: the selection alone (steps 1, 2b and 3), for calls whose
// gather runs as its own kernel; it also writes every head's largest logit
// (p.hmax) for that kernel.
template <typename T, int D, int GM, bool GATHER = true>
__global__ void __launch_bounds__(kSgThreads) k_selgat(const __grid_constant__ StepParams p) {
  constexpr int NTH = kSgThreads, NW = kSgWarps;
  constexpr bool BF = sizeof(T) == 2;
  // Dynamic: the N_v score keys (rank 0's copy is used); after the cut, the
  // kept rows' V slices.
  extern __shared__ __align__(16) uint32_t key_s[];
  __shared__ SgSmem<GM> sm;

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank(), ncl = (int)cluster.num_blocks();
  const int gsel = blockIdx.y, b = blockIdx.z, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const Seq sq = load_seq(p, b, false);  // an input: read before the wait
  const int G = p.G, H = p.H, ns = p.ns, nv = sq.nv;
  // This CTA's output: kv-head g, dimensions [d0, d0 + W) (the plan makes
  // the cluster split every kv-head evenly, W a multiple of 16).
  const int rpg = !GATHER ? 1 : p.granularity ? ncl : ncl / p.Hkv;
  const int W = GATHER ? D / rpg : 16;
  const int g = !GATHER ? 0 : p.granularity ? gsel : rank / rpg;
  const int d0 = GATHER ? (rank % rpg) * W : 0;
  const int64_t hrow0 = (int64_t)b * H + g * G;
  const int nsel = p.granularity ? p.Hkv : 1;
  // Fused: the next kernel is the next call's score kernel, which reads only
  // its inputs before its own wait, so it may start now.  Select only: the
  // gather kernel reads the score partials before its wait, which this
  // kernel's wait guarantees complete.
  if constexpr (GATHER) pdl_trigger();
  pdl_wait();
  if constexpr (!GATHER) pdl_trigger();
  const float inv_tau = p.inv_tau;

  // 1. Split statistics -> per-head max, normalisers and masses (Eq. 5,
  //    Eq. 6), and for this CTA's heads the text-only max and sum.  Sixteen
  //    lanes per head (two heads per warp); lane l16 folds splits l16,
  //    l16 + 16, ..., four records requested at a time (one round trip for
  //    up to 64 splits).  The first round's records are requested before
  //    anything else: they are on the critical path.
  const float* stb = p.split_st + (int64_t)b * H * p.nsp_max * ST_N;
  const int sub = lane >> 4, l16 = lane & 15;
  auto fetch4 = [&](int h, int s0, float4 (&x)[4], float4 (&y)[4]) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int s = s0 + 16 * k;
      if (h < H && s < ns) {
        const float4* r = reinterpret_cast<const float4*>(stb + ((int64_t)h * p.nsp_max + s) * ST_N);
        x[k] = __ldcg(r);
        y[k] = __ldcg(r + 1);
      } else {
        x[k] = y[k] = make_float4(-CUDART_INF_F, 0.f, 0.f, 0.f);
      }
    }
  };
  float4 rx[4], ry[4];
  fetch4(2 * warp + sub, l16, rx, ry);

  // This CTA's slice of the visual tokens; each thread's first logit row is
  // requested next so that it arrives while the statistics are merged.
  const int per = (nv + ncl - 1) / ncl;
  const int i0 = min(nv, rank * per), i1 = min(nv, i0 + per);
  const int hbeg = p.granularity ? gsel * G : 0;
  const int hcnt = p.granularity ? G : H;
  const bool vec = (hbeg & 3) == 0 && (hcnt & 3) == 0;
  const bool pre = vec && hcnt <= 32 && i0 + tid < i1;
  float4 zpre[8];
  if (pre) {
    const float4* zr = reinterpret_cast<const float4*>(p.z_ws + ((int64_t)b * p.max_visual + i0 + tid) * p.hp + hbeg);
#pragma unroll
    for (int q = 0; q < 8; ++q) zpre[q] = 4 * q < hcnt ? __ldcg(zr + q) : make_float4(0.f, 0.f, 0.f, 0.f);
  }

  for (int h0 = 2 * warp; h0 < H; h0 += 2 * NW) {
    const int h = h0 + sub;
    if (h0 != 2 * warp) fetch4(h, l16, rx, ry);  // the first round's records are in flight already
    float m = -CUDART_INF_F, a1v = 0.f, atv = 0.f, a1t = 0.f, att = 0.f;
    float mt = -CUDART_INF_F, lt = 0.f;  // text only
    for (int s0 = l16;; s0 += 64) {
      if (s0 != l16) fetch4(h, s0, rx, ry);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float mn = fmaxf(m, fmaxf(rx[k].x, ry[k].x));
        if (mn > m) {
          const float f1 = exp2_rel(m, mn), ft = exp2_tau(m, mn, inv_tau);
          a1v *= f1; a1t *= f1; atv *= ft; att *= ft;
          m = mn;
        }
        a1v = fmaf(exp2_rel(ry[k].x, m), ry[k].y, a1v);
        atv = fmaf(exp2_tau(ry[k].x, m, inv_tau), ry[k].z, atv);
        a1t = fmaf(exp2_rel(rx[k].x, m), rx[k].y, a1t);
        att = fmaf(exp2_tau(rx[k].x, m, inv_tau), rx[k].z, att);
        if (rx[k].x > mt) { lt *= exp2_rel(mt, rx[k].x); mt = rx[k].x; }
        lt = fmaf(exp2_rel(rx[k].x, mt), rx[k].y, lt);
      }
      if (s0 + 64 >= ns) break;
    }
    float M = m, Mt = mt;
#pragma unroll
    for (int o = 1; o < 16; o <<= 1) {
      M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      Mt = fmaxf(Mt, __shfl_xor_sync(0xffffffffu, Mt, o));
    }
    const float f1 = exp2_rel(m, M), ft = exp2_tau(m, M, inv_tau), fl = exp2_rel(mt, Mt);
    float L1v = a1v * f1, Ltv = atv * ft, L1t = a1t * f1, Ltt = att * ft, Lt = lt * fl;
#pragma unroll
    for (int o = 1; o < 16; o <<= 1) {
      L1v += __shfl_xor_sync(0xffffffffu, L1v, o);
      Ltv += __shfl_xor_sync(0xffffffffu, Ltv, o);
      L1t += __shfl_xor_sync(0xffffffffu, L1t, o);
      Ltt += __shfl_xor_sync(0xffffffffu, Ltt, o);
      Lt += __shfl_xor_sync(0xffffffffu, Lt, o);
    }
    if (l16 == 0 && h < H) {
      const float L1 = L1v + L1t, Lta = Ltv + Ltt;
      sm.hM[h] = M;
      sm.hInv[h] = L1 > 0.f ? 1.f / L1 : 0.f;
      sm.hMass[h] = Lta > 0.f ? Ltv / Lta : 0.f;
      sm.hMass1[h] = L1 > 0.f ? L1v / L1 : 0.f;
      if (GATHER && h >= g * G && h < g * G + G) { sm.hMt[h - g * G] = Mt; sm.hLt[h - g * G] = Lt; }
    }
  }
  __syncthreads();

  // 2a. Text partials of the score splits for this CTA's dimensions, requested
  //     now and summed after the importance pass: thread (element
  //     e = (head, 4 dimensions), split group sg of four) takes splits
  //     sg, sg + 4, ...
  // Four threads per element when NE <= 128, else two (NE <= 256).
  const int W4 = W / 4, NE = G * W4;
  const int TSH = NE > NTH / 4 ? 1 : 2, TSG = 1 << TSH;
  const int te = tid >> TSH, tsg = tid & (TSG - 1);
  const bool tlive = te < NE;
  const int th = tlive ? te / W4 : 0, tdim = d0 + 4 * (tlive ? te % W4 : 0);
  const float* tst = p.split_st + (hrow0 + th) * p.nsp_max * ST_N + ST_MT;
  const float* tso = p.split_o + (hrow0 + th) * p.nsp_max * D + tdim;
  float tmx[kSgTextSplits];
  float4 tov[kSgTextSplits];
  if constexpr (GATHER) {
#pragma unroll
    for (int k = 0; k < kSgTextSplits; ++k) {
      const int s = tsg + TSG * k;
      const bool ok = tlive && s < ns;
      tmx[k] = ok ? __ldcg(tst + (int64_t)s * ST_N) : -CUDART_INF_F;
      tov[k] = ok ? __ldcg(reinterpret_cast<const float4*>(tso + (int64_t)s * D)) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }

  // Rank 0: head mean, head max (Sec. 4.3) and the budget (Eq. 7), on the
  // last warp (whose importance rows come last).
  if (rank == 0) {
    if (warp == NW - 1) {
      float smn = 0.f, mx = 0.f, s1 = 0.f;
      for (int h = lane; h < H; h += 32) {
        smn += sm.hMass[h];
        mx = fmaxf(mx, sm.hMass[h]);
        s1 += sm.hMass1[h];
      }
      smn = warp_sum(smn);
      mx = warp_max(mx);
      s1 = warp_sum(s1);
      if (lane == 0) {
        const int K = min(budget_k(p, mx, nv), GATHER ? min(p.kept_cap, kSliceMaxKept) : p.kept_cap);
        sm.K = K;
        p.kept_count[(int64_t)b * nsel + gsel] = K;
        if (gsel == 0 && p.mass_stats) {
          float* ms = p.mass_stats + (int64_t)b * 4;
          ms[0] = smn / H; ms[1] = mx; ms[2] = s1 / H; ms[3] = (float)K;
        }
      }
    } else if (gsel == 0) {
      for (int h = tid; h < H; h += NTH - 32) {
        p.mass[(int64_t)b * H + h] = sm.hMass[h];
        if constexpr (!GATHER) p.hmax[(int64_t)b * H + h] = sm.hM[h];
      }
    }
  }

  // 2b. Importance S_i (Eq. 2) of this CTA's slice, as float bits (S >= 0
  //     orders like its bits), into rank 0's key array.
  const float inv_cnt = 1.f / (float)hcnt;
  uint32_t* key0 = ncl > 1 ? cluster.map_shared_rank(key_s, 0) : key_s;
  unsigned bad = 0;
  for (int i = i0 + tid; i < i1; i += NTH) {
    const float* zr = p.z_ws + ((int64_t)b * p.max_visual + i) * p.hp + hbeg;
    float a = 0.f;
    if (pre && i == i0 + tid) {
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (4 * q < hcnt) {
          const int h = hbeg + 4 * q;
          a = fmaf(fexp2_rel(zpre[q].x, sm.hM[h]), sm.hInv[h], a);
          a = fmaf(fexp2_rel(zpre[q].y, sm.hM[h + 1]), sm.hInv[h + 1], a);
          a = fmaf(fexp2_rel(zpre[q].z, sm.hM[h + 2]), sm.hInv[h + 2], a);
          a = fmaf(fexp2_rel(zpre[q].w, sm.hM[h + 3]), sm.hInv[h + 3], a);
        }
      }
    } else if (vec) {
      for (int hh = 0; hh < hcnt; hh += 4) {
        const float4 z4 = __ldcg(reinterpret_cast<const float4*>(zr + hh));
        const int h = hbeg + hh;
        a = fmaf(fexp2_rel(z4.x, sm.hM[h]), sm.hInv[h], a);
        a = fmaf(fexp2_rel(z4.y, sm.hM[h + 1]), sm.hInv[h + 1], a);
        a = fmaf(fexp2_rel(z4.z, sm.hM[h + 2]), sm.hInv[h + 2], a);
        a = fmaf(fexp2_rel(z4.w, sm.hM[h + 3]), sm.hInv[h + 3], a);
      }
    } else {
      for (int hh = 0; hh < hcnt; ++hh)
        a = fmaf(fexp2_rel(__ldcg(zr + hh), sm.hM[hbeg + hh]), sm.hInv[hbeg + hh], a);
    }
    const float sc = a * inv_cnt;
    if (!isfinite(sc)) bad = 1;
    key0[i] = min(__float_as_uint(sc), 0x3fffffffu);  // scores lie in [0, 1]: the top two bits are zero
  }
  if (bad) atomicOr(p.err, ERR_NONFINITE);

  // 2c. The text part: sum exp2(m_s - m_text) * o_s over the splits, then over
  //     the element's four split groups.
  if constexpr (GATHER) {
    const float tmh = sm.hMt[th];
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < kSgTextSplits; ++k) {
      const float w = exp2_rel(tmx[k], tmh);
      a.x = fmaf(w, tov[k].x, a.x); a.y = fmaf(w, tov[k].y, a.y); a.z = fmaf(w, tov[k].z, a.z); a.w = fmaf(w, tov[k].w, a.w);
    }
    for (int s = tsg + TSG * kSgTextSplits; tlive && s < ns; s += TSG) {
      const float w = exp2_rel(__ldcg(tst + (int64_t)s * ST_N), tmh);
      const float4 v = __ldcg(reinterpret_cast<const float4*>(tso + (int64_t)s * D));
      a.x = fmaf(w, v.x, a.x); a.y = fmaf(w, v.y, a.y); a.z = fmaf(w, v.z, a.z); a.w = fmaf(w, v.w, a.w);
    }
    for (int o = 1; o < TSG; o <<= 1) {
      a.x += __shfl_xor_sync(0xffffffffu, a.x, o);
      a.y += __shfl_xor_sync(0xffffffffu, a.y, o);
      a.z += __shfl_xor_sync(0xffffffffu, a.z, o);
      a.w += __shfl_xor_sync(0xffffffffu, a.w, o);
    }
    if (tlive && tsg == 0) sm.to[te] = a;
  }
  if (ncl > 1) cluster.sync();  // rank 0 now sees every key
  else __syncthreads();
  if (!GATHER && rank != 0) return;  // nothing reads this CTA's shared memory any more

  // 3. Rank 0: the Top-K_t cut (Eq. 3) and the ascending compaction, with
  //    every thread's eight keys in registers, into the output and into its
  //    shared memory.
  if (rank == 0) {
    const int K = sm.K;
    int32_t* kept = p.kept_idx + ((int64_t)b * nsel + gsel) * p.kept_cap;
    const bool take_all = K >= nv;
    const int nvalid = min(max(nv - kCutKeys * tid, 0), kCutKeys);
    uint32_t kr[kCutKeys];
    {
      const uint4* kp = reinterpret_cast<const uint4*>(key_s + kCutKeys * tid);
      const uint4 a = nvalid > 0 ? kp[0] : make_uint4(0u, 0u, 0u, 0u);
      const uint4 c = nvalid > 4 ? kp[1] : make_uint4(0u, 0u, 0u, 0u);
      kr[0] = a.x; kr[1] = a.y; kr[2] = a.z; kr[3] = a.w; kr[4] = c.x; kr[5] = c.y; kr[6] = c.z; kr[7] = c.w;
    }
    RadixCut cut{0u, (unsigned)K, 0u, false};
    __syncthreads();  // every key is in registers: the key array holds the warps' histograms from here on
    if (K > 0 && !take_all) cut = radix_cut_regs<NTH>(kr, nvalid, K, key_s, sm.tot);
    if (K > 0) compact_kept_regs<NTH, GATHER>(kr, nvalid, K, take_all, cut, sm.wsum, kept, sm.kept);
    for (int i = max(K, 0) + tid; i < p.kept_cap; i += NTH) kept[i] = -1;
  }
  if constexpr (!GATHER) return;
  if (ncl > 1) cluster.sync();  // rank 0 holds the kept list
  else __syncthreads();
  // Every CTA copies the budget and the kept list from rank 0, then lets
  // rank 0 go: its shared memory may be released once every CTA of the
  // cluster has arrived (the matching wait is the kernel's last instruction).
  int K;
  if (ncl > 1) {
    K = *cluster.map_shared_rank(&sm.K, 0);
    if (rank != 0 && tid < K) sm.kept[tid] = cluster.map_shared_rank(&sm.kept[0], 0)[tid];
    asm volatile("barrier.cluster.arrive.release;\n" ::: "memory");
    __syncthreads();
  } else {
    K = sm.K;
  }

  // 4. Kept rows: their logits and this CTA's V slices to shared memory
  //    (asynchronous copies; V in 16-byte pieces, bf16 rows of 128 bytes with
  //    swizzled pieces, fp32 rows packed), all requested together.  Rows past
  //    K, and rows whose index or page is bad, are zero.
  unsigned char* vst = reinterpret_cast<unsigned char*>(key_s);  // the keys are no longer read
  const int CPR = W * (int)sizeof(T) / 16;                       // 16-byte pieces of a row slice
  const int K16 = (K + 15) & ~15;
  unsigned err = 0;
  // Logits first (the older copy group: the softmax waits for it alone).
  for (int i = tid; i < K * G; i += NTH) {
    const int j = i / G, h = i % G;
    const int id = sm.kept[j];
    if (id >= 0 && id < nv) cp_async4(smem_u32(&sm.pz[h][j]), p.z_ws + ((int64_t)b * p.max_visual + id) * p.hp + g * G + h);
    else sm.pz[h][j] = -CUDART_INF_F;
  }
  asm volatile("cp.async.commit_group;\n" ::: "memory");
  for (int i = tid; i < (BF ? K16 : K) * CPR; i += NTH) {
    const int j = i / CPR, c = i % CPR;
    const unsigned off = BF ? sg_voff(j, c) : (unsigned)((j * CPR + c) * 16);
    const T* vr = nullptr;
    if (j < K) {
      const int id = sm.kept[j];
      if (id >= 0 && id < nv) {
        vr = kv_row<T>(p.v, p, b, g, sq.vs + id);
        if (!vr) err |= ERR_PAGE;
      } else {
        err |= ERR_KEPT;
      }
    }
    if (vr) cp_async16(smem_u32(vst + off), reinterpret_cast<const char*>(vr + d0) + 16 * c);
    else *reinterpret_cast<uint4*>(vst + off) = make_uint4(0u, 0u, 0u, 0u);
  }
  asm volatile("cp.async.commit_group;\n" ::: "memory");
  asm volatile("cp.async.wait_group 1;\n" ::: "memory");
  __syncthreads();
  // Per head: kept max, probabilities, sum.  bf16 caches: the probabilities
  // as bf16 (the tensor-core operand), zero past K and for heads past G.
  for (int h = warp; h < (BF ? 8 : G); h += NW) {
    if (h >= G) {
      for (int t = lane; t < K16; t += 32) sm.pb[h][t] = __float2bfloat16_rn(0.f);
      continue;
    }
    float m = -CUDART_INF_F;
    for (int t = lane; t < K; t += 32) m = fmaxf(m, sm.pz[h][t]);
    m = warp_max(m);
    float l = 0.f;
    for (int t = lane; t < (BF ? K16 : K); t += 32) {
      const float e = t < K ? exp2_rel(sm.pz[h][t], m) : 0.f;
      if constexpr (BF) sm.pb[h][t] = __float2bfloat16_rn(e);
      else sm.pz[h][t] = e;
      l += e;
    }
    l = warp_sum(l);
    if (lane == 0) { sm.fin[h][0] = m; sm.fin[h][1] = l; }
  }
  asm volatile("cp.async.wait_group 0;\n" ::: "memory");  // the V rows
  __syncthreads();

  // P.V.  bf16: on the tensor cores, mma m16n8k16 with A = V^T (16
  // dimensions x 16 kept rows, ldmatrix.trans from the stage) and B = P^T
  // (16 kept rows x 8 heads); warp w owns the 16-dimension tile w % (W / 16)
  // over every (16 / (W / 16))-th step of 16 kept rows.  fp32: thread (part,
  // head, dimension) sums every parts-th kept row on the CUDA cores.
  const int nmt = W / 16;
  if constexpr (BF) {
    const int mt = warp % nmt, kg = warp / nmt, ngr = NW / nmt;
    const int gr = lane >> 2, tg = lane & 3;
    const int vrow = (lane & 7) + 8 * (lane >> 4), vcol = 8 * ((lane >> 3) & 1);
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int ks = kg; ks < K16 / 16; ks += ngr) {
      const __nv_bfloat16* pr = &sm.pb[gr][16 * ks + 2 * tg];
      const uint32_t b0 = *reinterpret_cast<const uint32_t*>(pr);
      const uint32_t b1 = *reinterpret_cast<const uint32_t*>(pr + 8);
      const int col = 16 * mt + vcol;
      uint32_t a0, a1, a2, a3;
      ldsm_x4_t(smem_u32(vst) + sg_voff(16 * ks + vrow, col >> 3), a0, a1, a2, a3);
      mma_bf16(acc, a0, a1, a2, a3, b0, b1);
    }
    float* rw = sm.red[warp];
    rw[(2 * tg) * 16 + gr] = acc[0];
    rw[(2 * tg + 1) * 16 + gr] = acc[1];
    rw[(2 * tg) * 16 + gr + 8] = acc[2];
    rw[(2 * tg + 1) * 16 + gr + 8] = acc[3];
  } else {
    const int items = GM * W, parts = NTH / items;
    const int part = tid / items, it = tid % items, h = it / W, d = it % W;
    float a = 0.f;
    if (part < parts && h < G) {
      const float* vf = reinterpret_cast<const float*>(vst);
      for (int j = part; j < K; j += parts) a = fmaf(sm.pz[h][j], vf[j * W + d], a);
    }
    (&sm.red[0][0])[tid] = a;
  }
  if (err) atomicOr(p.err, err);
  __syncthreads();

  // Combine (thread per (head, dimension)): kept part and text part in
  // log-sum-exp form, normalised over the kept and text tokens only.
  for (int i = tid; i < G * W; i += NTH) {
    const int h = i / W, d = i % W;
    float kv = 0.f;
    if constexpr (BF) {
      const int mt = d / 16, dd = d % 16;
      for (int kg = 0; kg < NW / nmt; ++kg) kv += sm.red[kg * nmt + mt][h * 16 + dd];
    } else {
      const int items = GM * W;
      for (int part = 0; part < NTH / items; ++part) kv += (&sm.red[0][0])[part * items + h * W + d];
    }
    const float4 t4 = sm.to[h * W4 + d / 4];
    const float tv = (d & 3) == 0 ? t4.x : (d & 3) == 1 ? t4.y : (d & 3) == 2 ? t4.z : t4.w;
    const float mk = sm.fin[h][0], lk = sm.fin[h][1], mt = sm.hMt[h], lt = sm.hLt[h];
    const float M = fmaxf(mk, mt);
    const float ak = exp2_rel(mk, M), at = exp2_rel(mt, M);
    const float den = ak * lk + at * lt;
    const float o = den > 0.f ? (ak * kv + at * tv) / den : 0.f;
    reinterpret_cast<T*>(p.out)[(hrow0 + h) * D + d0 + d] = from_f<T>(o);
  }
  if (ncl > 1) asm volatile("barrier.cluster.wait.acquire;\n" ::: "memory");
}

// ------------------------------------------------------------------ launching

cudaError_t launch_ex(void (*kernel)(StepParams), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                      int cluster, const StepParams& p) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attrs[2];
  int na = 0;
  attrs[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[na].val.programmaticStreamSerializationAllowed = 1;
  ++na;
  if (cluster > 1) {
    attrs[na].id = cudaLaunchAttributeClusterDimension;
    attrs[na].val.clusterDim.x = cluster;
    attrs[na].val.clusterDim.y = 1;
    attrs[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attrs;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, kernel, p);
}

template <int D, int NT>
size_t mma_smem() { return MmaCfg<D, NT>::SMEM; }
template <int D, int GM>
size_t f32_smem() { return sizeof(F32Smem<D, GM>); }
template <typename T, int D, int GM>
size_t gather_smem() { return sizeof(GatherSmem<T, D, GM>); }

// Warps per CTA and ring slots per warp of the bulk-tensor score kernel: two
// CTAs (8 warps) share an SM, each warp with 24 KB of its tiles in flight.
constexpr int kTmaWarps = 4;
template <int D>
constexpr int tma_slots() { return D == 128 ? 3 : 5; }
template <int D, int NT>
size_t tma_smem() { return TmaCfg<D, NT, kTmaWarps, tma_slots<D>()>::SMEM; }

template <int D>
cudaError_t launch_score_d(const StepParams& p, cudaStream_t st) {
  const dim3 grid(p.ns, p.Hkv, p.B);
  if (D == 128 && p.use_tc && !p.anchor) {
    if (p.G <= 8) return launch_ex(k_score_tc<8>, grid, dim3(kTcThreads), TcCfg::SMEM, st, 1, p);
    return launch_ex(k_score_tc<16>, grid, dim3(kTcThreads), TcCfg::SMEM, st, 1, p);
  }
  if (p.dtype == 0 && p.use_tma) {
    constexpr int NW = kTmaWarps, S = tma_slots<D>();
    if (p.anchor) {
      if (p.G <= 8) return launch_ex(k_score_tma<D, 1, NW, S, true>, grid, dim3(32 * NW), tma_smem<D, 1>(), st, 1, p);
      return launch_ex(k_score_tma<D, 2, NW, S, true>, grid, dim3(32 * NW), tma_smem<D, 2>(), st, 1, p);
    }
    if (p.G <= 8) return launch_ex(k_score_tma<D, 1, NW, S, false>, grid, dim3(32 * NW), tma_smem<D, 1>(), st, 1, p);
    return launch_ex(k_score_tma<D, 2, NW, S, false>, grid, dim3(32 * NW), tma_smem<D, 2>(), st, 1, p);
  }
  if (p.dtype == 0) {
    if (p.G <= 8) return launch_ex(k_score_mma<D, 1>, grid, dim3(kThreads), mma_smem<D, 1>(), st, 1, p);
    return launch_ex(k_score_mma<D, 2>, grid, dim3(kThreads), mma_smem<D, 2>(), st, 1, p);
  }
  if (p.G <= 4) return launch_ex(k_score_f32<D, 4>, grid, dim3(kThreads), f32_smem<D, 4>(), st, 1, p);
  if (p.G <= 8) return launch_ex(k_score_f32<D, 8>, grid, dim3(kThreads), f32_smem<D, 8>(), st, 1, p);
  return launch_ex(k_score_f32<D, 16>, grid, dim3(kThreads), f32_smem<D, 16>(), st, 1, p);
}

template <int GM>
size_t slice_smem() { return sizeof(SliceSmem<GM>); }

// CTAs of a chunk-gather instance resident on one SM (queried once).
template <int D, int NT, int S>
int gm_blocks_per_sm() {
  static const int n = [] {
    int b = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, k_gather_mma<D, NT, S>, 32 * kGmWarps,
                                                      GmCfg<D, NT, S>::SMEM) != cudaSuccess)
      b = 0;
    return b;
  }();
  return n;
}
// True when the two-slot form runs n CTAs in fewer waves than the three-slot one.
template <int D, int NT>
bool gm_fewer_waves(long long n, int num_sms) {
  const long long r2 = (long long)gm_blocks_per_sm<D, NT, 2>() * num_sms;
  const long long r3 = (long long)gm_blocks_per_sm<D, NT, kGmSlots>() * num_sms;
  if (r2 <= 0 || r3 <= 0) return false;
  return (n + r2 - 1) / r2 < (n + r3 - 1) / r3;
}

template <typename T, int D>
cudaError_t launch_gather_td(const StepParams& p, cudaStream_t st) {
  if (p.gslice) {
    const dim3 grid(D / kSliceDims, p.Hkv, p.B);
    if (p.G <= 4) return launch_ex(k_gather_slice<T, D, 4>, grid, dim3(kGatherThreads), slice_smem<4>(), st, 1, p);
    if (p.G <= 8) return launch_ex(k_gather_slice<T, D, 8>, grid, dim3(kGatherThreads), slice_smem<8>(), st, 1, p);
    return launch_ex(k_gather_slice<T, D, 16>, grid, dim3(kGatherThreads), slice_smem<16>(), st, 1, p);
  }
  const dim3 grid(p.nc, p.Hkv, p.B);
  if (sizeof(T) == 2) {
    // A single ring slot when no chunk can hold more than one tile per warp.
    const int kmax = min(p.kept_cap, p.max_visual);
    const bool one = p.nk == 0 || (kmax + p.nk - 1) / p.nk <= GmCfg<D, 1, 1>::MAX_CHUNK;
    const long long n = (long long)p.nc * p.Hkv * p.B;
    if (p.G <= 8) {
      if (one) return launch_ex(k_gather_mma<D, 1, 1>, grid, dim3(32 * kGmWarps), GmCfg<D, 1, 1>::SMEM, st, 1, p);
      if (gm_fewer_waves<D, 1>(n, p.num_sms))
        return launch_ex(k_gather_mma<D, 1, 2>, grid, dim3(32 * kGmWarps), GmCfg<D, 1, 2>::SMEM, st, 1, p);
      return launch_ex(k_gather_mma<D, 1, kGmSlots>, grid, dim3(32 * kGmWarps), GmCfg<D, 1, kGmSlots>::SMEM, st, 1, p);
    }
    if (one) return launch_ex(k_gather_mma<D, 2, 1>, grid, dim3(32 * kGmWarps), GmCfg<D, 2, 1>::SMEM, st, 1, p);
    if (gm_fewer_waves<D, 2>(n, p.num_sms))
      return launch_ex(k_gather_mma<D, 2, 2>, grid, dim3(32 * kGmWarps), GmCfg<D, 2, 2>::SMEM, st, 1, p);
    return launch_ex(k_gather_mma<D, 2, kGmSlots>, grid, dim3(32 * kGmWarps), GmCfg<D, 2, kGmSlots>::SMEM, st, 1, p);
  }
  if (p.G <= 4) return launch_ex(k_gather<T, D, 4>, grid, dim3(kGatherThreads), gather_smem<T, D, 4>(), st, 1, p);
  if (p.G <= 8) return launch_ex(k_gather<T, D, 8>, grid, dim3(kGatherThreads), gather_smem<T, D, 8>(), st, 1, p);
  return launch_ex(k_gather<T, D, 16>, grid, dim3(kGatherThreads), gather_smem<T, D, 16>(), st, 1, p);
}

cudaError_t set_smem(void (*kernel)(StepParams), size_t bytes) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

// The score and gather kernels' shared memory depends only on their template shape.
cudaError_t configure_fixed_kernels() {
  cudaError_t e = cudaSuccess;
#define VP_SET(kernel, bytes) if (e == cudaSuccess) e = set_smem(kernel, bytes)
  VP_SET((k_score_tc<8>), (TcCfg::SMEM));
  VP_SET((k_score_tc<16>), (TcCfg::SMEM));
  VP_SET((k_gather_mma<128, 1, kGmSlots>), (GmCfg<128, 1, kGmSlots>::SMEM));
  VP_SET((k_gather_mma<128, 2, kGmSlots>), (GmCfg<128, 2, kGmSlots>::SMEM));
  VP_SET((k_gather_mma<64, 1, kGmSlots>), (GmCfg<64, 1, kGmSlots>::SMEM));
  VP_SET((k_gather_mma<64, 2, kGmSlots>), (GmCfg<64, 2, kGmSlots>::SMEM));
  VP_SET((k_gather_mma<128, 1, 2>), (GmCfg<128, 1, 2>::SMEM));
  VP_SET((k_gather_mma<128, 2, 2>), (GmCfg<128, 2, 2>::SMEM));
  VP_SET((k_gather_mma<64, 1, 2>), (GmCfg<64, 1, 2>::SMEM));
  VP_SET((k_gather_mma<64, 2, 2>), (GmCfg<64, 2, 2>::SMEM));
  VP_SET((k_gather_mma<128, 1, 1>), (GmCfg<128, 1, 1>::SMEM));
  VP_SET((k_gather_mma<128, 2, 1>), (GmCfg<128, 2, 1>::SMEM));
  VP_SET((k_gather_mma<64, 1, 1>), (GmCfg<64, 1, 1>::SMEM));
  VP_SET((k_gather_mma<64, 2, 1>), (GmCfg<64, 2, 1>::SMEM));
  VP_SET((k_score_tma<128, 1, kTmaWarps, tma_slots<128>(), false>), (tma_smem<128, 1>()));
  VP_SET((k_score_tma<128, 2, kTmaWarps, tma_slots<128>(), false>), (tma_smem<128, 2>()));
  VP_SET((k_score_tma<64, 1, kTmaWarps, tma_slots<64>(), false>), (tma_smem<64, 1>()));
  VP_SET((k_score_tma<64, 2, kTmaWarps, tma_slots<64>(), false>), (tma_smem<64, 2>()));
  VP_SET((k_score_tma<128, 1, kTmaWarps, tma_slots<128>(), true>), (tma_smem<128, 1>()));
  VP_SET((k_score_tma<128, 2, kTmaWarps, tma_slots<128>(), true>), (tma_smem<128, 2>()));
  VP_SET((k_score_tma<64, 1, kTmaWarps, tma_slots<64>(), true>), (tma_smem<64, 1>()));
  VP_SET((k_score_tma<64, 2, kTmaWarps, tma_slots<64>(), true>), (tma_smem<64, 2>()));
  VP_SET((k_score_mma<128, 1>), (mma_smem<128, 1>()));
  VP_SET((k_score_mma<128, 2>), (mma_smem<128, 2>()));
  VP_SET((k_score_mma<64, 1>), (mma_smem<64, 1>()));
  VP_SET((k_score_mma<64, 2>), (mma_smem<64, 2>()));
  VP_SET((k_score_f32<128, 4>), (f32_smem<128, 4>()));
  VP_SET((k_score_f32<128, 8>), (f32_smem<128, 8>()));
  VP_SET((k_score_f32<128, 16>), (f32_smem<128, 16>()));
  VP_SET((k_score_f32<64, 4>), (f32_smem<64, 4>()));
  VP_SET((k_score_f32<64, 8>), (f32_smem<64, 8>()));
  VP_SET((k_score_f32<64, 16>), (f32_smem<64, 16>()));
  VP_SET((k_gather<__nv_bfloat16, 128, 4>), (gather_smem<__nv_bfloat16, 128, 4>()));
  VP_SET((k_gather<__nv_bfloat16, 128, 8>), (gather_smem<__nv_bfloat16, 128, 8>()));
  VP_SET((k_gather<__nv_bfloat16, 128, 16>), (gather_smem<__nv_bfloat16, 128, 16>()));
  VP_SET((k_gather<__nv_bfloat16, 64, 4>), (gather_smem<__nv_bfloat16, 64, 4>()));
  VP_SET((k_gather<__nv_bfloat16, 64, 8>), (gather_smem<__nv_bfloat16, 64, 8>()));
  VP_SET((k_gather<__nv_bfloat16, 64, 16>), (gather_smem<__nv_bfloat16, 64, 16>()));
  VP_SET((k_gather<float, 128, 4>), (gather_smem<float, 128, 4>()));
  VP_SET((k_gather<float, 128, 8>), (gather_smem<float, 128, 8>()));
  VP_SET((k_gather<float, 128, 16>), (gather_smem<float, 128, 16>()));
  VP_SET((k_gather<float, 64, 4>), (gather_smem<float, 64, 4>()));
  VP_SET((k_gather<float, 64, 8>), (gather_smem<float, 64, 8>()));
  VP_SET((k_gather<float, 64, 16>), (gather_smem<float, 64, 16>()));
  VP_SET((k_gather_slice<__nv_bfloat16, 128, 4>), (slice_smem<4>()));
  VP_SET((k_gather_slice<__nv_bfloat16, 128, 8>), (slice_smem<8>()));
  VP_SET((k_gather_slice<__nv_bfloat16, 128, 16>), (slice_smem<16>()));
  VP_SET((k_gather_slice<__nv_bfloat16, 64, 4>), (slice_smem<4>()));
  VP_SET((k_gather_slice<__nv_bfloat16, 64, 8>), (slice_smem<8>()));
  VP_SET((k_gather_slice<__nv_bfloat16, 64, 16>), (slice_smem<16>()));
  VP_SET((k_gather_slice<float, 128, 4>), (slice_smem<4>()));
  VP_SET((k_gather_slice<float, 128, 8>), (slice_smem<8>()));
  VP_SET((k_gather_slice<float, 128, 16>), (slice_smem<16>()));
  VP_SET((k_gather_slice<float, 64, 4>), (slice_smem<4>()));
  VP_SET((k_gather_slice<float, 64, 8>), (slice_smem<8>()));
  VP_SET((k_gather_slice<float, 64, 16>), (slice_smem<16>()));
#undef VP_SET
  if (e == cudaSuccess) {  // the chunk gather's occupancies, now that its shared memory is set
    gm_blocks_per_sm<128, 1, 2>(); gm_blocks_per_sm<128, 1, kGmSlots>();
    gm_blocks_per_sm<128, 2, 2>(); gm_blocks_per_sm<128, 2, kGmSlots>();
    gm_blocks_per_sm<64, 1, 2>(); gm_blocks_per_sm<64, 1, kGmSlots>();
    gm_blocks_per_sm<64, 2, 2>(); gm_blocks_per_sm<64, 2, kGmSlots>();
  }
  return e;
}

size_t select_smem_bytes(int max_visual) { return ((size_t)(max_visual > 0 ? max_visual : 1) + 3) / 4 * 16; }

}  // namespace

cudaError_t launch_score(const StepParams& p, cudaStream_t st) {
  return p.D == 128 ? launch_score_d<128>(p, st) : launch_score_d<64>(p, st);
}

cudaError_t launch_gather(const StepParams& p, cudaStream_t st) {
  if (p.fused == 1) return cudaSuccess;  // the select kernel gathered
  if (p.dtype == 0)
    return p.D == 128 ? launch_gather_td<__nv_bfloat16, 128>(p, st) : launch_gather_td<__nv_bfloat16, 64>(p, st);
  return p.D == 128 ? launch_gather_td<float, 128>(p, st) : launch_gather_td<float, 64>(p, st);
}

cudaError_t launch_compact(const CompactParams& c, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((c.max_seq + kCompactRows - 1) / kCompactRows, c.Hkv, c.B);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_compact, c);
}

// Dynamic shared memory of k_selgat: the score keys, then the cut's per-warp
// histograms, then the kept rows' V slices of W dimensions (bf16: one or two
// halves of rows of 128 bytes; fp32: packed rows).
size_t selgat_smem_bytes(int max_visual, int dtype, int W = 64) {
  const size_t keys = select_smem_bytes(max_visual);
  const size_t stage = (size_t)kSliceMaxKept * (dtype == 0 ? (W > 64 ? 256 : 128) : W * 4);
  const size_t hist = (size_t)2 * kSgWarps * 256 * 4;  // the cut's per-warp histograms
  size_t n = keys > stage ? keys : stage;
  return n > hist ? n : hist;
}

template <typename T, int D>
cudaError_t launch_selgat_td(const StepParams& p, dim3 grid, size_t smem, cudaStream_t st) {
  if (p.G <= 4) return launch_ex(k_selgat<T, D, 4>, grid, dim3(kSgThreads), smem, st, p.cl, p);
  return launch_ex(k_selgat<T, D, 8>, grid, dim3(kSgThreads), smem, st, p.cl, p);
}

cudaError_t launch_select(const StepParams& p, cudaStream_t st) {
  const dim3 grid(p.cl, p.granularity ? p.Hkv : 1, p.B);
  if (p.fused == 2)
    return launch_ex(k_selgat<__nv_bfloat16, 128, 8, false>, grid, dim3(kSgThreads),
                     selgat_smem_bytes(p.max_visual, 0), st, p.cl, p);
  if (p.fused == 1) {
    const size_t smem = selgat_smem_bytes(p.max_visual, p.dtype, selgat_slice_dims(p));
    if (p.dtype == 0)
      return p.D == 128 ? launch_selgat_td<__nv_bfloat16, 128>(p, grid, smem, st)
                        : launch_selgat_td<__nv_bfloat16, 64>(p, grid, smem, st);
    return p.D == 128 ? launch_selgat_td<float, 128>(p, grid, smem, st) : launch_selgat_td<float, 64>(p, grid, smem, st);
  }
  const size_t smem = select_smem_bytes(p.max_visual);
  if ((p.max_visual + p.cl - 1) / p.cl <= kSelSliceSmall) return launch_ex(k_select<512>, grid, dim3(512), smem, st, p.cl, p);
  return launch_ex(k_select<1024>, grid, dim3(1024), smem, st, p.cl, p);
}

namespace {
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      f = nullptr;
    cudaGetLastError();
    return reinterpret_cast<EncodeTiledFn>(f);
  }();
  return fn;
}

// 4-D descriptor of one cache: dims {D, token, kv-head, sequence or page}, the
// last three ordered by increasing stride, boxes of 64 dimensions x R rows.
// Returns false for a layout whose extent along the token axis cannot be
// bounded by the caller's memory.
bool encode_one(const KvView& kv, const StepParams& p, CUtensorMap* map, int* tpos, int* gpos, int* bpos, int R) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || !kv.data) return false;
  struct Ax { int64_t stride, size; int id; };  // id: 0 token, 1 kv-head, 2 sequence / page
  Ax ax[3] = {{kv.st, 0, 0}, {kv.sh, p.Hkv, 1}, {kv.sb, p.paged ? kv.num_pages : p.B, 2}};
  if (p.paged) ax[0].size = p.page_size;
  for (int i = 0; i < 3; ++i)
    for (int j = i + 1; j < 3; ++j)
      if (ax[j].stride < ax[i].stride) { Ax t = ax[i]; ax[i] = ax[j]; ax[j] = t; }
  if (ax[0].stride < p.D) return false;
  if (!p.paged) {
    // The token extent is the room its stride leaves before the next axis.
    int k = 0;
    while (ax[k].id != 0) ++k;
    if (k == 2 || ax[k].stride <= 0) return false;
    ax[k].size = ax[k + 1].stride / ax[k].stride;
  }
  for (int i = 0; i < 3; ++i) {
    if (ax[i].size < 1 || ax[i].stride <= 0) return false;
    if (i < 2 && ax[i + 1].stride < ax[i].stride * ax[i].size) return false;  // axes must nest
  }
  cuuint64_t dims[4] = {(cuuint64_t)p.D, (cuuint64_t)ax[0].size, (cuuint64_t)ax[1].size, (cuuint64_t)ax[2].size};
  // Rows at or past max_seq are never read: the copy fills them with zeros.
  for (int i = 0; i < 3; ++i)
    if (!p.paged && ax[i].id == 0 && ax[i].size > p.max_seq) dims[i + 1] = (cuuint64_t)p.max_seq;
  const cuuint64_t strides[3] = {(cuuint64_t)ax[0].stride * 2, (cuuint64_t)ax[1].stride * 2, (cuuint64_t)ax[2].stride * 2};
  cuuint32_t box[4] = {64, 1, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  for (int i = 0; i < 3; ++i) {
    if (ax[i].id == 0) { box[i + 1] = (cuuint32_t)R; *tpos = i + 1; }
    if (ax[i].id == 1) *gpos = i + 1;
    if (ax[i].id == 2) *bpos = i + 1;
  }
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(kv.data), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}
}  // namespace

void encode_kv_maps(StepParams& p) {
  const bool want_tc = p.use_tc != 0;
  p.use_tma = 0;
  p.use_tc = 0;
  if (p.dtype != 0 || (p.D != 64 && p.D != 128)) return;
  if (p.paged && p.page_size < 8) return;  // box origins must stay 1024-byte aligned in shared memory
  const int R = p.paged ? (p.page_size < kTmaTile ? p.page_size : kTmaTile) : kTmaTile;
  int kt = 0, kg = 0, kb = 0, vt = 0, vg = 0, vb = 0;
  if (!encode_one(p.k, p, &p.tmk, &kt, &kg, &kb, R) || !encode_one(p.v, p, &p.tmv, &vt, &vg, &vb, R)) return;
  if (kt != vt || kg != vg || kb != vb) return;  // both caches must share an axis order
  p.tpos = kt; p.gpos = kg; p.bpos = kb;
  if (want_tc && tc_eligible(p.dtype, p.D, p.G, p.paged, p.page_size)) {
    // Page ids of a split's boxes are staged in shared memory: bound them.
    const int R2 = p.paged ? (p.page_size < kTcRows ? p.page_size : kTcRows) : kTcRows;
    const int64_t boxes = p.paged ? (int64_t)tc_max_split_tiles(p.max_seq, p.ns, p.split_w) * (kTcRows / R2) : 0;
    if (boxes <= kTcMaxBoxes && encode_one(p.k, p, &p.tmk2, &kt, &kg, &kb, R2) &&
        encode_one(p.v, p, &p.tmv2, &vt, &vg, &vb, R2) && kt == p.tpos && vt == p.tpos && kg == p.gpos &&
        vg == p.gpos && kb == p.bpos && vb == p.bpos)
      p.use_tc = 1;
    p.use_tma = 1;
    return;
  }
  if (p.paged) {
    // Page ids of a CTA's boxes are staged in shared memory: bound them.
    const int64_t tiles = (p.max_seq + kTmaTile - 1) / kTmaTile;
    const int64_t per_cta = (2 * tiles + p.ns - 1) / p.ns + 1;
    const int64_t boxes = per_cta * (kTmaTile / R);
    if (boxes > kTmaMaxBoxes) return;
  }
  p.use_tma = 1;
}

cudaError_t configure_kernels(int max_visual, int H, int nsp_max) {
  (void)H;
  (void)nsp_max;
  const int need = (int)select_smem_bytes(max_visual);
  cudaError_t e = cudaSuccess;
  for (void (*k)(StepParams) : {k_select<512>, k_select<1024>}) {
    cudaFuncAttributes attr;
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&attr, k);
    if (e == cudaSuccess && attr.maxDynamicSharedSizeBytes < need) e = set_smem(k, need);
  }
  {
    cudaFuncAttributes attr;
    const int need = (int)selgat_smem_bytes(max_visual, 0);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&attr, k_selgat<__nv_bfloat16, 128, 8, false>);
    if (e == cudaSuccess && attr.maxDynamicSharedSizeBytes < need) e = set_smem(k_selgat<__nv_bfloat16, 128, 8, false>, need);
  }
  void (*const selgat[2][4])(StepParams) = {
      {k_selgat<__nv_bfloat16, 128, 4>, k_selgat<__nv_bfloat16, 128, 8>, k_selgat<__nv_bfloat16, 64, 4>,
       k_selgat<__nv_bfloat16, 64, 8>},
      {k_selgat<float, 128, 4>, k_selgat<float, 128, 8>, k_selgat<float, 64, 4>, k_selgat<float, 64, 8>}};
  for (int dt = 0; dt < 2; ++dt) {
    const int need_sg = (int)selgat_smem_bytes(max_visual, dt, dt == 0 ? kSgMaxW : 64);
    for (void (*k)(StepParams) : selgat[dt]) {
      cudaFuncAttributes attr;
      if (e == cudaSuccess) e = cudaFuncGetAttributes(&attr, k);
      if (e == cudaSuccess && attr.maxDynamicSharedSizeBytes < need_sg) e = set_smem(k, need_sg);
    }
  }
  return e == cudaSuccess ? configure_fixed_kernels() : e;
}

}  // namespace vp
