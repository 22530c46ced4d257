// Internal definitions shared by the host side (vp_api.cu) and the kernels
// (vp_kernels.cu) of libvp.  Not part of the public ABI.
#pragma once

#include <cuda.h>  // CUtensorMap (type only; the library does not link the driver)
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

namespace vp {

// Text of the last failure of a call that has no context (vp_init,
// vp_decode_step_noalloc) in this thread; vp_last_error(NULL) returns it.
std::string& context_free_error();

// Device error word bits (vp_check_errors reports them).
enum : unsigned {
  ERR_SPAN = 1u,       // vis_start / vis_len outside the live cache or max_visual
  ERR_TEXT = 2u,       // text_len < 1 (no current token)
  ERR_LEN = 4u,        // vis_len + text_len > max_seq
  ERR_PAGE = 8u,       // block-table entry outside [0, num_pages) or row past max_pages
  ERR_KEPT = 16u,      // a kept index outside [0, N_v)
  ERR_NONFINITE = 32u, // a non-finite score reached the selection
  ERR_TIMEOUT = 64u    // a bounded wait for an asynchronous copy gave up
};

// Split statistics written by the score kernel for every (sequence, query
// head, split), padded to two float4; maxima are in log2 units (z * log2 e).
// The text half comes first: the gather kernel reads only that float4.
enum { ST_MT = 0, ST_L1T = 1, ST_LTT = 2, ST_MV = 4, ST_L1V = 5, ST_LTV = 6, ST_N = 8 };

struct KvView {
  const void* data;
  int64_t sb, sh, st;          // strides in elements
  const int32_t* block_table;  // paged only
  int32_t max_pages, num_pages;
};

struct StepParams {
  // bulk-tensor (TMA) descriptors of the K and V caches (bf16), when use_tma
  CUtensorMap tmk;  // 64-byte aligned type
  CUtensorMap tmv;
  int use_tma;
  // the same caches in boxes of up to 128 rows, for the tensor-core score
  // kernel (decode step, bf16, D = 128, at most 16 query heads per kv-head)
  CUtensorMap tmk2;
  CUtensorMap tmv2;
  int use_tc;
  int anchor;  // 1: a layer after the anchor layer -- text plus the given kept set, no selection
  int tpos, gpos, bpos;  // descriptor dimension (1..3) of the token, kv-head and sequence/page axes
  // shapes
  int dtype;  // 0 = bf16, 1 = fp32 (vp_dtype)
  int B, H, Hkv, G, D;
  int max_visual, max_seq;
  int paged, page_size, page_shift;
  // inputs
  const void* q;
  KvView k, v;
  const int32_t* vis_start;
  const int32_t* vis_len;
  const int32_t* text_len;
  // budget
  int mode, granularity;
  float inv_tau;   // 1 / tau
  float c_log2;    // logit scale * log2(e)
  int r_lo_ppm, r_hi_ppm, ratio_ppm, fixed_k;
  // outputs
  void* out;
  int32_t* kept_idx;
  int kept_cap;
  int32_t* kept_count;
  float* mass;
  float* mass_stats;
  // workspace
  float* z_ws;        // [max_batch][max_visual][hp] visual logits, log2 units
  float* split_st;    // [max_batch][H][nsp_max][ST_N] (one partial per cluster of splits)
  float* split_o;     // [max_batch][H][nsp_max][D]    text partial outputs
  float* gpart_o;     // [max_batch][Hkv][nk_max][G][D] kept-visual partial outputs
  float* gpart_st;    // [max_batch][Hkv][nk_max][G][2] {max, sum}
  float* mt_o;        // [max_batch][H][D] text output merged over the splits
  float* mt_st;       // [max_batch][H][2] its {max, sum}
  float* hmax;        // [max_batch][H] largest logit of every head over all tokens (log2 units)
  // Diagnostics (Sec. 4.3, App. B), off when both pointers are NULL.
  unsigned act_delta_bits;  // float bits of delta (> 0): a score S_i is active when its bits are larger
  int32_t* n_act;           // [B][nsel] N_act(delta)
  uint32_t* act_bits;       // [B][nsel][act_words] activity bits, OR-accumulated
  int act_words;
  unsigned* tickets;  // [max_batch][Hkv] (zero between calls)
  unsigned* err;      // device error word
  int hp;             // z_ws row stride (H rounded up to a multiple of 4)
  int ns, nsp_max;    // score splits (= text partials) per (sequence, kv-head); allocated
  int cl;             // CTAs in a select cluster
  int nk, nk_max;     // gather chunks used by this call / allocated
  int nm;             // gather CTAs that also merge a slice of the text partials (0: ns == 1)
  int nc;             // gather CTAs per (sequence, kv-head) = max(nk, nm)
  int gslice;         // 1: kept sets fit the single-pass slice gather (kept_cap <= kSliceMaxKept)
  int fused;          // select kernel: 0 k_select; 1 k_selgat, which also gathers (fused_select_gather_ok);
                      // 2 k_selgat selecting only (fast_select_ok)
  int split_w;        // weight of one score split (bulk-tensor kernel)
  int num_sms;        // SMs of the device (launch shapes chosen per call)
};

// ---------------------------------------------------------------- host planning

constexpr int kNkMax = 64;    // kept chunks per (sequence, kv-head)
constexpr int kGmMaxChunk = 2048;   // kept rows of one chunk of the chunk gather
constexpr int kSliceMaxKept = 256;  // kept rows per (sequence, kv-head) the slice gather holds
constexpr int kTcRows = 128;  // rows of a tile of the tensor-core score kernel
// Split weights of the tensor-core score kernel's tiles, in proportion to
// their cost: a tile wholly inside the visual span carries K only (half the
// bytes of a tile with K and V) but takes about 0.7 of its time (the same
// per-tile pipeline steps, plus writing its logits out).  Measured on
// 8 x (4096 visual + 16384 text) tokens: 10 : 20 (bytes) 0.80 of the HBM
// peak, 10 : 18 0.83, 10 : 16 0.84, 10 : 14 0.85, 10 : 12 0.84.
constexpr int kTcWv = 10, kTcWt = 14;
constexpr int kTcMaxBoxes = 384;  // page ids per cache a tensor-core score CTA stages

// The 128-row tiles of one split of the tensor-core score kernel, for a
// sequence of vis_len visual tokens starting at vis_start and text_len text
// tokens.  Tiles [v0, v1) lie wholly inside the visual span (K only, weight
// kTcWv); every other tile carries text or padding rows (K and V, weight
// kTcWt).  Split s owns tiles [u0, u0 + n): the tiles whose weight prefix
// falls in [s * per, (s + 1) * per), per = max(split_w, ceil(W / ns)), so the
// splits partition the sequence's tiles; tc_max_split_tiles bounds n.
struct TcRange {
  int u0, n, v0, v1;
  __host__ __device__ bool pure(int i) const { return u0 + i >= v0 && u0 + i < v1; }
};
__host__ __device__ inline TcRange tc_split(int vis_start, int vis_len, int text_len, int s, int ns, int split_w) {
  const int T = vis_len + text_len;
  const int NTl = (T + kTcRows - 1) / kTcRows;
  TcRange r;
  r.v0 = (vis_start + kTcRows - 1) / kTcRows;
  const int vend = (vis_start + vis_len) / kTcRows;
  r.v1 = NTl < vend ? NTl : vend;
  if (r.v1 < r.v0) r.v1 = r.v0;
  const int W = kTcWt * NTl - (kTcWt - kTcWv) * (r.v1 - r.v0);
  const int fair = (W + ns - 1) / ns;
  const int per = split_w > fair ? split_w : fair;
  const int wa = kTcWt * r.v0, wc = wa + kTcWv * (r.v1 - r.v0);  // weight before and up to the end of the span's tiles
  auto tile_of = [&](int w) {  // first tile whose weight prefix reaches w
    if (w <= wa) return (w + kTcWt - 1) / kTcWt;
    if (w <= wc) return r.v0 + (w - wa + kTcWv - 1) / kTcWv;
    return r.v1 + (w - wc + kTcWt - 1) / kTcWt;
  };
  const int w0 = s * per < W ? s * per : W, w1 = (s + 1) * per < W ? (s + 1) * per : W;
  r.u0 = tile_of(w0);
  r.n = tile_of(w1) - r.u0;
  return r;
}
// The most tiles a tc_split split holds for any sequence of at most max_seq
// tokens: per is largest for a sequence with no visual tile (every tile
// weighs kTcWt), and a split's tiles weigh at least kTcWv each, plus one for
// the tile its weight range starts inside.
inline int tc_max_split_tiles(int max_seq, int ns, int split_w) {
  const long long ntl = (max_seq + kTcRows - 1) / kTcRows;
  const long long fair = (kTcWt * ntl + ns - 1) / ns;
  const long long per = split_w > fair ? split_w : fair;
  return (int)(per / kTcWv + 1);
}
constexpr int kNsMax = 256;   // score splits per (sequence, kv-head)
constexpr int kMaxMerge = 8;  // gather CTAs merging slices of the text partials

// Launch plan of one call: score CTAs sized to the work (see below),
// select clusters that spread the importance scores of few sequences over
// several SMs, gather chunks of 256 to 2048 kept rows.
struct Plan {
  int ns, cl, nk, nm, nc, gslice;
  int split_w;  // weight (tiles, text tiles counting 2) of one score split
};

// tc: the score splits are for the tensor-core kernel (128-row tiles).
inline Plan make_plan(int batch, int Hkv, int D, int num_sms, int max_visual, int max_seq, int kept_cap,
                      int granularity, bool tc = false) {
  const long long units = (long long)batch * Hkv;
  const int TR = tc ? kTcRows : 32;
  // Fixed-weight splits sized for the longest sequence (tiles wholly inside
  // the visual span carry K only and weigh 1, the others K and V and weigh
  // 2): shorter sequences use fewer splits, so every working score CTA
  // carries about the same work.
  long long w_max = tc ? (long long)kTcWt * ((max_seq + TR - 1) / TR) - (long long)(kTcWt - kTcWv) * (max_visual / TR)
                       : 2LL * ((max_seq + TR - 1) / TR) - max_visual / TR;
  if (w_max < 1) w_max = 1;
  // Work of the longest sequence in tiles for the split count (32-row tiles:
  // the visual span counted once more).  Score CTAs are small enough that
  // two fit on an SM.
  const long long tiles = tc ? w_max : (max_visual + 31) / 32 + 2LL * ((max_seq + 31) / 32);
  const long long slots = 2LL * num_sms;
  // Split count: minimise (waves of CTAs) x (tiles per CTA + a fixed cost per
  // CTA for its start, its pipeline fill and its partial), keeping a minimum
  // of work per CTA; the smaller count wins a tie.  The costs were measured
  // across the sweep workloads: about 12 tiles of 32 rows for the mma.sync
  // kernel, about 6 weight units of 128 rows for the tensor-core kernel.
  long long ns_hi = tiles / (tc ? 2 * kTcWv : 8);
  if (ns_hi > kNsMax) ns_hi = kNsMax;
  if (ns_hi < 1) ns_hi = 1;
  const double fixed = tc ? 6.0 * kTcWv : 12.0;
  long long ns = 1;
  double best = 0.0;
  for (long long c = 1; c <= ns_hi; ++c) {
    const double waves = (double)((units * c + slots - 1) / slots);
    const double cost = waves * ((double)tiles / (double)c + fixed);
    if (c == 1 || cost < best * (1.0 - 1e-9)) { best = cost; ns = c; }
  }
  const long long sel = (long long)batch * (granularity ? Hkv : 1);
  int cl = 1;
  while (cl < 8 && sel * cl * 2 <= num_sms) cl *= 2;
  // Kept chunks of about 2048 rows, smaller (down to 256) while the gather
  // grid would not fill the GPU once (measured against 1024-row chunks and a
  // twice-filled grid: the chunk gather 5% to 22% faster across the sweep).
  long long nk = (kept_cap + kGmMaxChunk - 1) / kGmMaxChunk;
  const long long nk_want = (slots + units - 1) / units, nk_small = (kept_cap + 255) / 256;
  if (nk < nk_want) nk = nk_want < nk_small ? nk_want : nk_small;
  if (nk < 1) nk = 1;
  if (nk > kNkMax) nk = kNkMax;
  // Text-partial merge slices: as many as there are kept chunks (a power of
  // two up to D / 16 and kMaxMerge), so that no CTA merges text alone.
  int nm = 0;
  if (ns > 1) {
    const long long cap_m = D / 16 < kMaxMerge ? D / 16 : kMaxMerge;
    nm = 1;
    while (2LL * nm <= cap_m && 2LL * nm <= nk) nm *= 2;
  }
  // Small kept sets of few sequences: one CTA per 16 output dimensions, so
  // that the whole gather is one short wave; otherwise one CTA per chunk.
  const int gslice = kept_cap <= kSliceMaxKept && units * (D / 16) <= slots ? 1 : 0;
  const int split_w = (int)((w_max + ns - 1) / ns);
  return Plan{(int)ns, cl, (int)nk, nm, (int)(nk > nm ? nk : nm), gslice, split_w};
}

// Workspace layout for up to `batch` sequences (offsets in bytes, 256-aligned).
// The first `zero_bytes` (tickets, error word) must be zero before a call.
struct WsLayout {
  size_t o_tickets, o_err, zero_bytes, o_z, o_st, o_o, o_go, o_gs, o_mo, o_ms, o_hm, total;
  int hp, nsp_max, nk_max;
};

inline size_t ws_round(size_t x) { return (x + 255) / 256 * 256; }

inline WsLayout ws_layout(int batch, int H, int Hkv, int D, int max_visual, int max_seq, int num_sms) {
  WsLayout w;
  w.hp = (H + 3) / 4 * 4;
  w.nk_max = kNkMax;
  w.nsp_max = 1;
  for (int bb = 1; bb <= batch; ++bb)
    for (int tc = 0; tc < 2; ++tc) {
      const Plan pl = make_plan(bb, Hkv, D, num_sms, max_visual, max_seq, 0, 0, tc != 0);
      if (pl.ns > w.nsp_max) w.nsp_max = pl.ns;
    }
  const size_t B = (size_t)batch, G = (size_t)(H / Hkv);
  size_t off = 0;
  w.o_tickets = off; off = ws_round(off + B * Hkv * 4);
  w.o_err = off; off = ws_round(off + 4);
  w.zero_bytes = off;
  w.o_z = off; off = ws_round(off + B * (size_t)(max_visual > 0 ? max_visual : 1) * w.hp * 4);
  w.o_st = off; off = ws_round(off + B * H * (size_t)w.nsp_max * ST_N * 4);
  w.o_o = off; off = ws_round(off + B * H * (size_t)w.nsp_max * D * 4);
  w.o_go = off; off = ws_round(off + B * Hkv * (size_t)w.nk_max * G * D * 4);
  w.o_gs = off; off = ws_round(off + B * Hkv * (size_t)w.nk_max * G * 2 * 4);
  w.o_mo = off; off = ws_round(off + B * H * (size_t)D * 4);
  w.o_ms = off; off = ws_round(off + B * H * 2 * 4);
  w.o_hm = off; off = ws_round(off + B * H * 4);
  w.total = off;
  return w;
}

// Cache compaction for FastV + VisionPulse (vp_compact_kv).
struct CompactParams {
  KvView src;                  // contiguous or paged (block_table set)
  int paged, page_size, page_shift;
  void* dst;                   // contiguous destination
  int64_t dsb, dsh, dst_t;     // its strides in elements
  const int32_t* vis_start;
  const int32_t* vis_len;
  const int32_t* text_len;
  const int32_t* kept_idx;
  int kept_cap;
  const int32_t* kept_count;
  int B, Hkv, D, esz, max_visual, max_seq;
  unsigned* err;
};
cudaError_t launch_compact(const CompactParams& c, cudaStream_t s);

// Launchers (vp_kernels.cu).  Return the launch error, if any.
cudaError_t launch_score(const StepParams& p, cudaStream_t s);
cudaError_t launch_select(const StepParams& p, cudaStream_t s);
cudaError_t launch_gather(const StepParams& p, cudaStream_t s);
// Kernel attributes: raises (never lowers) the select kernel's dynamic
// shared-memory limit for these shapes and sets the other kernels' limits.
cudaError_t configure_kernels(int max_visual, int H, int nsp_max);
// Fills p.tmk / p.tmv / p.use_tma for a bf16 cache whose layout a 4-D tensor
// descriptor can describe without reaching past the caller's memory; leaves
// use_tma = 0 otherwise (the score kernel then copies rows one by one).
// With p.use_tc set on entry (a plan made for the tensor-core kernel) it also
// fills p.tmk2 / p.tmv2 and keeps use_tc only if that kernel can run.
void encode_kv_maps(StepParams& p);
// The tensor-core score kernel's shape conditions (decode step, bf16, D = 128,
// at most 16 query heads per kv-head, pages of at least 8 rows).
inline bool tc_eligible(int dtype, int D, int G, int paged, int page_size) {
  return dtype == 0 && D == 128 && G >= 1 && G <= 16 && (!paged || page_size >= 8);
}

// Whether one kernel (select + gather) serves the call: kept sets of at most
// kSliceMaxKept rows, the budget known before the selection (not top-p), no
// diagnostics, at most 8 query heads per kv-head, the select cluster's CTAs
// splitting the output dimensions of every kv-head evenly into slices of 16
// to 128 dimensions (64 with fp32 caches), and the score keys of a sequence
// fitting in the cut's registers (eight per thread of 512: N_v <= 4096).
// The select clusters (at most half as many CTAs as SMs) run in one wave.
// Output dimensions of one CTA of the fused select + gather: the cluster's
// ranks split into the kv-heads (one kept set per sequence) or take the
// selection's kv-head (per-kv-head sets), each rank a slice of D; 0 if the
// ranks do not divide evenly.
inline int selgat_slice_dims(const StepParams& p) {
  const int hunits = p.granularity ? 1 : p.Hkv;
  if (p.cl % hunits) return 0;
  const int rpg = p.cl / hunits;
  return p.D % rpg ? 0 : p.D / rpg;
}
inline bool fused_select_gather_ok(const StepParams& p, int kept_cap) {
  if (p.anchor || p.mode == 4 || p.n_act || p.act_bits || p.G > 8 || kept_cap > kSliceMaxKept ||
      p.max_visual > 4096)
    return false;
  const int W = selgat_slice_dims(p);
  return W >= 16 && W <= (p.dtype == 0 ? 128 : 64);
}

// Whether the selection of a call the fused kernel does not serve runs in
// k_selgat's select-only form (its register-resident cut holds at most 4096
// keys) rather than k_select: a budget known before the selection, no
// diagnostics.
inline bool fast_select_ok(const StepParams& p) {
  return !p.anchor && p.mode != 4 && !p.n_act && !p.act_bits && p.max_visual <= 4096;
}
inline int select_kind(const StepParams& p, int kept_cap) {
  return fused_select_gather_ok(p, kept_cap) ? 1 : fast_select_ok(p) ? 2 : 0;
}

// Launch plan and copy descriptors of a decode step (p's shapes, inputs and
// dtype set): the tensor-core score kernel where it can run and pays off,
// otherwise the mma.sync kernels with their own split count.  The
// tensor-core kernel moves 128-row tiles and holds TMEM, so a CTA starts
// later: it is chosen when every (sequence, kv-head) carries at least 32
// weight units of 128-row tiles (about 2000 cache rows) and the call has
// work for many such CTAs (measured: below either bound the mma.sync
// kernel was faster, above both the tensor-core kernel).
// path: 0 the choice above, 1 never the tensor-core kernel, 2 only it
// (false when it cannot serve the call).
inline bool plan_step(StepParams& p, int num_sms, int kept_cap, int granularity, int path = 0) {
  p.num_sms = num_sms;
  const long long w_tc = 2LL * ((p.max_seq + kTcRows - 1) / kTcRows) - p.max_visual / kTcRows;
  const bool eligible = tc_eligible(p.dtype, p.D, p.G, p.paged, p.page_size);
  const bool tc = path == 2 ? eligible
                            : path == 0 && eligible && w_tc >= 32 && (long long)p.B * p.Hkv * w_tc >= 16LL * num_sms;
  if (path == 2 && !tc) return false;
  for (int pass = 0; pass < 2; ++pass) {
    const bool want = tc && pass == 0;
    const Plan pl = make_plan(p.B, p.Hkv, p.D, num_sms, p.max_visual, p.max_seq, kept_cap, granularity, want);
    p.ns = pl.ns; p.cl = pl.cl; p.nk = pl.nk; p.nm = pl.nm; p.nc = pl.nc; p.gslice = pl.gslice;
    p.split_w = pl.split_w;
    p.use_tc = want ? 1 : 0;
    encode_kv_maps(p);
    if (p.use_tc || !want) return true;
    if (path == 2) return false;
  }
  return true;
}

}  // namespace vp
