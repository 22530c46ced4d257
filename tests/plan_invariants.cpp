// Host-only check of the launch planner (make_plan, ws_layout, tc_split,
// select_kind): over a grid of shapes, every plan covers the whole cache with
// its score splits, stays inside the workspace the context allocated, splits
// every sequence's tiles for the tensor-core kernel within the page-id
// staging bound, keeps every gather chunk within the chunk kernel's limit and
// picks the slice gather only for kept sets it holds; a table of call shapes
// gets its expected select form, and a table of the chunk gather's call
// shapes its chunk count, CTAs per (sequence, kv-head) and whether the lone
// CTA combines in place.  Prints one line per violation and exits non-zero if
// there was any.
#include <cstdio>

#include "vp_internal.h"

namespace {

int fails = 0;

void check(bool ok, const char* what, int B, int Hkv, int D, int sms, int mv, int ms, int cap, int tc, int gran) {
  if (ok) return;
  if (++fails <= 20)
    std::printf("FAIL %s: B=%d Hkv=%d D=%d sms=%d max_visual=%d max_seq=%d kept_cap=%d tc=%d gran=%d\n", what, B, Hkv,
                D, sms, mv, ms, cap, tc, gran);
}

bool pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }

// The select form (select_kind) the planner picks for a call shape on a
// 152-SM device: 1 fused select + gather, 2 select only, 0 the
// shared-memory select; and the fused kernel's slice width.
struct FormCase {
  const char* name;
  int B, H, Hkv, D, max_visual, max_seq, kept_cap, gran, dtype, mode, diag;
  int want_kind, want_w;
};

int check_forms() {
  using namespace vp;
  const FormCase cases[] = {
      // name, B, H, Hkv, D, N_v, max_seq, kept_cap, gran, dtype, mode, diag, kind, W
      {"B=1 decode (28/4, N_v 1296)", 1, 28, 4, 128, 1296, 4113, 64, 0, 0, 0, 0, 1, 64},
      {"long reasoning (B=8, N_v 4096)", 8, 28, 4, 128, 4096, 21000, 204, 0, 0, 0, 0, 1, 64},
      {"batched serving (B=32, N_v 2304)", 32, 28, 4, 128, 2304, 6500, 115, 0, 0, 0, 0, 1, 128},
      {"sweep B=64, 32/8, N_v 2304, 5%", 64, 32, 8, 128, 2304, 3400, 115, 0, 0, 0, 0, 2, 0},
      {"sweep B=64, N_v 6400 (keys beyond the register cut)", 64, 32, 8, 128, 6400, 7500, 320, 0, 0, 0, 0, 0, 0},
      {"kept sets above 256 rows", 8, 28, 4, 128, 4096, 21000, 2048, 0, 0, 0, 0, 2, 0},
      {"top-p budget", 1, 28, 4, 128, 1296, 4113, 1296, 0, 0, 4, 0, 0, 0},
      {"diagnostics on", 1, 28, 4, 128, 1296, 4113, 64, 0, 0, 0, 1, 0, 0},
      {"tiny fp32 (8/2, D 64)", 1, 8, 2, 64, 576, 720, 28, 0, 1, 0, 0, 1, 16},
      {"fp32 caches, one CTA per kv-head (W 128 > 64)", 32, 28, 4, 128, 2304, 6500, 115, 0, 1, 0, 0, 2, 0},
      {"per-kv-head sets, B=3", 3, 28, 4, 128, 577, 700, 28, 1, 0, 0, 0, 1, 16},
      {"G = 16 (more than 8 heads per kv-head)", 2, 32, 2, 128, 1024, 3000, 51, 0, 0, 0, 0, 2, 0},
  };
  int bad = 0;
  for (const FormCase& c : cases) {
    StepParams p{};
    p.B = c.B; p.H = c.H; p.Hkv = c.Hkv; p.G = c.H / c.Hkv; p.D = c.D;
    p.max_visual = c.max_visual; p.max_seq = c.max_seq; p.granularity = c.gran; p.dtype = c.dtype;
    p.mode = c.mode;
    p.n_act = c.diag ? reinterpret_cast<int32_t*>(16) : nullptr;
    const Plan pl = make_plan(c.B, c.Hkv, c.D, 152, c.max_visual, c.max_seq, c.kept_cap, c.gran, false);
    p.cl = pl.cl; p.gslice = pl.gslice;
    const int kind = select_kind(p, c.kept_cap);
    const int w = kind == 1 ? selgat_slice_dims(p) : 0;
    if (kind != c.want_kind || w != c.want_w) {
      std::printf("FAIL select form of %s: kind %d (want %d), slice %d (want %d), cluster %d\n", c.name, kind,
                  c.want_kind, w, c.want_w, pl.cl);
      ++bad;
    }
  }
  return bad;
}

// Chunk-gather plans of the benchmarked sweep shapes (B = 64, 32/8 heads,
// D = 128, 1024 text tokens; fixed ratios 5% / 20% / 50% and top-p, whose
// cap is the whole span) and of the dense layers of the anchor pipeline: the
// GPU parity tests at these sizes run every combine form through them.
struct ChunkCase {
  const char* name;
  int B, Hkv, D, max_visual, max_seq, kept_cap, tc;
  int want_nk, want_nm, want_nc;
};

int check_chunks() {
  using namespace vp;
  const int T = 1024 + 18;
  const ChunkCase cases[] = {
      // name, B, Hkv, D, N_v, max_seq, kept_cap, tc, nk, nm, nc
      {"sweep N_v 576, 50% (one score split: text from its partial)", 64, 8, 128, 576, 576 + T, 288, 0, 1, 0, 1},
      {"sweep N_v 2304, 50%", 64, 8, 128, 2304, 2304 + T, 1152, 1, 1, 0, 1},
      {"sweep N_v 6400, 20%", 64, 8, 128, 6400, 6400 + T, 1280, 1, 1, 0, 1},
      {"sweep N_v 6400, 50% (two chunks, text from the split partial)", 64, 8, 128, 6400, 6400 + T, 3200, 1, 2, 0, 2},
      {"sweep N_v 16384, 5% (lone CTA, merged text slice)", 64, 8, 128, 16384, 16384 + T, 820, 1, 1, 1, 1},
      {"sweep N_v 16384, 20%", 64, 8, 128, 16384, 16384 + T, 3277, 1, 2, 2, 2},
      {"sweep N_v 16384, 50%", 64, 8, 128, 16384, 16384 + T, 8192, 1, 4, 4, 4},
      {"sweep N_v 16384, top-p (cap = span, chunk starts differ)", 64, 8, 128, 16384, 16384 + T, 16384, 1, 8, 8, 8},
      {"dense layer of the anchor pipeline, B = 1", 1, 4, 128, 1296, 4113, 1296, 0, 6, 4, 6},
  };
  int bad = 0;
  for (const ChunkCase& c : cases) {
    const Plan pl = make_plan(c.B, c.Hkv, c.D, 152, c.max_visual, c.max_seq, c.kept_cap, 0, c.tc != 0);
    if (pl.gslice || pl.nk != c.want_nk || pl.nm != c.want_nm || pl.nc != c.want_nc) {
      std::printf("FAIL chunk plan of %s: nk %d nm %d nc %d gslice %d (want %d %d %d 0)\n", c.name, pl.nk, pl.nm,
                  pl.nc, pl.gslice, c.want_nk, c.want_nm, c.want_nc);
      ++bad;
    }
  }
  return bad;
}

}  // namespace

int main() {
  using namespace vp;
  const int Bs[] = {1, 2, 3, 7, 8, 32, 64, 100, 256};
  const int Hkvs[] = {1, 2, 4, 8};
  const int Ds[] = {64, 128};
  const int SMs[] = {152, 148, 132, 1};
  const int MVs[] = {0, 1, 576, 2304, 16384, 32767};
  const int extra[] = {1, 513, 16384, 40000};
  long long plans = 0;
  for (int B : Bs)
    for (int Hkv : Hkvs)
      for (int D : Ds)
        for (int sms : SMs)
          for (int mv : MVs)
            for (int ex : extra) {
              const int ms = mv + ex, H = 7 * Hkv;
              const WsLayout ws = ws_layout(B, H, Hkv, D, mv, ms, sms);
              const int caps[] = {0, 1, 128, 129, 256, 257, 2048, 2049, mv, 100000};
              for (int cap : caps)
                for (int tc = 0; tc < 2; ++tc)
                  for (int gran = 0; gran < 2; ++gran) {
                    const Plan pl = make_plan(B, Hkv, D, sms, mv, ms, cap, gran, tc != 0);
                    ++plans;
                    const long long TR = tc ? kTcRows : 32;
                    long long w_max = tc ? (long long)kTcWt * ((ms + TR - 1) / TR) - (long long)(kTcWt - kTcWv) * (mv / TR)
                                         : 2LL * ((ms + TR - 1) / TR) - mv / TR;
                    if (w_max < 1) w_max = 1;
#define CHECK(cond) check((cond), #cond, B, Hkv, D, sms, mv, ms, cap, tc, gran)
                    CHECK(pl.ns >= 1 && pl.ns <= kNsMax);
                    CHECK(pl.split_w >= 1 && (long long)pl.ns * pl.split_w >= w_max);
                    CHECK(pl.ns <= ws.nsp_max);
                    CHECK(pl.nk >= 1 && pl.nk <= kNkMax && pl.nk <= ws.nk_max);
                    const int kmax = cap < mv ? cap : mv;
                    CHECK((kmax + pl.nk - 1) / pl.nk <= kGmMaxChunk);
                    CHECK((pl.ns == 1) == (pl.nm == 0));
                    CHECK(pl.nm == 0 || (pow2(pl.nm) && pl.nm <= D / 16 && pl.nm <= kMaxMerge && pl.nm <= pl.nk));
                    CHECK(pl.nc == (pl.nk > pl.nm ? pl.nk : pl.nm));
                    CHECK(!pl.gslice || cap <= kSliceMaxKept);
                    CHECK(pl.cl == 1 || pl.cl == 2 || pl.cl == 4 || pl.cl == 8);
                    if (tc && cap == 0 && gran == 0) {
                      // The tensor-core splits of sequences up to these shapes
                      // partition every sequence's tiles, each split within
                      // tc_max_split_tiles (the page-id staging bound).
                      const int nvs[] = {0, 1, mv / 3, mv};
                      for (int nv : nvs)
                        for (int vs : {0, 13, 128, 1000})
                          for (int tl : {1, 200, ms - nv}) {
                            if (tl < vs || tl < 1 || nv + tl > ms) continue;
                            const int NTl = (nv + tl + kTcRows - 1) / kTcRows;
                            int next = 0, total = 0;
                            for (int sp = 0; sp < pl.ns; ++sp) {
                              const TcRange r = tc_split(vs, nv, tl, sp, pl.ns, pl.split_w);
                              CHECK(r.n >= 0 && r.u0 == next);
                              CHECK(r.n <= tc_max_split_tiles(ms, pl.ns, pl.split_w));
                              next = r.u0 + r.n;
                              total += r.n;
                            }
                            CHECK(total == NTl);
                          }
                    }
#undef CHECK
                  }
            }
  std::printf("%lld plans, %d violations\n", plans, fails);
  fails += check_forms();
  fails += check_chunks();
  return fails ? 1 : 0;
}
