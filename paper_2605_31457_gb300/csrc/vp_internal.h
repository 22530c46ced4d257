// Internal definitions shared by the host side (vp_api.cu) and the kernels
// (vp_kernels.cu) of libvp.  Not part of the public ABI.
#pragma once

#include <stdint.h>
#include <cuda_runtime.h>

namespace vp {

// Device error word bits (vp_check_errors reports them).
enum : unsigned {
  ERR_SPAN = 1u,       // vis_start / vis_len outside the live cache or max_visual
  ERR_TEXT = 2u,       // text_len < 1 (no current token)
  ERR_LEN = 4u,        // vis_len + text_len > max_seq
  ERR_PAGE = 8u,       // block-table entry outside [0, num_pages) or row past max_pages
  ERR_KEPT = 16u,      // a kept index outside [0, N_v)
  ERR_NONFINITE = 32u  // a non-finite score reached the selection
};

// Split statistics written by the score kernel for every (sequence, query
// head, split); maxima are in log2 units (z * log2 e).
enum { ST_MV = 0, ST_L1V, ST_LTV, ST_MT, ST_L1T, ST_LTT, ST_N };

struct KvView {
  const void* data;
  int64_t sb, sh, st;          // strides in elements
  const int32_t* block_table;  // paged only
  int32_t max_pages, num_pages;
};

struct StepParams {
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
  float* z_ws;        // [max_batch][H][max_visual] visual logits, log2 units
  float* split_st;    // [max_batch][H][ns_max][ST_N]
  float* split_o;     // [max_batch][H][ns_max][D]  text partial outputs
  float* gpart_o;     // [max_batch][Hkv][nk_max][G][D] kept-visual partial outputs
  float* gpart_st;    // [max_batch][Hkv][nk_max][G][2] {max, sum}
  unsigned* tickets;  // [max_batch][Hkv] (zero between calls)
  unsigned* err;      // device error word
  int ns, ns_max;     // score splits used by this call / allocated
  int nk, nk_max;     // gather chunks used by this call / allocated
};

// Launchers (vp_kernels.cu).  Return the launch error, if any.
cudaError_t launch_score(const StepParams& p, cudaStream_t s);
cudaError_t launch_select(const StepParams& p, cudaStream_t s);
cudaError_t launch_gather(const StepParams& p, cudaStream_t s);
cudaError_t configure_kernels(int max_visual);
// Raises (never lowers) the select kernel's dynamic shared-memory limit.
cudaError_t raise_select_smem(int max_visual);
size_t select_smem_bytes(int max_visual);

}  // namespace vp
