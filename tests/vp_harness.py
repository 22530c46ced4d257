"""Parity harness: runs the CUDA path through the C ABI and the CPU oracle on
the same seeded inputs and compares them element by element.

Tolerances (GPU vs oracle):
  * outputs and masses: max abs 2e-2 for bf16 caches, 1e-5 for fp32 caches;
  * K_t exact, except when the oracle's M_vis,max * N_v lies within 1e-4
    (relative) of an integer, where float32 and float64 may round to
    neighbouring ceilings; then K_t may differ by one and the oracle
    re-selects with the GPU's K_t;
  * kept sets identical except for indices whose oracle score lies within
    1e-3 (relative) of the K-th largest score; the output is then compared
    with the oracle's attention over the GPU's kept set.
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np
import torch

from oracle import vp_oracle as O
from paper_2605_31457_gb300 import workloads as W

TOL = {W.BF16: 2e-2, W.FP32: 1e-5}
K_NEAR_INT = 1e-4
TIE_REL = 1e-3


@dataclass
class Inputs:
    """One layer's inputs on the host (exact cache-dtype values) and device."""
    recipe: W.Recipe
    q: torch.Tensor          # [B, H, D] cache dtype (CPU)
    k: torch.Tensor          # [B, Hkv, Tcap, D] cache dtype (CPU, logical order)
    v: torch.Tensor
    vis_start: np.ndarray
    vis_len: np.ndarray
    text_len: np.ndarray
    block_table: np.ndarray | None = None
    n_pages: int = 0


def make_inputs(r: W.Recipe, layer=0, step=0, t_cap=None, q_override=None) -> Inputs:
    t_cap = r.capacity(step + 1) if t_cap is None else t_cap
    li = W.make_layer(r, layer, t_cap=t_cap)
    q = W.make_queries(r, layer, li, steps=step + 1)[step] if q_override is None else q_override
    inp = Inputs(r, W.round_to(q, r.dtype), W.round_to(li.k, r.dtype), W.round_to(li.v, r.dtype),
                 r.vis_starts.copy(), r.vis_lens.copy(), r.text_lens + step)
    if r.paged:
        inp.block_table, inp.n_pages, _ = W.page_table(r.batch, t_cap, r.page_size, r.seed)
    return inp


LAYOUTS = ("bhtd", "bthd", "tbhd", "padded")


def place(x: torch.Tensor, layout: str, dev) -> torch.Tensor:
    """Device copy of a [B, Hkv, T, D] (or paged [P, Hkv, S, D]) cache viewed in
    that logical order, with memory laid out as ``layout`` says:
      bhtd    sequence, head, token, dim (dense);
      bthd    sequence, token, head, dim (heads interleaved per token);
      tbhd    token outermost (a layout the tensor-map path declines);
      padded  bhtd with every row padded by 16 bytes."""
    if layout == "bhtd":
        return x.to(dev)
    if layout == "bthd":
        return x.permute(0, 2, 1, 3).contiguous().to(dev).permute(0, 2, 1, 3)
    if layout == "tbhd":
        return x.permute(2, 0, 1, 3).contiguous().to(dev).permute(1, 2, 0, 3)
    if layout == "padded":
        pad = 16 // x.element_size()
        y = torch.full((*x.shape[:3], x.shape[3] + pad), float("nan"), dtype=x.dtype)
        y[..., : x.shape[3]] = x
        return y.to(dev)[..., : x.shape[3]]
    raise ValueError(layout)


class Device:
    """Device copies of an Inputs plus a library context and output buffers."""

    def __init__(self, vp, inp: Inputs, budget: dict, max_batch=None, max_seq=None, layout="bhtd",
                 score_path=None):
        self.vp = vp
        r = inp.recipe
        dev = torch.device("cuda")
        self.inp = inp
        self.B, self.H, self.Hkv, self.D = r.batch, r.heads, r.kv_heads, r.head_dim
        dtype = vp.VP_BF16 if r.dtype == W.BF16 else vp.VP_FP32
        max_visual = int(max(inp.vis_len.max(), 1))
        max_seq = max_seq or int((inp.vis_len + inp.text_len).max())
        self.cfg = vp.make_config(max_batch or r.batch, r.heads, r.kv_heads, r.head_dim, max_visual,
                                  max(max_seq, max_visual + 1), dtype, int(r.paged), r.page_size)
        self.ctx = vp.vp_init(self.cfg)
        if score_path is not None:
            vp.vp_set_score_path(self.ctx, score_path)
        self.q = inp.q.to(dev)
        if r.paged:
            pk = W.scatter_pages(inp.k, inp.block_table, inp.n_pages, r.page_size)
            pv = W.scatter_pages(inp.v, inp.block_table, inp.n_pages, r.page_size)
            self.k_t, self.v_t = place(pk, layout, dev), place(pv, layout, dev)
            self.bt = torch.from_numpy(inp.block_table).to(dev)
            self.kc, self.vc = vp.kv_paged(self.k_t, self.bt), vp.kv_paged(self.v_t, self.bt)
        else:
            self.k_t, self.v_t = place(inp.k, layout, dev), place(inp.v, layout, dev)
            self.kc, self.vc = vp.kv_contiguous(self.k_t), vp.kv_contiguous(self.v_t)
        self.vs = torch.from_numpy(inp.vis_start.astype(np.int32)).to(dev)
        self.vl = torch.from_numpy(inp.vis_len.astype(np.int32)).to(dev)
        self.tl = torch.from_numpy(inp.text_len.astype(np.int32)).to(dev)
        self.span = vp.span(self.vs, self.vl)
        self.set_budget(budget)

    def set_budget(self, budget: dict):
        vp = self.vp
        self.budget_dict = dict(budget)
        self.budget = vp.make_budget(**budget)
        self.kept_cap = max(1, vp.vp_max_kept(self.budget, self.cfg.max_visual))
        nsel = self.Hkv if budget.get("granularity", 0) else 1
        dev = torch.device("cuda")
        self.out = torch.empty((self.B, self.H, self.D), dtype=self.q.dtype, device=dev)
        self.kept = torch.empty((self.B, nsel, self.kept_cap), dtype=torch.int32, device=dev)
        self.count = torch.empty((self.B, nsel), dtype=torch.int32, device=dev)
        self.mass = torch.empty((self.B, self.H), dtype=torch.float32, device=dev)
        self.stats = torch.empty((self.B, 4), dtype=torch.float32, device=dev)

    def run(self, check_errors=True):
        vp = self.vp
        vp.vp_decode_step(self.ctx, self.B, self.q, self.kc, self.vc, self.span, self.tl, self.budget,
                          self.out, self.kept, self.kept_cap, self.count, self.mass, self.stats)
        if check_errors:
            vp.vp_check_errors(self.ctx)
        torch.cuda.synchronize()
        return dict(out=self.out.float().cpu().numpy(), kept=self.kept.cpu().numpy(),
                    count=self.count.cpu().numpy(), mass=self.mass.cpu().numpy(),
                    stats=self.stats.cpu().numpy())

    def close(self):
        self.vp.vp_free(self.ctx)
        self.ctx = None


def oracle_seq(inp: Inputs, b: int, budget: dict, force_k=None):
    bd = {k: v for k, v in budget.items()}
    return O.decode_step(inp.q[b].double().numpy(), inp.k[b].double().numpy(), inp.v[b].double().numpy(),
                         int(inp.vis_start[b]), int(inp.vis_len[b]), int(inp.text_len[b]),
                         force_k=force_k, **bd)


def _near_integer(x):
    return abs(x - round(x)) <= K_NEAR_INT * max(1.0, abs(x))


TOP_P_REL = 1e-4


def _top_p_ambiguous(s, ratio_ppm, k):
    """Whether float32 sums in another order could make k the top-p budget:
    the k largest scores reach the target and the k - 1 largest fall short,
    both within TOP_P_REL of it."""
    s32 = np.sort(np.asarray(s, dtype=np.float32).astype(np.float64))[::-1]
    c = np.cumsum(s32)
    target = ratio_ppm / 1e6 * c[-1]
    ok_hi = c[k - 1] >= target * (1 - TOP_P_REL) if k >= 1 else target <= 0
    ok_lo = k == 1 or c[k - 2] < target * (1 + TOP_P_REL)
    return bool(ok_hi and ok_lo)


def compare_seq(inp: Inputs, gpu: dict, b: int, budget: dict, report: dict | None = None):
    """Asserts parity of sequence b; returns the oracle result used."""
    r = inp.recipe
    tol = TOL[r.dtype]
    ref = oracle_seq(inp, b, budget)
    nv = int(inp.vis_len[b])
    gran = budget.get("granularity", 0)
    k_gpu = int(gpu["count"][b][0])
    for c in gpu["count"][b]:
        assert int(c) == k_gpu, "per-kv-head counts must share K_t"
    if k_gpu != ref["k_t"]:
        if budget.get("mode", 0) == O.TOP_P:
            assert _top_p_ambiguous(ref["s"], budget["ratio_ppm"], k_gpu), \
                f"seq {b}: top-p K_t gpu {k_gpu} vs oracle {ref['k_t']}"
        else:
            raw = ref["mass_stats"][1] * nv
            assert budget.get("mode", 0) == O.ADAPTIVE and _near_integer(raw) and abs(k_gpu - ref["k_t"]) == 1, \
                f"seq {b}: K_t gpu {k_gpu} vs oracle {ref['k_t']} (M_max*N_v = {raw!r})"
        ref = oracle_seq(inp, b, budget, force_k=k_gpu)
    # masses
    np.testing.assert_allclose(gpu["mass"][b], ref["mass"], rtol=0, atol=tol, err_msg=f"mass seq {b}")
    np.testing.assert_allclose(gpu["stats"][b][:3], ref["mass_stats"][:3], rtol=0, atol=tol,
                               err_msg=f"mass_stats seq {b}")
    assert gpu["stats"][b][3] == float(k_gpu)
    # kept sets
    kept_sets = []
    sets = ref["kept"]
    scores = ref["s"] if gran else [ref["s"]]
    for gsel, want in enumerate(sets):
        got = gpu["kept"][b][gsel]
        assert np.all(got[k_gpu:] == -1), f"seq {b}: slots past K_t must be -1"
        got = got[:k_gpu]
        assert np.all(np.diff(got) > 0), f"seq {b}: kept indices must be strictly ascending"
        assert got.size == 0 or (got.min() >= 0 and got.max() < nv)
        diff = set(got.tolist()) ^ set(want.tolist())
        if diff:
            s = scores[gsel]
            theta = np.sort(s)[::-1][k_gpu - 1]
            outside = [i for i in diff if abs(s[i] - theta) > TIE_REL * theta]
            assert not outside, f"seq {b}: kept sets differ outside the tie zone at {sorted(outside)[:10]}"
            if report is not None:
                report["tie_mismatch"] = report.get("tie_mismatch", 0) + len(diff)
        kept_sets.append(got)
    # output, against the oracle's attention over the GPU's kept set
    z = ref["z"]
    vis_start = int(inp.vis_start[b])
    T = nv + int(inp.text_len[b])
    v = inp.v[b, :, :T].double().numpy()
    G = r.heads // r.kv_heads
    want = np.empty_like(ref["out"])
    for h in range(r.heads):
        sel = kept_sets[h // G] if gran else kept_sets[0]
        keep = np.ones(T, dtype=bool)
        keep[vis_start:vis_start + nv] = False
        keep[vis_start + sel] = True
        want[h] = O.pruned_attention(z[h:h + 1], v[h // G:h // G + 1], keep)[0]
    np.testing.assert_allclose(gpu["out"][b], want, rtol=0, atol=tol, err_msg=f"out seq {b}")
    if report is not None:
        report["max_out_err"] = max(report.get("max_out_err", 0.0), float(np.abs(gpu["out"][b] - want).max()))
        report["max_mass_err"] = max(report.get("max_mass_err", 0.0),
                                     float(np.abs(gpu["mass"][b] - ref["mass"]).max()))
    return ref


def check_all(vp, inp: Inputs, budget: dict, seqs=None, report=None, layout="bhtd", score_path=None):
    dev = Device(vp, inp, budget, layout=layout, score_path=score_path)
    try:
        gpu = dev.run()
    finally:
        dev.close()
    for b in (range(inp.recipe.batch) if seqs is None else seqs):
        compare_seq(inp, gpu, b, budget, report)
    return gpu
