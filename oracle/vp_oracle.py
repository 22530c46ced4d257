"""CPU oracle for one VisionPulse decode step (test infrastructure only).

This module is test infrastructure.  Only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py`` (its ``cpu_baseline`` leg and its ``--impl reference`` arm)
may import it.  The library path (``libvp.so`` and its Python binding) never
imports, links or runs anything here, and this module imports nothing from the
library: the two share no code.

What it computes, for one attention layer acting as the anchor layer l_a and
one decode step t (VisionPulse, Sec. 4.2-4.3 and Sec. 5.2):

  1. pre-softmax logits  Z_{t,h}(q_t, j) = scale * <q_h, k_j>     (Eq. 6's Z)
  2. attention probabilities at tau = 1 and at tau                  (Eq. 6)
     -- both normalised over EVERY cached token j (visual and text)
  3. per-head visual mass m_{t,h}, its head mean M_vis and the
     head-max M_vis,max                                             (Eq. 5, Sec. 4.3)
  4. the retention budget K_t = M_vis,max * N_v, clamped            (Eq. 7, Sec. 5.2)
  5. importance S_i = (1/H) sum_h A_{t,h}(q_t, v_i)                  (Eq. 2)
  6. X_v^t = Top-K_t(S)                                              (Eq. 3)
  7. attention of q_t over X_v^t plus all text tokens               (Sec. 4.2, Sec. 5.7)
  8. for a layer after the anchor: attention over all text tokens and
     the anchor's kept set, with no selection of its own         (Sec. 4.2, Sec. 5.1)
  9. the active visual token count N_act(delta) and the per-token
     activity flags behind persistent inactivity                   (Sec. 4.3, App. B)
 10. FastV prefill pruning before VisionPulse: the surviving visual tokens
     and the cache that holds only them                              (App., prefill pruning)

Everything is float64 computed from the exact input values (bf16 or fp32
inputs are widened without rounding).  There is no blocking, fusion or
reordering beyond the definitions above.

Readings of points the paper leaves open:
  * Eq. 2 uses the plain softmax (tau = 1); tau enters only the mass (Eq. 6).
  * H is the number of query heads; under grouped-query attention query head h
    reads kv-head h // G with G = H / Hkv.
  * The softmax normaliser of Eq. 6 runs over all cached tokens (visual, text
    and the current token); a visual-only normaliser would make the mass 1.
  * K_t = ceil(M_vis,max * N_v) with the product and the ceiling taken in
    float32 (the kernel's precision, since a float decides an integer here);
    clamp [K_lo, K_hi] with K_lo = ceil(r_lo N_v), K_hi = max(K_lo, floor(r_hi N_v)),
    ratios given in parts per million and multiplied in exact integers.
  * Top-K ranks S_i rounded to float32 (the kernel's precision); equal keys
    go to the lower visual index.  Indices are returned ascending and relative
    to the start of the visual span.
  * granularity 1 ("per kv-head") averages S over the G query heads of each
    kv-head only and keeps K_t (from the head-max over all H heads) per kv-head.
"""

from __future__ import annotations

import math

import numpy as np

# Budget modes (same numbering as the C header, restated here so that the
# oracle depends on nothing in the library).
ADAPTIVE = 0      # Eq. 7 with the clamp of Sec. 5.2
FIXED_RATIO = 1   # "FastV-VP (Fix Ratio)", Sec. 5.4 / Table 2
FIXED_K = 2       # constant Top-k budget, App. A.2
DENSE = 3         # keep every visual token (full budget)
TOP_P = 4         # Top-p budgeting, App. A.2: smallest top set with a share p of the scores

PPM = 1_000_000


def logits(q: np.ndarray, k: np.ndarray, scale: float) -> np.ndarray:
    """Pre-softmax attention logits Z_{t,h}(q_t, j) (the Z of Eq. 6, Sec. 4.3).

    q: [H, D] query of the current token, k: [Hkv, T, D] cached keys.
    Query head h reads kv-head h // G (grouped-query attention, G = H / Hkv).
    Returns z: [H, T], z[h, j] = scale * <q[h], k[h // G, j]>.
    """
    H = q.shape[0]
    Hkv = k.shape[0]
    G = H // Hkv
    z = np.empty((H, k.shape[1]), dtype=np.float64)
    for h in range(H):
        z[h] = scale * (k[h // G].astype(np.float64) @ q[h].astype(np.float64))
    return z


def softmax_tau(z: np.ndarray, tau: float) -> np.ndarray:
    """Temperature-scaled attention probabilities A^{(tau)} of Eq. 6 (Sec. 4.3).

    A^{(tau)}_{h}(j) = exp(Z_h(j) / tau) / sum_{j'} exp(Z_h(j') / tau), the sum
    running over every cached token j' of the row.  tau = 1 gives the plain
    attention probability A of Eq. 2.  The row maximum is subtracted first;
    this changes nothing mathematically.
    """
    m = z.max(axis=-1, keepdims=True)
    e = np.exp((z - m) / tau)
    return e / e.sum(axis=-1, keepdims=True)


def visual_mass(a_tau: np.ndarray, vis: np.ndarray):
    """Visual attention mass, Eq. 5 and the head-max variant of Sec. 4.3.

    a_tau: [H, T] probabilities, vis: boolean [T] marking the visual span.
    Returns (m [H], M_vis = mean_h m, M_vis,max = max_h m).  With no visual
    token every m is 0.
    """
    m = a_tau[:, vis].sum(axis=1) if vis.any() else np.zeros(a_tau.shape[0])
    return m, float(m.mean()), float(m.max())


def _ceil_div(a: int, b: int) -> int:
    return -((-a) // b)


def budget_bounds(n_v: int, r_lo_ppm: int, r_hi_ppm: int):
    """Clamp range of Sec. 5.2, "(0.01N, 0.05N)" read as [K_lo, K_hi].

    K_lo = ceil(r_lo * N_v), K_hi = max(K_lo, floor(r_hi * N_v)), with the
    ratios in parts per million and the products in exact integers.
    """
    k_lo = _ceil_div(r_lo_ppm * n_v, PPM)
    k_hi = max(k_lo, (r_hi_ppm * n_v) // PPM)
    return k_lo, k_hi


def budget(m_max: float, n_v: int, mode: int = ADAPTIVE, r_lo_ppm: int = 10_000,
           r_hi_ppm: int = 50_000, ratio_ppm: int = 0, fixed_k: int = 0) -> int:
    """Step-wise retention budget K_t.

    ADAPTIVE    : K_t = M_vis,max * N_v (Eq. 7), rounded up, clamped to
                  [K_lo, K_hi] (Sec. 5.2).  The float32 product and ceiling
                  mirror the precision in which the kernel takes the decision.
    FIXED_RATIO : K_t = ceil(r * N_v), at least 1 ("Fix Ratio", Table 2).
    FIXED_K     : K_t = min(k, N_v) (Top-k budgeting, App. A.2).
    DENSE       : K_t = N_v.
    N_v = 0 gives K_t = 0 in every mode.
    """
    if n_v <= 0:
        return 0
    if mode == DENSE:
        return n_v
    if mode == FIXED_K:
        return max(0, min(int(fixed_k), n_v))
    if mode == FIXED_RATIO:
        return min(max(_ceil_div(ratio_ppm * n_v, PPM), 1), n_v)
    if mode != ADAPTIVE:
        raise ValueError(f"unknown budget mode {mode}")
    prod = np.float32(m_max) * np.float32(n_v)          # float32 product
    raw = int(math.ceil(float(prod)))
    k_lo, k_hi = budget_bounds(n_v, r_lo_ppm, r_hi_ppm)
    return min(max(raw, k_lo), k_hi, n_v)


def top_p_budget(s: np.ndarray, ratio_ppm: int) -> int:
    """Top-p budget of App. A.2 (studied with p = 0.10).  The paper does not
    say over which set the probabilities are normalised; read here as the
    importance scores of the visual span: K_t is the smallest k whose k
    largest scores (ranked as in Eq. 3, float32-rounded, ties to the lower
    index) sum to at least p times the sum of all visual scores.  p is given
    in parts per million; p <= 0 keeps nothing, p >= 1 keeps every token.
    """
    n = len(s)
    if n == 0 or ratio_ppm <= 0:
        return 0
    if ratio_ppm >= PPM:
        return n
    s32 = np.asarray(s, dtype=np.float32)
    order = np.lexsort((np.arange(n), -s32.astype(np.float64)))
    c = np.cumsum(s32[order].astype(np.float64))
    target = (ratio_ppm / PPM) * c[-1]
    return min(int(np.searchsorted(c, target, side="left")) + 1, n)


def importance(a: np.ndarray, vis: np.ndarray, heads=None) -> np.ndarray:
    """Importance score of Eq. 2: S_i = (1/H) sum_h A_h(q_t, v_i) over visual i.

    a: [H, T] plain (tau = 1) probabilities.  ``heads`` restricts the average
    to a subset of query heads (the per-kv-head reading); None = all H heads.
    """
    rows = a if heads is None else a[list(heads)]
    return rows[:, vis].mean(axis=0)


def select_topk(s: np.ndarray, k: int) -> np.ndarray:
    """X_v^t = Top-K_t(S), Eq. 3.  Largest scores first, ties to the lower index.

    Scores are ranked as float32 values (the precision the kernel decides in).
    Returns the kept visual indices in ascending order.
    """
    key = np.asarray(s, dtype=np.float32)
    order = sorted(range(len(key)), key=lambda i: (-float(key[i]), i))
    return np.array(sorted(order[:k]), dtype=np.int64)


def pruned_attention(z: np.ndarray, v: np.ndarray, keep: np.ndarray) -> np.ndarray:
    """Attention output over the kept tokens only (Sec. 4.2; the "dynamic
    visual sparse attention" of Sec. 5.7).

    z: [H, T] logits, v: [Hkv, T, D] values, keep: boolean [T] (kept visual
    tokens plus every text token).  Dropped tokens are excluded from the
    softmax, not given weight zero inside a larger normaliser:
        out_h = sum_{j in keep} exp(z_hj) v_j / sum_{j in keep} exp(z_hj).
    """
    H = z.shape[0]
    G = H // v.shape[0]
    out = np.empty((H, v.shape[2]), dtype=np.float64)
    for h in range(H):
        zk = z[h, keep]
        w = np.exp(zk - zk.max())
        out[h] = (w @ v[h // G][keep].astype(np.float64)) / w.sum()
    return out


def decode_step(q, k, v, vis_start: int, vis_len: int, text_len: int, *,
                mode: int = ADAPTIVE, tau: float = 0.1, scale: float = 0.0,
                r_lo_ppm: int = 10_000, r_hi_ppm: int = 50_000, ratio_ppm: int = 0,
                fixed_k: int = 0, granularity: int = 0, force_k=None) -> dict:
    """One VisionPulse decode step for one sequence at the anchor layer.

    q: [H, D]; k, v: [Hkv, >=T, D] with T = vis_len + text_len live tokens.
    Visual tokens occupy [vis_start, vis_start + vis_len); every other live
    token (prompt, generated reasoning, current token) is text.
    ``force_k`` overrides the budget (used by tests to re-select with the
    other side's K_t near an integer boundary).

    Returns a dict with
      out [H, D] float64, k_t int, kept list of index arrays (one per sequence
      for granularity 0, one per kv-head for granularity 1), mass [H]
      (tau-mass per head), mass_stats [M_vis(tau), M_vis,max(tau),
      M_vis(tau=1), K_t], z [H, T], s (importance, [N_v] or [Hkv, N_v]).
    """
    q = np.asarray(q, dtype=np.float64)
    H, D = q.shape
    Hkv = k.shape[0]
    G = H // Hkv
    T = vis_len + text_len
    if text_len < 1:
        raise ValueError("text_len must count at least the current token")
    if not (0 <= vis_start <= text_len):
        raise ValueError("visual span must lie inside the live cache")
    if scale == 0.0:
        scale = 1.0 / math.sqrt(D)
    k = np.asarray(k[:, :T], dtype=np.float64)
    v = np.asarray(v[:, :T], dtype=np.float64)
    vis = np.zeros(T, dtype=bool)
    vis[vis_start:vis_start + vis_len] = True

    z = logits(q, k, scale)                                  # Eq. 6's Z
    a1 = softmax_tau(z, 1.0)                                 # Eq. 2's A
    a_tau = softmax_tau(z, tau)                              # Eq. 6
    mass, m_mean, m_max = visual_mass(a_tau, vis)            # Eq. 5 + head-max
    _, m_mean1, _ = visual_mass(a1, vis)
    if mode == TOP_P:
        if granularity != 0:
            raise ValueError("the top-p budget is defined for one kept set per sequence")
        k_t = top_p_budget(importance(a1, vis), ratio_ppm)
    else:
        k_t = budget(m_max, vis_len, mode, r_lo_ppm, r_hi_ppm, ratio_ppm, fixed_k)
    if force_k is not None:
        k_t = int(force_k)

    if granularity == 0:
        s = importance(a1, vis)                              # Eq. 2
        kept = [select_topk(s, k_t)]                         # Eq. 3
        out = _attend(z, v, vis_start, vis, kept, G, per_head=False)
    else:
        s = np.stack([importance(a1, vis, range(g * G, (g + 1) * G)) for g in range(Hkv)])
        kept = [select_topk(s[g], k_t) for g in range(Hkv)]
        out = _attend(z, v, vis_start, vis, kept, G, per_head=True)

    return dict(out=out, k_t=k_t, kept=kept, mass=mass,
                mass_stats=np.array([m_mean, m_max, m_mean1, float(k_t)]),
                z=z, s=s)


def _attend(z, v, vis_start, vis, kept, G, per_head):
    """Pruned attention with the kept set(s); text tokens are always kept."""
    H = z.shape[0]
    out = np.empty((H, v.shape[2]), dtype=np.float64)
    for h in range(H):
        sel = kept[h // G] if per_head else kept[0]
        keep = ~vis
        keep[vis_start + sel] = True
        out[h] = pruned_attention(z[h:h + 1], v[h // G:h // G + 1], keep)[0]
    return out



def anchor_attention(q, k, v, vis_start: int, vis_len: int, text_len: int, kept, *,
                     scale: float = 0.0) -> np.ndarray:
    """Decode attention of a layer after the anchor layer (Sec. 4.2: the
    importance scores are computed at l_a and pruning starts from l_a; Sec.
    5.1 prunes at l_a = 17): the query attends to every text token and to the
    visual tokens of the anchor's kept set X_v^t only, with no budget or
    selection of its own.

    q: [H, D]; k, v: [Hkv, >=T, D]; kept: a list holding one array of visual
    indices (relative to the span) shared by all heads, or one per kv-head.
    Returns out [H, D] float64.
    """
    q = np.asarray(q, dtype=np.float64)
    H, D = q.shape
    Hkv = k.shape[0]
    G = H // Hkv
    T = vis_len + text_len
    if text_len < 1:
        raise ValueError("text_len must count at least the current token")
    if scale == 0.0:
        scale = 1.0 / math.sqrt(D)
    z = logits(q, np.asarray(k[:, :T], dtype=np.float64), scale)
    vis = np.zeros(T, dtype=bool)
    vis[vis_start:vis_start + vis_len] = True
    kept = [np.asarray(s, dtype=np.int64) for s in kept]
    return _attend(z, np.asarray(v[:, :T], dtype=np.float64), vis_start, vis, kept, G, per_head=len(kept) > 1)


def active_count(s: np.ndarray, delta: float):
    """Active visual token count of Sec. 4.3 (the equation defining
    N_act^t(delta)): how many visual tokens have a head-averaged attention
    probability (the S of Eq. 2) above delta, and which ones.  Scores and the
    threshold are compared in float32, the precision the kernel decides in.
    A token whose flag stays False at every step of a decode is persistently
    inactive (App. B, "Persistent visual redundancy during reasoning").

    s: [N_v] importance scores (or [Hkv, N_v] for per-kv-head selection).
    Returns (N_act, boolean activity flags of the same shape as s).
    """
    active = np.asarray(s, dtype=np.float32) > np.float32(delta)
    return active.sum(axis=-1), active


def fastv_survivors(q_last, k, vis_start: int, vis_len: int, text_len: int, ratio_ppm: int = 500_000, *,
                    scale: float = 0.0) -> np.ndarray:
    """FastV's prefill-stage selection (the appendix "Complementarity with
    Prefill Pruning": compression ratio 0.5, then VisionPulse decodes over
    the rest).  FastV ranks visual tokens by the attention they receive from
    the last prompt token at the pruning layer, averaged over heads -- the S
    of Eq. 2 with that token as the query (Sec. 4.2 follows FastV's estimator
    at every step) -- and keeps the top ratio, at least one token.

    q_last: [H, D] query of the last prompt token; k: [Hkv, T, D].
    Returns the kept visual indices, ascending, relative to vis_start.
    """
    q_last = np.asarray(q_last, dtype=np.float64)
    H, D = q_last.shape
    T = vis_len + text_len
    if scale == 0.0:
        scale = 1.0 / math.sqrt(D)
    z = logits(q_last, np.asarray(k[:, :T], dtype=np.float64), scale)
    vis = np.zeros(T, dtype=bool)
    vis[vis_start:vis_start + vis_len] = True
    s = importance(softmax_tau(z, 1.0), vis)
    n_keep = budget(0.0, vis_len, mode=FIXED_RATIO, ratio_ppm=ratio_ppm)
    return select_topk(s, n_keep)


def compact_cache(x, vis_start: int, vis_len: int, text_len: int, kept) -> np.ndarray:
    """The cache of one sequence after prefill pruning: the rows before the
    visual span, the surviving visual rows in ascending order, then the rows
    after the span.  x: [Hkv, T, D] with T >= vis_len + text_len.
    Returns [Hkv, len(kept) + text_len, D]."""
    x = np.asarray(x)
    kept = np.asarray(kept, dtype=np.int64)
    T = vis_len + text_len
    rows = np.concatenate([np.arange(vis_start), vis_start + kept, np.arange(vis_start + vis_len, T)])
    return x[:, rows]
