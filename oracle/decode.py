"""Oracle: Dynamic Contiguous Verification with draft-guided decoding (Algorithm 1).

Test infrastructure only (see ``oracle/__init__.py``).

One iteration (Sec. 3.3, "Inference with Drafts") does, in order:
  (i)   draft invalidation: x[p + i] <- MASK for i in [0, L)            (Eq. remasking)
  (ii)  one forward pass giving the top-1 id and confidence everywhere   (Eq. 2)
  (iii) K = sum_{i<L} prod_{j<=i} 1(c_{p+j} > tau_commit)               (Eq. compute_k)
  (iv)  commit x[p:p+K] <- x_hat[p:p+K]; for every i >= p + L,
        x_i <- x_hat_i if c_i > tau_draft (else keep)                    (Eq. draft_update)
  then p <- p + K; loop while p is inside the sequence                   (Algorithm 1)

Readings where the paper is silent or inconsistent (each one is also a test):
  * indices are absolute: the loop runs while p < N + M and drafts cover
    [p + L, N + M) (Algorithm 1 mixes a relative bound with an absolute p);
  * both thresholds are strict ``>`` (Eq. compute_k, Eq. draft_update and Algorithm 1;
    the prose of Sec. 3.2 says ``>=``);
  * the window is clipped to the sequence end: L' = min(L, N + M - p);
  * K = 0 would repeat the same deterministic state forever, so K is raised to
    ``min_commit`` (default 1; 0 keeps the literal rule, bounded by ``max_steps``);
  * p in the draft region is the window start of the current iteration, before the
    advance (the order of Algorithm 1);
  * drafts are refreshed at every future position, masked or already drafted;
  * decisions compare the confidence and the threshold as float32 values, the
    precision in which the CUDA kernel takes them;
  * ``confidence = 1`` replaces the top-1 probability by the marginal-entropy confidence
    c = exp(-H), H = -sum_v P(v) ln P(v) over the whole vocabulary (App. F.3 tries other
    confidence definitions; this one needs only the same single forward, and H is the
    per-token entropy of Eq. entropy_bound); exp(-H) <= sum_v P(v)^2 <= p1, so it never
    accepts a position the top-1 probability would reject;
  * every step records Eq. entropy_bound on the set it committed in parallel,
    sum_{i in U} H_i - max_{j in U} H_j with U = [p, p + K) and the step's own marginal
    entropies (0 when K = 1);
  * ``acceptance = 1`` replaces DCV by the non-contiguous rule DC-Leap is contrasted with
    (Eq. threshold_pd, Sec. 2.1 and Sec. 3.1): every masked position whose confidence
    exceeds tau_commit is committed at once, independently of its neighbours.  As the
    paper runs every method semi-autoregressively with block length 32 (Sec. 4.1), the
    rule applies to the masked positions of the current block [b0, b0 + Bk),
    b0 = N + Bk * floor((p - N) / Bk), with p the leftmost uncommitted position; there
    are no drafts and nothing to re-mask.  Eq. threshold_pd allows an empty set (the
    same stall as K = 0); when fewer than ``min_commit`` positions pass, the
    ``min_commit`` most confident masked positions of the block are committed instead
    (ties to the lower position).  With tau_commit >= 1 nothing passes, which is the
    low-confidence remasking of the base LLaDA sampler: ``min_commit`` tokens per step,
    the most confident first.  A committed position stays committed (an explicit flag:
    the committed token may itself be the MASK id, R8);
  * the approximate cache (``kv_cache = 1``; the paper pairs DC-Leap with a dLLM cache in
    Sec. 4 / Tab. 6 without describing its policy): per row, a step computes all
    positions at the first step and whenever the block-aligned prefix end
    N + Bk * floor((p - N) / Bk) changes, else only the positions from that prefix end on,
    attending to the keys and values the prefix had at its last refresh
    (``model.forward_rows``);
  * the dual cache (``kv_cache = 2``; a serving refinement, not in the paper): refreshes
    as above, and between refreshes only the positions of the current block
    [b0, min(b0 + Bk, T)) are computed, b0 that prefix end, their queries attending to the
    stored keys and values of every position (the block's fresh, the rest from the last
    refresh); the generation positions outside the block keep the predictions of the step
    that last computed them, K is capped at the block end (commits use fresh predictions
    only) and the drafts past p + L read the kept predictions.
"""
from __future__ import annotations

import dataclasses

import numpy as np


@dataclasses.dataclass
class DecodeConfig:
    tau_commit: float = 0.70      # Sec. 4.1 default
    tau_draft: float = 0.98       # Sec. 4.1 default
    max_window: int = 0           # L; 0 means gen_len // 2 (Sec. 4.1)
    block_len: int = 32           # semi-AR block (Sec. 4.1); sets the prefix-cache refresh
    gen_len: int = 0              # M
    min_commit: int = 1
    contiguous_drafts: bool = False  # App. E variant: drafts only as an unbroken chain
    kv_cache: int = 0             # 0: none; 1: prefix cache; 2: dual (prefix + suffix) cache
    confidence: int = 0           # 0: top-1 probability (Eq. threshold_pd); 1: exp(-entropy)
    acceptance: int = 0           # 0: DCV (Eq. compute_k); 1: Eq. threshold_pd in the block

    def window(self) -> int:
        return self.max_window if self.max_window > 0 else max(1, self.gen_len // 2)


def exceeds(c, tau) -> np.ndarray:
    """1(c > tau), taken in float32 (the precision of the CUDA decision)."""
    return np.asarray(c, dtype=np.float32) > np.float32(tau)


def window_length(c_window, tau_commit: float) -> int:
    """Eq. compute_k: K = sum_i prod_{j<=i} 1(c_j > tau_commit) over the given window."""
    ind = exceeds(c_window, tau_commit).astype(np.int64)
    return int(np.cumprod(ind).sum())


def remask(x: np.ndarray, p: int, window: int, mask_id: int) -> None:
    """Eq. remasking, clipped to the sequence end (in place on one row)."""
    x[p:min(p + window, x.shape[0])] = mask_id


def commit_and_draft(x: np.ndarray, p: int, ids: np.ndarray, c: np.ndarray,
                     cfg: DecodeConfig, window: int, k_max: int | None = None) -> int:
    """Steps (iii)-(iv) on one row; ids/c are indexed by absolute position.  Returns K.
    ``k_max`` (the dual cache between refreshes) caps K: commits stop at the block end."""
    T = x.shape[0]
    w_eff = min(window, T - p)
    K = window_length(c[p:p + w_eff], cfg.tau_commit)
    K = min(max(K, cfg.min_commit), w_eff)
    if k_max is not None:
        K = min(K, k_max)
    x[p:p + K] = ids[p:p + K]                                   # commit verified tokens
    lo = p + window                                             # future region i >= p + L
    if lo < T:
        ok = exceeds(c[lo:T], cfg.tau_draft)
        if cfg.contiguous_drafts:                               # App. E: unbroken chain only
            ok = np.cumprod(ok.astype(np.int64)).astype(bool)
        seg = x[lo:T]
        seg[ok] = ids[lo:T][ok]
    return K


def threshold_commit(x: np.ndarray, committed: np.ndarray, ids: np.ndarray, c: np.ndarray,
                     lo: int, hi: int, cfg: DecodeConfig) -> list:
    """Eq. threshold_pd on the uncommitted positions of [lo, hi) of one row (ids / c / x /
    committed indexed by absolute position): M_i = 1(c_i > tau_commit) for each one
    independently, and every position with M_i = 1 is committed in the same step.  When
    fewer than ``min_commit`` pass, the ``min_commit`` uncommitted positions of highest
    confidence are committed instead (float32 confidences, ties to the lower position);
    they include every passing one.  Returns the committed positions, in increasing order."""
    cand = [i for i in range(lo, hi) if not committed[i]]
    passing = [i for i in cand if exceeds(c[i], cfg.tau_commit)]
    if len(passing) >= cfg.min_commit:
        chosen = passing
    else:
        ranked = sorted(cand, key=lambda i: (-float(np.float32(c[i])), i))
        chosen = sorted(ranked[:cfg.min_commit])
    for i in chosen:
        x[i] = ids[i]
        committed[i] = True
    return chosen


def entropy_confidence(H) -> np.ndarray:
    """c = exp(-H) of the marginal entropy H (nats): 1 for a certain prediction, 1/V for a
    uniform one."""
    return np.exp(-np.asarray(H, dtype=np.float64))


def jpde_bound(H_set) -> float:
    """Eq. entropy_bound: sum_{i in U} H_i - max_{j in U} H_j for the marginal entropies of
    a set U of positions decoded in parallel (0 for fewer than two positions)."""
    H_set = np.asarray(H_set, dtype=np.float64)
    if H_set.size < 2:
        return 0.0
    return float(H_set.sum() - H_set.max())


def decision_confidence(p1, H, cfg: DecodeConfig) -> np.ndarray:
    """The c compared with the thresholds: p1, or exp(-H) with ``cfg.confidence = 1``."""
    if cfg.confidence == 0:
        return np.asarray(p1, dtype=np.float64)
    if cfg.confidence != 1:
        raise ValueError("confidence must be 0 (top-1 probability) or 1 (exp(-entropy))")
    if H is None:
        raise ValueError("the entropy confidence needs the marginal entropies")
    return entropy_confidence(H)


def prefix_end(p: int, n_prompt: int, block_len: int) -> int:
    """Block-aligned start of the current block: N + Bk * floor((p - N) / Bk)."""
    return n_prompt + block_len * ((p - n_prompt) // block_len)


def computed_range(p: int, n_prompt: int, T: int, cfg: DecodeConfig, refresh: bool) -> tuple:
    """Positions [start, end) a cached step computes (R18 / dual cache): everything at a
    refresh; else from the prefix end to T (prefix cache) or to the current block's end
    (dual cache)."""
    if refresh:
        return 0, T
    pe = prefix_end(p, n_prompt, cfg.block_len)
    return pe, (T if cfg.kv_cache == 1 else min(pe + cfg.block_len, T))


def generate(predict_fn, prompt: np.ndarray, cfg: DecodeConfig, mask_id: int,
             max_steps: int = 1 << 30, record: bool = True) -> dict:
    """Algorithm 1 for a batch of independent rows.

    predict_fn(tokens[T]) -> (ids[M], p1[M], p2[M]) or (ids, p1, p2, H[M]) for the
    generation positions (H, the marginal entropies, is needed by ``confidence = 1``).  With
    ``cfg.kv_cache = 1`` it is called as predict_fn(tokens[T], start, state): only positions
    >= start need be computed and ``state`` is the row's cache; start is 0 at the first
    step and whenever prefix_end(p) changes (a refresh), else prefix_end(p).  With
    ``cfg.kv_cache = 2`` it is called as predict_fn(tokens[T], start, state, end): only
    positions in [start, end) need be computed (end = T at a refresh, else the block end);
    the predictions of the other generation positions are kept from the step that last
    computed them.
    Returns the final x [B][T], per-row steps, the K of every step, the start and end of
    every step's computed positions (-1 for finished rows), Eq. entropy_bound of every
    step's committed set (NaN without entropies), and (if ``record``) the forward input of
    every step and the predictions it used (ids, p1, p2, H).
    """
    prompt = np.atleast_2d(np.asarray(prompt, dtype=np.int32))
    B, N = prompt.shape
    M = cfg.gen_len
    T = N + M
    L = cfg.window()
    if cfg.acceptance not in (0, 1):
        raise ValueError("acceptance must be 0 (DCV) or 1 (Eq. threshold_pd)")
    if cfg.acceptance == 1 and cfg.block_len < 1:
        raise ValueError("Eq. threshold_pd decoding needs a block length >= 1")
    if cfg.kv_cache not in (0, 1, 2):
        raise ValueError("kv_cache must be 0 (none), 1 (prefix) or 2 (dual)")
    if cfg.kv_cache == 2 and cfg.acceptance != 0:
        raise ValueError("the dual cache is defined for the DCV acceptance")
    x = np.full((B, T), mask_id, dtype=np.int32)
    x[:, :N] = prompt
    committed = np.zeros((B, T), dtype=bool)  # (Eq. threshold_pd only: commits out of order)
    committed[:, :N] = True
    p = np.full(B, N, dtype=np.int64)
    steps = np.zeros(B, dtype=np.int64)
    ks, starts, ends, inputs, preds, bounds = [], [], [], [], [], []
    caches = [{"pe": None} for _ in range(B)]
    n_iter = 0
    while (p < T).any() and n_iter < max_steps:
        k_step = np.zeros(B, dtype=np.int64)
        s_step = np.full(B, -1, dtype=np.int64)
        e_step = np.full(B, -1, dtype=np.int64)
        in_step = np.empty((B, T), dtype=np.int32)
        pr = np.zeros((4, B, M))
        pr[3] = np.nan
        jp = np.zeros(B)
        for b in range(B):
            if p[b] >= T:
                in_step[b] = x[b]
                continue
            if cfg.acceptance == 0:
                remask(x[b], int(p[b]), L, mask_id)              # (i)
            in_step[b] = x[b]
            k_max = None
            if cfg.kv_cache:                                     # (ii), approximate cache
                pe = prefix_end(int(p[b]), N, cfg.block_len)
                refresh = caches[b]["pe"] != pe
                s_step[b], e_step[b] = computed_range(int(p[b]), N, T, cfg, refresh)
                if cfg.kv_cache == 1:
                    out = predict_fn(x[b].copy(), int(s_step[b]), caches[b])
                else:                                            # dual: the block between refreshes
                    fresh = predict_fn(x[b].copy(), int(s_step[b]), caches[b], int(e_step[b]))
                    kept = caches[b].get("pred")
                    out = []
                    for f_arr, k_arr in zip(fresh, kept if kept is not None else fresh):
                        merged = np.array(k_arr, copy=True)
                        lo_g, hi_g = max(int(s_step[b]), N) - N, int(e_step[b]) - N
                        merged[lo_g:hi_g] = np.asarray(f_arr)[lo_g:hi_g]
                        out.append(merged)
                    caches[b]["pred"] = [a.copy() for a in out]
                    if not refresh:
                        k_max = int(e_step[b]) - int(p[b])
                caches[b]["pe"] = pe
            else:                                                # (ii)
                s_step[b] = 0
                e_step[b] = T
                out = predict_fn(x[b].copy())
            ids, p1, p2 = out[:3]
            H = out[3] if len(out) > 3 else None
            full_ids = np.zeros(T, dtype=np.int32)
            full_c = np.zeros(T, dtype=np.float64)
            full_ids[N:] = ids
            full_c[N:] = decision_confidence(p1, H, cfg)
            p0 = int(p[b])
            if cfg.acceptance == 0:
                k_step[b] = commit_and_draft(x[b], p0, full_ids, full_c, cfg, L, k_max)  # (iii)-(iv)
                jp[b] = np.nan if H is None else jpde_bound(np.asarray(H)[p0 - N:p0 - N + k_step[b]])
                p[b] += k_step[b]                                # dynamically advance
            else:                                                # Eq. threshold_pd in the block
                lo = prefix_end(p0, N, cfg.block_len)
                chosen = threshold_commit(x[b], committed[b], full_ids, full_c, lo,
                                          min(lo + cfg.block_len, T), cfg)
                k_step[b] = len(chosen)
                jp[b] = np.nan if H is None else jpde_bound(np.asarray(H)[np.asarray(chosen, int) - N])
                while p[b] < T and committed[b, p[b]]:           # leftmost uncommitted
                    p[b] += 1
            steps[b] += 1
            pr[0, b], pr[1, b], pr[2, b] = ids, p1, p2
            if H is not None:
                pr[3, b] = H
        ks.append(k_step)
        starts.append(s_step)
        ends.append(e_step)
        bounds.append(jp)
        if record:
            inputs.append(in_step)
            preds.append(pr)
        n_iter += 1
    return {"x": x, "p": p, "steps": steps, "k": np.array(ks), "start": np.array(starts), "end": np.array(ends),
            "jpde": np.array(bounds), "inputs": inputs,
            "preds": preds, "n_iter": n_iter, "done": bool((p >= T).all())}

