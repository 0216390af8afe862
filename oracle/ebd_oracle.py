"""CPU oracle of one Early-Bird (EB) decoding step -- TEST INFRASTRUCTURE.

Only the tests, the smoke check and the benchmark's CPU-baseline /
reference arm may import this module.  The CUDA library never calls it, and
it shares no code with the CUDA path: it reads the same seeded inputs and
nothing else.

Everything is the plain definition, in float64, on bf16-decoded inputs:
  * window attention:   O = softmax(Q K^T / sqrt(D)) V, bidirectional, over the
    cached prefix followed by the window and, with a dual cache, by a cached
    suffix (Sec. 3: bidirectional mask predictor; Sec. 6.3 "Effect of
    KV-Cache Configuration": prefix and dual cache);
  * cache append:       the K/V of the rows committed in a step written into
    the cache at their positions (Sec. 6.3);
  * LM head:            full logits row l = W h, materialised;
  * vocabulary ranges:  the softmax state of a row over a range of the
    vocabulary and the merge of the ranges' states into the statistics (the
    vocabulary-parallel LM head);
  * statistics:         softmax in two passes (max, then sum), then
    kappa = max_v p(v)  (App. B, Eq. app-confidence), x_hat = argmax_v p(v),
    H~ = (-sum_v p log p) / log|V|  (Sec. 5.1), Delta = p(top1) - p(top2)
    (Sec. 5.2, "margin over the strongest competitor");
  * LBS router:         App. C.1 (Eq. lbs_feat and the encoder described
    there), by direct loops;
  * LBS filters:        App. E algorithm "Inference with LBS Block Selection and
    LPS Parallel Commit", block-selection branch (size fallback, router +
    EOS removal, MaxGapFilter, min-tokens fallback), Sec. 5.1;
  * LPS router:         App. D.1;
  * accept / commit:    the same App. E algorithm, union accept rule,
    anti-stall fallback, parallel commit, block resolution (Sec. 5.2).

Readings where the paper is silent or ambiguous (each is marked "Reading"
where it is used):
  R1  entropy in nats; H~ = H / ln V with V the full vocabulary.
  R2  argmax over the whole vocabulary; ties go to the lowest index.
  R3  Delta = p(top1) - p(top2); a duplicated maximum gives Delta = 0.
  R4  rho = |B n M| / |B| at the current step, before the commit.
  R5  pos = (i - b) / |B| with b = min B and |B| the size at selection, both
      frozen while the block is active; not clamped to [0, 1].
  R6  sigma(O) > 0.5 is evaluated as O > 0.
  R7  EOS removal applies to the router candidate set only.
  R8  gap = difference of absolute positions of consecutive candidates; the
      first candidate is always kept; at the first gap > g_max that candidate
      and all later ones are dropped (g_max = 1 then yields a contiguous block,
      as Sec. 6.4 states for the block-forward setting).
  R9  min-tokens fallback takes the first min(L_B, |M|) masked positions.
  R10 M is the set of masked rows of the current window (block-forward
      restriction, Sec. 6.4).
  R11 the LBS sequence is the masked rows compacted in ascending position,
      E_pos indexed by rank; zero padding to L is never attended to.
  R12 LBS encoder: post-norm layers, LayerNorm eps 1e-5, exact-erf GELU,
      scaled dot-product attention with scale 1/sqrt(d/heads), biases on
      every Linear, no final LayerNorm, dropout off.
  R13 LPS: feature order (kappa, H~, Delta, rho, pos); pre-norm blocks, no
      final LayerNorm; the sequence is the still-masked rows of B in
      ascending position; attention stays inside the block.
  R14 kappa >= tau is inclusive; p_psi > tau_psi is strict; the anti-stall
      fallback takes the lowest position among equal kappa.
  R15 a router that does not run leaves NaN in its per-row output.
  R21 dual cache: the keys right of the active block are those of the
      positions after the window; a step passes them as a range of cached
      positions [s0, s0 + S).  Appending on commit writes a row's K/V at
      its absolute position once its mask is 0 after the step; positions
      outside the cache are skipped.
  R20 the baselines' fixed-block rule (App. B, Eq. prelim-update) is read as
      two modes on the rows of the active fixed block: 'threshold' commits
      the masked rows with kappa >= tau, or, when none reaches tau, the one
      with the highest kappa (the anti-stall fallback of the App. E
      algorithm; Fast-dLLM's confidence rule); 'topm' commits the
      min(m, |M|) masked rows with the highest kappa (Top-m), ties to the
      lowest position.  The active block is the first block of B positions
      that still holds a masked position.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np
from scipy.special import erf

NEAR_TIE = 1e-3        # spec near-tie margin (logit gap, tau, tau_psi, O_phi)
NEAR_TIE_STALL = 1e-4  # margin on kappa for the anti-stall argmax
LN_EPS = 1e-5


# ----------------------------------------------------------------------------
# decoding of stored inputs
# ----------------------------------------------------------------------------
def bf16(u16) -> np.ndarray:
    """bf16 bits (uint16) -> float64 (exact)."""
    a = np.asarray(u16, dtype=np.uint16)
    return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# elementary layers (fp64)
# ----------------------------------------------------------------------------
def gelu(x):
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def layer_norm(x, g, b):
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS) * g + b


def linear(x, W, name):
    return x @ W[name + ".w"].T + W[name + ".b"]


def softmax_rows(s):
    m = s.max(axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / e.sum(axis=-1, keepdims=True)


def self_attention(x, W, name, n_heads):
    """Multi-head scaled dot-product self-attention over the rows of x."""
    n, d = x.shape
    dh = d // n_heads
    qkv = linear(x, W, name + ".qkv")
    q, k, v = qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]
    heads = []
    for h in range(n_heads):
        sl = slice(h * dh, (h + 1) * dh)
        a = softmax_rows(q[:, sl] @ k[:, sl].T / math.sqrt(dh))
        heads.append(a @ v[:, sl])
    return linear(np.concatenate(heads, axis=1), W, name + ".out")


def sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


# ----------------------------------------------------------------------------
# (1) window attention -- Sec. 3 (bidirectional), Sec. 6.3 (prefix cache)
# ----------------------------------------------------------------------------
def window_attention(q, k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix=None):
    """q[R][Hq][D], k_win/v_win[R][Hkv][D], k_cache/v_cache[B][P][Hkv][D]
    (bf16 bits) -> O[R][Hq][D] float64.  Sequence b's window queries attend,
    without any mask, to its first prefix_len[b] cached keys followed by its
    own window keys and, if suffix is given (dual cache, Reading R21), by
    the cached keys at positions [suffix[b][0], suffix[b][0] + suffix[b][1]).
    Query head h reads key/value head h // (Hq/Hkv)."""
    R, Hq, D = q.shape
    Hkv = k_win.shape[1]
    group = Hq // Hkv
    out = np.zeros((R, Hq, D))
    for b in range(len(prefix_len)):
        r0, r1 = int(cu_rows[b]), int(cu_rows[b + 1])
        if r1 == r0:
            continue
        P = int(prefix_len[b])
        s0, S = (int(suffix[b][0]), int(suffix[b][1])) if suffix is not None else (0, 0)
        for h in range(Hq):
            g = h // group
            K = np.concatenate([bf16(k_cache[b, :P, g]), bf16(k_win[r0:r1, g]),
                                bf16(k_cache[b, s0:s0 + S, g])])
            V = np.concatenate([bf16(v_cache[b, :P, g]), bf16(v_win[r0:r1, g]),
                                bf16(v_cache[b, s0:s0 + S, g])])
            Q = bf16(q[r0:r1, h])
            A = softmax_rows(Q @ K.T / math.sqrt(D))
            out[r0:r1, h] = A @ V
    return out


def kv_append(k_cache, v_cache, k_win, v_win, cu_rows, row_pos, mask):
    """Prefix-cache append on commit (Sec. 6.3; Reading R21): returns copies
    of the caches in which every window row r of sequence b with mask[r] == 0
    has its K/V (bit patterns) at position row_pos[r]; positions outside the
    cache are skipped."""
    kc, vc = np.array(k_cache, copy=True), np.array(v_cache, copy=True)
    Pm = kc.shape[1]
    for b in range(len(cu_rows) - 1):
        for r in range(int(cu_rows[b]), int(cu_rows[b + 1])):
            pos = int(row_pos[r])
            if mask[r] == 0 and 0 <= pos < Pm:
                kc[b, pos] = k_win[r]
                vc[b, pos] = v_win[r]
    return kc, vc


# ----------------------------------------------------------------------------
# (2) LM head and the per-position statistics -- App. B, Sec. 5.1, Sec. 5.2
# ----------------------------------------------------------------------------
def lm_logits(hidden, w_lm, chunk: int = 8192):
    """l[r][v] = sum_k h[r][k] W[v][k] in float64.  W is decoded a slab of
    vocabulary rows at a time only to bound memory; every logit is the same
    single dot product."""
    H = bf16(hidden)
    V = w_lm.shape[0]
    out = np.empty((H.shape[0], V))
    for v0 in range(0, V, chunk):
        out[:, v0:v0 + chunk] = H @ bf16(w_lm[v0:v0 + chunk]).T
    return out


@dataclass
class RowStats:
    conf: np.ndarray        # kappa
    entropy: np.ndarray     # H in nats
    ent_norm: np.ndarray    # H~
    gap: np.ndarray         # Delta
    argmax: np.ndarray      # x_hat
    logit_gap: np.ndarray   # l(top1) - l(top2)
    near_tie: np.ndarray    # logit_gap < NEAR_TIE


def softmax_stats(logits) -> RowStats:
    """Two-pass softmax over each full logits row, then the statistics by
    their definitions (Readings R1-R3)."""
    logits = np.atleast_2d(logits)
    n, V = logits.shape
    conf = np.empty(n); ent = np.empty(n); gap = np.empty(n)
    am = np.empty(n, dtype=np.int64); lg = np.empty(n)
    for r in range(n):
        l = logits[r]
        M = l.max()                              # pass 1
        e = np.exp(l - M)                        # pass 2
        p = e / e.sum()
        conf[r] = p.max()                        # kappa = max_v p(v)
        am[r] = int(np.argmax(p))                # first maximum = lowest index
        nz = p[p > 0]
        ent[r] = -(nz * np.log(nz)).sum()        # H = -sum p log p
        l2 = np.partition(l, V - 2)[V - 2] if V >= 2 else -np.inf
        p2 = math.exp(l2 - M) / e.sum() if V >= 2 else 0.0
        gap[r] = conf[r] - p2                    # Delta = p1 - p2
        lg[r] = M - l2
    ent_norm = ent / math.log(V)
    return RowStats(conf=conf, entropy=ent, ent_norm=ent_norm, gap=gap,
                    argmax=am, logit_gap=lg, near_tie=lg < NEAR_TIE)


# ----------------------------------------------------------------------------
# (2b) the statistics from vocabulary ranges (the vocabulary-parallel LM head)
# ----------------------------------------------------------------------------
@dataclass
class RangeState:
    """Softmax state of each row over a range of the vocabulary: m = max
    logit, S = sum exp(l - m), T = sum exp(l - m)(l - m), l2 = second largest
    logit (duplicates count; -inf for a one-entry range), idx = vocabulary
    index of the first maximum."""
    m: np.ndarray
    S: np.ndarray
    T: np.ndarray
    l2: np.ndarray
    idx: np.ndarray


def range_state(logits_range, v0: int) -> RangeState:
    """The state of each row over logits_range[:, j] = l[v0 + j], by its
    definition."""
    L = np.atleast_2d(np.asarray(logits_range, dtype=np.float64))
    n, w = L.shape
    m = L.max(axis=1)
    e = np.exp(L - m[:, None])
    S = e.sum(axis=1)
    T = (e * (L - m[:, None])).sum(axis=1)
    l2 = np.partition(L, w - 2, axis=1)[:, w - 2] if w >= 2 else np.full(n, -np.inf)
    idx = v0 + np.argmax(L, axis=1)
    return RangeState(m=m, S=S, T=T, l2=l2, idx=idx.astype(np.int64))


def merge_range_states(states: List[RangeState], V: int) -> RowStats:
    """The statistics of the whole vocabulary from the states of ranges that
    partition it: with the common maximum M = max_g m_g,
    S = sum_g S_g exp(m_g - M), T = sum_g exp(m_g - M)(T_g + (m_g - M) S_g)
    (each range's sums re-centred on M), kappa = 1/S, H = ln S - T/S,
    Delta = (1 - exp(l2 - M))/S with l2 the largest of the argmax range's l2
    and the other ranges' maxima, x_hat = the lowest index among the ranges
    whose maximum is M (Readings R1-R3)."""
    m = np.stack([s.m for s in states])          # G x n
    M = m.max(axis=0)
    w = np.exp(m - M)
    S = (np.stack([s.S for s in states]) * w).sum(axis=0)
    T = (w * (np.stack([s.T for s in states]) + (m - M) * np.stack([s.S for s in states]))).sum(axis=0)
    idx = np.where(m == M, np.stack([s.idx for s in states]), np.iinfo(np.int64).max).min(axis=0)
    n = len(M)
    l2 = np.empty(n)
    for r in range(n):
        win = [g for g in range(len(states)) if m[g, r] == M[r] and states[g].idx[r] == idx[r]][0]
        others = [m[g, r] for g in range(len(states)) if g != win]
        l2[r] = max([states[win].l2[r]] + others)
    conf = 1.0 / S
    ent = np.log(S) - T / S
    p2 = np.exp(l2 - M) / S
    return RowStats(conf=conf, entropy=ent, ent_norm=ent / math.log(V), gap=conf - p2,
                    argmax=idx, logit_gap=M - l2, near_tie=(M - l2) < NEAR_TIE)


# ----------------------------------------------------------------------------
# (3) LBS router -- Sec. 5.1 Eq. (2), App. C.1 Eq. lbs_feat
# ----------------------------------------------------------------------------
def lbs_router(ent_norm_seq, xhat_seq, w_emb, W) -> np.ndarray:
    """O_phi for the masked rows (ascending position, compacted; Reading R11).
    W maps parameter names to float64 arrays."""
    n = len(ent_norm_seq)
    if n == 0:
        return np.zeros(0)
    z = lbs_input(ent_norm_seq, xhat_seq, w_emb, W)
    for l in range(2):
        z = lbs_encoder_layer(z, W, f"lbs.l{l}")
    return linear(z, W, "lbs.head")[:, 0]


def lbs_input(ent_norm_seq, xhat_seq, w_emb, W):
    """Z_phi of Eq. lbs_feat (App. C.1) for the n masked rows:
    W_combine [F_ent(H~) ; W_tok W_e(x_hat)] + E_pos[:n]."""
    n = len(ent_norm_seq)
    Ht = np.asarray(ent_norm_seq, dtype=np.float64)[:, None]           # n x 1
    # entropy branch F_ent: Linear(1->64) -> GELU -> Linear(64->64) -> LN
    e = layer_norm(linear(gelu(linear(Ht, W, "lbs.ent1")), W, "lbs.ent2"),
                   W["lbs.ent_ln.g"], W["lbs.ent_ln.b"])
    # token branch: frozen embedding W_e[x_hat], projected by W_tok
    Ex = bf16(w_emb[np.asarray(xhat_seq, dtype=np.int64)])                # n x d_base
    t = linear(Ex, W, "lbs.tok")
    # fusion of [e ; t], then the learned positional embedding indexed by rank
    return linear(np.concatenate([e, t], axis=1), W, "lbs.comb") + W["lbs.pos"][:n]


def lbs_encoder_layer(z, W, p):
    """Post-norm Transformer encoder layer, d=128, 4 heads, FFN 256, GELU
    (App. C.1; Reading R12)."""
    z = layer_norm(z + self_attention(z, W, p, 4), W[p + ".ln1.g"], W[p + ".ln1.b"])
    f = linear(gelu(linear(z, W, p + ".ff1")), W, p + ".ff2")
    return layer_norm(z + f, W[p + ".ln2.g"], W[p + ".ln2.b"])


def max_gap_filter(cand_pos: List[int], g_max: int) -> List[int]:
    """Reading R8: from the leftmost candidate, drop the first candidate whose
    distance to its predecessor exceeds g_max, and all after it."""
    kept: List[int] = []
    for p in cand_pos:
        if kept and p - kept[-1] > g_max:
            break
        kept.append(p)
    return kept


# ----------------------------------------------------------------------------
# (4) LPS router -- Sec. 5.2, App. D.1
# ----------------------------------------------------------------------------
def lps_router(feats, W) -> np.ndarray:
    """O_psi for the still-masked rows of the block; feats[n][5] =
    (kappa, H~, Delta, rho, pos) (Reading R13)."""
    x = np.asarray(feats, dtype=np.float64)
    if x.shape[0] == 0:
        return np.zeros(0)
    z = lps_input(x, W)
    for l in range(2):
        z = lps_block(z, W, f"lps.l{l}")
    return linear(z, W, "lps.head")[:, 0]


def lps_input(x, W):
    """Z_psi (App. D.1): a linear projection of the 5 features to d = 32,
    then LayerNorm, then GELU."""
    return gelu(layer_norm(linear(x, W, "lps.in"), W["lps.in_ln.g"], W["lps.in_ln.b"]))


def lps_block(z, W, p):
    """Pre-norm Transformer block, d=32, 4 heads, FFN 64, GELU (App. D.1)."""
    z = z + self_attention(layer_norm(z, W[p + ".ln1.g"], W[p + ".ln1.b"]), W, p, 4)
    y = layer_norm(z, W[p + ".ln2.g"], W[p + ".ln2.b"])
    return z + linear(gelu(linear(y, W, p + ".ff1")), W, p + ".ff2")


# ----------------------------------------------------------------------------
# (5) the EB decision for one sequence -- App. E algorithm
# ----------------------------------------------------------------------------
@dataclass
class DecisionParams:
    tau: float
    tau_psi: float
    l_min: int
    l_b: int
    g_max: int
    eos_id: int
    lps_enabled: bool = True


@dataclass
class SeqDecision:
    lbs_logit: np.ndarray     # per window row (NaN where LBS did not run)
    lps_prob: np.ndarray      # per window row (NaN where LPS did not score)
    accepted: np.ndarray      # u8 per row
    lbs_ran: bool = False
    flag_lbs: bool = False    # a near-tie can change the selected block
    flag_accept: bool = False  # a near-tie can change the accepted set


def select_block(pos, M, O, argmax, prm: DecisionParams):
    """Block-selection branch of the App. E algorithm, run when no block is
    active.  M: masked rows (ascending position); O: router logits of those
    rows, or None when |M| <= L_min (the router is not needed then).
    Returns the selected rows B (ascending)."""
    if len(M) <= prm.l_min:                                   # size fallback
        return list(M)
    C = [i for j, i in enumerate(M)                           # router + EOS removal
         if O[j] > 0.0 and argmax[i] != prm.eos_id]           # R6, R7
    kept = set(max_gap_filter([int(pos[i]) for i in C], prm.g_max))
    B = [i for i in C if int(pos[i]) in kept]                 # MaxGapFilter (R8)
    if len(B) < prm.l_min:                                    # min-tokens fallback
        B = list(M[:min(prm.l_b, len(M))])                    # R9
    return B


def lps_features(pos, mask, in_block, meta, st: RowStats):
    """The LPS inputs of the active block (Sec. 5.2, App. E): the still-masked
    rows BM of B in ascending position, and per row i of BM the tuple
    (kappa_i, H~_i, Delta_i, rho, pos_i) with rho = |B n M| / |B| (Reading R4)
    and pos_i = (i - b) / |B| (Reading R5), b and |B| from meta."""
    BM = [i for i in range(len(pos)) if in_block[i] and mask[i]]
    size = int(meta[1])
    rho = len(BM) / size if BM else 0.0
    feats = [(st.conf[i], st.ent_norm[i], st.gap[i], rho,
              (int(pos[i]) - int(meta[0])) / size) for i in BM]
    return BM, feats


def decide_sequence(pos, mask, tokens, in_block, meta, st: RowStats,
                    w_emb, W, prm: DecisionParams, lbs_fn=None, lps_fn=None) -> SeqDecision:
    """One step of the App. E algorithm for one sequence, on its window rows.

    pos/mask/tokens/in_block are this sequence's rows (ascending position);
    meta = [b, |B|] (|B| = 0: no active block).  mask, tokens, in_block and
    meta are updated in place.  st holds the statistics of these rows.
    lbs_fn(ent_norm_seq, xhat_seq) replaces the LBS router and lps_fn(feats)
    the LPS router's logit O_psi (tests only)."""
    n = len(pos)
    out = SeqDecision(lbs_logit=np.full(n, np.nan), lps_prob=np.full(n, np.nan),
                      accepted=np.zeros(n, np.uint8))
    M = [i for i in range(n) if mask[i]]                      # masked set (R10)
    if meta[1] == 0:                                           # B = empty: LBS
        in_block[:] = 0
        O = None
        if len(M) > prm.l_min:
            router = lbs_fn or (lambda h, x: lbs_router(h, x, w_emb, W))
            O = np.asarray(router(st.ent_norm[M], st.argmax[M]), dtype=np.float64)
            out.lbs_ran = True
            out.lbs_logit[M] = O
            out.flag_lbs = bool(np.any(np.abs(O) < NEAR_TIE) or
                                np.any(st.near_tie[M]))
        B = select_block(pos, M, O, st.argmax, prm)
        if B:
            for i in B:
                in_block[i] = 1
            meta[0], meta[1] = int(pos[B[0]]), len(B)
    Bset = [i for i in range(n) if in_block[i]]
    size = int(meta[1])
    BM, feats = lps_features(pos, mask, in_block, meta, st)   # R4, R5, R13
    if BM:
        p_psi = None
        if prm.lps_enabled:
            router = lps_fn or (lambda f: lps_router(f, W))
            p_psi = sigmoid(np.asarray(router(feats), dtype=np.float64))
            out.lps_prob[BM] = p_psi
        A = [i for j, i in enumerate(BM)                       # union accept rule
             if st.conf[i] >= prm.tau or
             (p_psi is not None and p_psi[j] > prm.tau_psi)]   # R14
        flag = any(abs(st.conf[i] - prm.tau) < NEAR_TIE for i in BM)
        if p_psi is not None:
            flag |= bool(np.any(np.abs(p_psi - prm.tau_psi) < NEAR_TIE))
        if not A:                                              # anti-stall fallback
            best = max(BM, key=lambda i: (st.conf[i], -i))
            A = [best]
            ks = sorted((st.conf[i] for i in BM), reverse=True)
            flag |= len(ks) > 1 and ks[0] - ks[1] < NEAR_TIE_STALL
        flag |= bool(np.any(st.near_tie[A]))
        out.flag_accept = bool(flag or out.flag_lbs)
        for i in A:                                            # parallel commit
            tokens[i] = int(st.argmax[i])
            mask[i] = 0
            out.accepted[i] = 1
    if size > 0 and not any(mask[i] for i in Bset):            # block resolved
        in_block[:] = 0
        meta[0], meta[1] = 0, 0
    return out


# ----------------------------------------------------------------------------
# (5b) the fixed-block rules of the baselines -- App. B, Eq. prelim-update
# ----------------------------------------------------------------------------
def decide_fixed_block(mask, tokens, st: RowStats, mode: str, tau: float,
                       top_m: int) -> SeqDecision:
    """One step of the standard block update on the rows of the active fixed
    block (Reading R20).  mask and tokens are updated in place."""
    n = len(mask)
    out = SeqDecision(lbs_logit=np.full(n, np.nan), lps_prob=np.full(n, np.nan),
                      accepted=np.zeros(n, np.uint8))
    M = [i for i in range(n) if mask[i]]
    if not M:
        return out
    by_conf = sorted(M, key=lambda i: (-st.conf[i], i))      # highest kappa first
    if mode == "threshold":
        A = [i for i in M if st.conf[i] >= tau]
        flag = any(abs(st.conf[i] - tau) < NEAR_TIE for i in M)
        if not A:
            A = [by_conf[0]]
            ks = [st.conf[i] for i in by_conf]
            flag |= len(ks) > 1 and ks[0] - ks[1] < NEAR_TIE_STALL
    elif mode == "topm":
        k = min(top_m, len(M))
        A = by_conf[:k]
        ks = [st.conf[i] for i in by_conf]
        flag = k < len(ks) and ks[k - 1] - ks[k] < NEAR_TIE_STALL
    else:
        raise ValueError(mode)
    out.flag_accept = bool(flag or np.any(st.near_tie[A]))
    for i in A:
        tokens[i] = int(st.argmax[i])
        mask[i] = 0
        out.accepted[i] = 1
    return out


def fixed_block_window(mask, block: int):
    """First fixed block [jB, jB + B) that holds a masked position (Reading
    R20); (L, L) when none does."""
    L = len(mask)
    for j0 in range(0, L, block):
        if any(mask[j0:j0 + block]):
            return j0, min(j0 + block, L)
    return L, L


# ----------------------------------------------------------------------------
# (6) one whole step over a batch of windows
# ----------------------------------------------------------------------------
@dataclass
class StepResult:
    attn_out: np.ndarray
    stats: RowStats
    lbs_logit: np.ndarray
    lps_prob: np.ndarray
    accepted: np.ndarray
    tokens: np.ndarray
    mask: np.ndarray
    in_block: np.ndarray
    blk_meta: np.ndarray
    flag_lbs: np.ndarray       # per sequence
    flag_accept: np.ndarray    # per sequence
    lbs_ran: np.ndarray        # per sequence


def decide(cu_rows, row_pos, tokens, mask, in_block, blk_meta, st: RowStats,
           w_emb, W, prm: DecisionParams) -> StepResult:
    """Decision over a batch given per-row statistics (copies the state)."""
    R = int(cu_rows[-1]); B = len(cu_rows) - 1
    tokens = np.array(tokens, dtype=np.int32); mask = np.array(mask, dtype=np.uint8)
    in_block = np.array(in_block, dtype=np.uint8); blk_meta = np.array(blk_meta, dtype=np.int32)
    lbs = np.full(R, np.nan); lps = np.full(R, np.nan); acc = np.zeros(R, np.uint8)
    fl = np.zeros(B, bool); fa = np.zeros(B, bool); ran = np.zeros(B, bool)
    for b in range(B):
        r0, r1 = int(cu_rows[b]), int(cu_rows[b + 1])
        sub = RowStats(*(getattr(st, f)[r0:r1] for f in
                         ("conf", "entropy", "ent_norm", "gap", "argmax",
                          "logit_gap", "near_tie")))
        t, m, ib, meta = tokens[r0:r1], mask[r0:r1], in_block[r0:r1], blk_meta[b]
        d = decide_sequence(row_pos[r0:r1], m, t, ib, meta, sub, w_emb, W, prm)
        lbs[r0:r1] = d.lbs_logit; lps[r0:r1] = d.lps_prob; acc[r0:r1] = d.accepted
        fl[b], fa[b], ran[b] = d.flag_lbs, d.flag_accept, d.lbs_ran
    return StepResult(attn_out=None, stats=st, lbs_logit=lbs, lps_prob=lps,
                      accepted=acc, tokens=tokens, mask=mask, in_block=in_block,
                      blk_meta=blk_meta, flag_lbs=fl, flag_accept=fa, lbs_ran=ran)


def step(inp, W, prm: DecisionParams, rows: Optional[np.ndarray] = None,
         attention: bool = True, suffix=None) -> StepResult:
    """One EB decoding step (window attention, LM head + statistics, decision)
    on a synthetic StepInputs-like object `inp`; suffix: the dual cache's
    ranges (window_attention)."""
    attn = (window_attention(inp.q, inp.k_win, inp.v_win, inp.k_cache,
                             inp.v_cache, inp.cu_rows, inp.prefix_len, suffix)
            if attention else None)
    st = softmax_stats(lm_logits(inp.hidden, inp.w_lm))
    res = decide(inp.cu_rows, inp.row_pos, inp.tokens, inp.mask, inp.in_block,
                 inp.blk_meta, st, inp.w_emb, W, prm)
    res.attn_out = attn
    return res


def weights_f64(named_bf16: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    return {k: bf16(v) for k, v in named_bf16.items()}


# ----------------------------------------------------------------------------
# (7) the generation loop of the App. E algorithm in the window setting
# ----------------------------------------------------------------------------
def loop_window(frontier: int, end: int, meta, in_block_pos: List[int],
                max_window: int = 64):
    """Window rule of the loop workload: with no active block the window is
    [f, min(f + 64, end)); with an active block it is [f, max B + 1), where f
    is the first masked response position."""
    if meta[1] == 0:
        return frontier, min(frontier + max_window, end)
    return frontier, max(in_block_pos) + 1


def generation_loop(shape, W, prm: DecisionParams, window_inputs, kv_rows,
                    w_lm, w_emb, max_steps: Optional[int] = None,
                    attention: bool = False, on_step=None, mode: str = "eb",
                    block: int = 32, top_m: int = 1, cache: str = "prefix",
                    window: str = "block"):
    """Run the App. E loop on the synthetic loop workload: a committed prompt
    of `shape.prefix` positions followed by `shape.gen_len` masked positions.
    window_inputs(step, positions) -> (hidden, q, k_win, v_win) and
    kv_rows(positions) -> (k, v) supply the per-step tensors.  Returns
    (tokens, steps, per-step commit counts, per-step records).  mode 'eb'
    runs the App. E algorithm; 'threshold' and 'topm' the fixed-block rules
    of the baselines (Reading R20) with blocks of `block` positions.  cache
    'dual' adds the positions right of the window as cached keys (Reading
    R21).  window 'full': every step's window is the whole response (the
    full-sequence setting: M is every masked position)."""
    P0, L = shape.prefix, shape.gen_len
    tokens = np.full(L, -1, np.int32)
    mask = np.ones(L, np.uint8)
    in_block = np.zeros(L, np.uint8)
    meta = np.zeros(2, np.int32)
    steps, commits, records = 0, [], []
    while mask.any():
        if max_steps is not None and steps >= max_steps:
            break
        if window == "full":
            lo, hi = 0, L
        elif mode == "eb":
            f = int(np.argmax(mask))
            blk = [i for i in range(L) if in_block[i]]
            lo, hi = loop_window(f, L, meta, blk)
        else:
            lo, hi = fixed_block_window(mask, block)
        positions = P0 + np.arange(lo, hi, dtype=np.int32)
        hid, q, kw, vw = window_inputs(steps, positions)
        st = softmax_stats(lm_logits(hid, w_lm))
        attn = None
        if attention:
            dual = cache == "dual"
            kc, vc = kv_rows(np.arange(P0 + (L if dual else lo), dtype=np.int32))
            suffix = np.array([[P0 + hi, L - hi]]) if dual else None
            attn = window_attention(q, kw, vw, kc[None], vc[None],
                                    np.array([0, hi - lo]), np.array([P0 + lo]), suffix)
        t, m, ib = tokens[lo:hi], mask[lo:hi], in_block[lo:hi]
        before = int(m.sum())
        if mode == "eb":
            d = decide_sequence(positions, m, t, ib, meta, st, w_emb, W, prm)
        else:
            d = decide_fixed_block(m, t, st, mode, prm.tau, top_m)
        if meta[1] == 0:
            in_block[:] = 0
        commits.append(before - int(m.sum()))
        records.append(dict(step=steps, window=(lo, hi), accepted=d.accepted.copy(),
                            flag=d.flag_accept, flag_lbs=d.flag_lbs, lbs_ran=d.lbs_ran,
                            attn=attn, stats=st))
        if on_step is not None:
            on_step(steps, records[-1])
        steps += 1
    return tokens, steps, commits, records
