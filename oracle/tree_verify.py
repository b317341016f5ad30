"""Tree-shaped speculative-decode verification attention (Sec. 5.3:
speculative decoding checks several draft tokens in one target-model pass)
-- test infrastructure only: the tests call it; the library never does.

A request has P context tokens in its paged cache and k draft tokens whose
K/V sit right after them (cache positions P .. P + k - 1).  The drafts form a
tree: parent[i] is the draft that draft i continues (-1: it continues the
context directly), listed parents first (parent[i] < i).  Draft i attends to
every context token and to the drafts on its own path back to the context,
itself included:

    visible(i) = {0 .. P-1} U {P + j : j = i or j an ancestor of i}
    o_i = sum_{t in visible(i)} softmax_t(scale * q_i . k_t) v_t

with the kv head of q head h = h // (Hq / Hkv).  A chain (parent[i] = i - 1)
is the causal suffix prefill; a star (every parent -1) is k independent
one-token decodes over the same context.  Computed in fp64 from bf16 bit
patterns, one (draft, head) at a time.

Parity pinned: the tests reduce a chain to the causal prefill oracle and a
star to one-token decodes (both the C oracle), check that relabelling the
drafts in another parents-first order permutes the outputs, and that a
draft's output ignores the K/V of drafts off its path.
"""

import numpy as np

from .oracle import bf16_to_f64


def ancestors(parent):
    """For each draft, the set of drafts on its path (itself included)."""
    parent = [int(p) for p in parent]
    paths = []
    for i, p in enumerate(parent):
        if not (-1 <= p < i):
            raise ValueError(f"draft {i}: parent {p} must be -1 or an earlier draft")
        paths.append(({i} | paths[p]) if p >= 0 else {i})
    return paths


def tree_verify_attention(q_bits, k_bits, v_bits, parent, scale):
    """q_bits [k][Hq][d]; k_bits, v_bits [P + k][Hkv][d] (context, then the
    drafts in order); parent [k].  Returns (out [k][Hq][d], lse [k][Hq])."""
    q = bf16_to_f64(q_bits)
    kk = bf16_to_f64(k_bits)
    vv = bf16_to_f64(v_bits)
    n_draft, Hq, d = q.shape
    L, Hkv, _ = kk.shape
    P = L - n_draft
    if P < 0 or Hq % Hkv:
        raise ValueError("bad shapes")
    g = Hq // Hkv
    paths = ancestors(parent)
    out = np.zeros((n_draft, Hq, d))
    lse = np.zeros((n_draft, Hq))
    for i in range(n_draft):
        keys = list(range(P)) + [P + j for j in sorted(paths[i])]
        for h in range(Hq):
            kh = h // g
            s = scale * (kk[keys, kh, :] @ q[i, h])
            m = s.max()
            wgt = np.exp(s - m)
            out[i, h] = (wgt @ vv[keys, kh, :]) / wgt.sum()
            lse[i, h] = m + np.log(wgt.sum())
    return out, lse
