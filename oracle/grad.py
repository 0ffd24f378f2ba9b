"""fp64 oracle of the gradients of the read-out with hard decisions.

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle/``): plain numpy in fp64,
shares no code with the CUDA library.

With the boundary and merge decisions of a forward pass held fixed (they are
piecewise constant in k and v, so their derivative is zero almost everywhere),
the read-out of Eq. (capacity_bounded_output) is a weighted causal linear
attention.  Every state is a sum of token states (Sec. 2 recurrent form; a
merge of Algorithm 2 sums two adjacent states), so

    o_t = sum_i lambda_{t,i} S_i q_t = sum_{s <= t} lambda_{t, slot_t(s)} (k_s . q_t) v_s,

where slot_t(s) is the logical slot (0 = oldest) of the state holding token s
after token t.  With W[t, s] = lambda_{t, slot_t(s)} for s <= t (0 above the
diagonal), o = ((Q K^T) * W) V, and for a loss with dL/do = G:

    dQ = ((G V^T) * W) K          dK = ((G V^T) * W)^T Q
    dV = ((Q K^T) * W)^T G        dlambda_{t,i} = sum_{s <= t, slot_t(s) = i} (q_t . k_s)(g_t . v_s)

The slots come from replaying Algorithm 2's decisions (the boundary flags and
merge indices the forward pass reports) on token ranges: every state holds a
contiguous range of tokens, a boundary appends a new range, a merge at index j
joins ranges j and j + 1.
"""
from __future__ import annotations

import numpy as np


def token_slots(boundary, merge_log):
    """slot[t, s]: logical slot of the state holding token s after token t
    (s <= t), -1 for s > t.  boundary [T] (b_t, the first token of an empty
    cache counted as a boundary), merge_log [T] (i* of the merge at token t, or
    -1), as the forward pass reports them (Algorithm 2 replayed on token ranges)."""
    boundary = np.asarray(boundary)
    merge_log = np.asarray(merge_log)
    T = boundary.shape[0]
    firsts = []  # first token of each state, chronological (states are contiguous ranges)
    slot = np.full((T, T), -1, dtype=np.int64)
    for t in range(T):
        if boundary[t] or not firsts:
            j = int(merge_log[t])
            if j >= 0:  # states j and j + 1 become one: the later range joins the earlier
                del firsts[j + 1]
            firsts.append(t)
        # token s belongs to the last state whose first token is <= s
        slot[t, : t + 1] = np.searchsorted(np.asarray(firsts), np.arange(t + 1), side="right") - 1
    return slot


def weights(boundary, merge_log, lam):
    """W[t, s] = lambda_{t, slot_t(s)} for s <= t, else 0 (lam [T, C]; None = ones)."""
    slot = token_slots(boundary, merge_log)
    T = slot.shape[0]
    W = np.zeros((T, T))
    for t in range(T):
        sl = slot[t, : t + 1]
        W[t, : t + 1] = 1.0 if lam is None else np.asarray(lam, dtype=np.float64)[t, sl]
    return W


def readout_dense(q, k, v, W):
    """o = ((Q K^T) * W) V: the read-out as a weighted causal linear attention."""
    q, k, v = (np.asarray(x, dtype=np.float64) for x in (q, k, v))
    return ((q @ k.T) * W) @ v


def readout_grads(q, k, v, lam, boundary, merge_log, g):
    """Gradients of L = sum_t g_t . o_t with the decisions held fixed.
    Returns dict(dq, dk, dv, dlam); dlam is None when lam is None."""
    q, k, v, g = (np.asarray(x, dtype=np.float64) for x in (q, k, v, g))
    slot = token_slots(boundary, merge_log)
    W = weights(boundary, merge_log, lam)
    A = q @ k.T            # (q_t . k_s)
    Bg = g @ v.T           # (g_t . v_s)
    dq = (Bg * W) @ k
    dk = (Bg * W).T @ q
    dv = (A * W).T @ g
    dlam = None
    if lam is not None:
        lam = np.asarray(lam, dtype=np.float64)
        dlam = np.zeros_like(lam)
        P = A * Bg
        T = q.shape[0]
        for t in range(T):
            np.add.at(dlam[t], slot[t, : t + 1], P[t, : t + 1])
    return dict(dq=dq, dk=dk, dv=dv, dlam=dlam)


def readout_grads_sampled(q, k, v, lam, boundary, merge_log, g, rows, cols):
    """The gradients of readout_grads at sampled tokens only, for sequences
    too long for the T x T weight matrix: dq and dlambda at the tokens `rows`,
    dk and dv at the tokens `cols`.  The same replay of Algorithm 2's decisions
    on token ranges, evaluated one row (all s <= t) or one column (all t >= s)
    of the dense form at a time.  Returns dict(rows, cols, dq, dlam, dk, dv)."""
    q, k, v, g = (np.asarray(x, dtype=np.float64) for x in (q, k, v, g))
    boundary = np.asarray(boundary)
    merge_log = np.asarray(merge_log)
    lam = None if lam is None else np.asarray(lam, dtype=np.float64)
    T, d = k.shape
    rows = sorted(int(t) for t in rows)
    cols = sorted(int(s) for s in cols)
    row_set = set(rows)
    dq = np.zeros((len(rows), d))
    dlam = None if lam is None else np.zeros((len(rows), lam.shape[1]))
    col_slot = np.full((len(cols), T), -1, dtype=np.int64)  # slot_t(s) of every sampled column s
    cols_arr = np.asarray(cols, dtype=np.int64)
    firsts = []
    for t in range(T):
        if boundary[t] or not firsts:
            j = int(merge_log[t])
            if j >= 0:
                del firsts[j + 1]
            firsts.append(t)
        fa = np.asarray(firsts)
        live = cols_arr <= t
        if live.any():
            col_slot[live, t] = np.searchsorted(fa, cols_arr[live], side="right") - 1
        if t in row_set:
            r = rows.index(t)
            sl = np.searchsorted(fa, np.arange(t + 1), side="right") - 1
            w = np.ones(t + 1) if lam is None else lam[t, sl]
            bg = v[: t + 1] @ g[t]   # (g_t . v_s)
            a = k[: t + 1] @ q[t]    # (q_t . k_s)
            dq[r] = (bg * w) @ k[: t + 1]
            if lam is not None:
                np.add.at(dlam[r], sl, a * bg)
    dk = np.zeros((len(cols), d))
    dv = np.zeros((len(cols), d))
    for c, s in enumerate(cols):
        ts = np.arange(s, T)
        w = np.ones(T - s) if lam is None else lam[ts, col_slot[c, s:]]
        dk[c] = ((g[s:] @ v[s]) * w) @ q[s:]
        dv[c] = ((q[s:] @ k[s]) * w) @ g[s:]
    return dict(rows=rows, cols=cols, dq=dq, dlam=dlam, dk=dk, dv=dv)


def readout_grads_linear(q, k, v, lam, boundary, merge_log, g):
    """The gradients of readout_grads in time linear in T: two sweeps over the
    tokens with the cache's states, never the T x T weights.

    Forward sweep (the states S_i of Sec. 2, built as the forward pass builds
    them): dq_t = sum_i lambda_{t,i} S_i^T g_t and dlambda_{t,i} = g_t . (S_i q_t)
    over the cache after token t.

    Reverse sweep (adjoint states): token s receives, from every later token t
    whose state list holds s in slot i, the term lambda_{t,i} g_t q_t^T, so
    dv_s = M(s) k_s and dk_s = M(s)^T v_s with M(s) = sum_{t >= s}
    lambda_{t, slot_t(s)} g_t q_t^T.  Walking t from T - 1 down to 0 with one
    d x d matrix A_i per state of the cache after token t: every A_i takes
    lambda_{t,i} g_t q_t^T; token t, which lies in the newest state, reads
    M(t) = A_newest; then token t's events are undone in reverse order (the
    state it opened is dropped, a merge it caused is split and both halves keep
    the merged state's A, since later tokens saw them as one).
    Returns dict(dq, dk, dv, dlam) like readout_grads."""
    q, k, v, g = (np.asarray(x, dtype=np.float64) for x in (q, k, v, g))
    boundary = np.asarray(boundary)
    merge_log = np.asarray(merge_log)
    lamf = None if lam is None else np.asarray(lam, dtype=np.float64)
    T, d = k.shape
    dv_ = v.shape[1]

    def lam_at(t, i):
        return 1.0 if lamf is None else lamf[t, i]

    # forward sweep: states and the events of every token (for the reverse one)
    states = []   # S_i, [dv, d]
    firsts = []   # first token of each state
    events = []   # per token: (opened a state, merge index, first token of the state the merge removed)
    dq = np.zeros((T, d))
    dlam = None if lamf is None else np.zeros_like(lamf)
    for t in range(T):
        opened = bool(boundary[t]) or not states
        j, removed_first = -1, -1
        if opened:
            j = int(merge_log[t])
            if j >= 0:  # states j and j + 1 become one
                states[j] = states[j] + states[j + 1]
                removed_first = firsts[j + 1]
                del states[j + 1]
                del firsts[j + 1]
            states.append(np.outer(v[t], k[t]))
            firsts.append(t)
        else:
            states[-1] = states[-1] + np.outer(v[t], k[t])
        events.append((opened, j, removed_first))
        for i, S in enumerate(states):
            w = lam_at(t, i)
            dq[t] += w * (S.T @ g[t])
            if dlam is not None:
                dlam[t, i] = g[t] @ (S @ q[t])
    # reverse sweep: adjoint matrices of the states after token t
    A = [np.zeros((dv_, d)) for _ in states]
    dk = np.zeros((T, d))
    dvv = np.zeros((T, dv_))
    for t in range(T - 1, -1, -1):
        gq = np.outer(g[t], q[t])
        for i in range(len(A)):
            A[i] += lam_at(t, i) * gq
        M = A[-1]  # token t lies in the newest state
        dvv[t] = M @ k[t]
        dk[t] = M.T @ v[t]
        opened, j, removed_first = events[t]
        if opened:
            A.pop()
            firsts.pop()
            if j >= 0:  # undo the merge: both halves keep what later tokens gave the merged state
                A.insert(j + 1, A[j].copy())
                firsts.insert(j + 1, removed_first)
    return dict(dq=dq, dk=dk, dv=dvv, dlam=dlam)
