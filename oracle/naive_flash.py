"""Brute-force fp64 online-softmax recurrence.  TEST INFRASTRUCTURE ONLY (tiny inputs).

This is the second, independent oracle: the per-row streaming recurrence of the paper's
Algorithm "ggml-vec FlashAttention in llama.cpp" (Method section), in pure Python loops:

* for every query row: running maximum M = -inf, running sum Sum = 0, accumulator VKQ = 0;
* for every key: s = scale * (q . k); remember M_old = M; start from ms = vs = 1;
  if s is a new maximum (strict >), set M = s, ms = exp(M_old - M) and rescale VKQ by ms;
  otherwise vs = exp(s - M);
  then VKQ += vs * v and Sum = Sum * ms + vs;
* finally VKQ / Sum.

LSE (not in the paper) is read off the final state as M + ln(Sum).  The causal mask and the
GQA head mapping follow the same readings as ``fav_oracle.c``: bottom-right alignment and
kv head = h // (Hq // Hkv).  Shares no code with the two-pass oracle.
"""
import math


def naive_flash_row(q, keys, values, scale):
    """One query row against a list of (key, value) rows, following the recurrence."""
    D = len(q)
    M = -math.inf
    Sum = 0.0
    VKQ = [0.0] * len(values[0])
    for kr, vr in zip(keys, values):
        dot = 0.0
        for d in range(D):
            dot += q[d] * kr[d]
        S = dot * scale
        M_old = M
        ms = 1.0
        vs = 1.0
        if S > M:
            M = S
            ms = math.exp(M_old - M)
            for d in range(len(VKQ)):
                VKQ[d] = VKQ[d] * ms
        else:
            vs = math.exp(S - M)
        for d in range(len(VKQ)):
            VKQ[d] = VKQ[d] + vr[d] * vs
        Sum = Sum * ms + vs
    inv = 1.0 / Sum
    return [x * inv for x in VKQ], M + math.log(Sum)


def naive_flash(q, k, v, scale, causal=False):
    """q [B][Hq][Nq][D], k/v [B][Hkv][Nkv][D] as nested lists or numpy arrays.

    Returns (o, lse) as nested lists [B][Hq][Nq][D] and [B][Hq][Nq].
    """
    B = len(q)
    Hq = len(q[0])
    Nq = len(q[0][0])
    Hkv = len(k[0])
    Nkv = len(k[0][0])
    if Hq % Hkv != 0:
        raise ValueError("Hq must be a multiple of Hkv")
    if causal and Nq > Nkv:
        raise ValueError("causal attention needs Nq <= Nkv")
    G = Hq // Hkv
    o = []
    lse = []
    for b in range(B):
        ob, lb = [], []
        for h in range(Hq):
            g = h // G
            oh, lh = [], []
            for i in range(Nq):
                n = (Nkv - Nq + i + 1) if causal else Nkv
                keys = [[float(x) for x in k[b][g][j]] for j in range(n)]
                vals = [[float(x) for x in v[b][g][j]] for j in range(n)]
                qi = [float(x) for x in q[b][h][i]]
                orow, l = naive_flash_row(qi, keys, vals, float(scale))
                oh.append(orow)
                lh.append(l)
            ob.append(oh)
            lb.append(lh)
        o.append(ob)
        lse.append(lb)
    return o, lse
