"""A decode MoE layer small enough to evaluate by hand.

Experts are selection matrices scaled by powers of two, and the router logits
are exact dyadic numbers, so every output has a closed form:

  z[t, e]  = s_t * a_e + b_e                         (router logits, exact)
  masked   : expert 1 is pruned (Eq. 2) although it has the largest logit
  top-2    : t0 -> (0, 3), t1 -> (2, 3), t2 -> (0, 2) by the lowest-id tie-break
  gates    : softmax over the two selected logits (Sec. 3.1 renormalisation)
  g_i      = cg_e * x[sg(e, i)],  u_i = cu_e * x[su(e, i)]
  a_i      = SiLU(g_i) * u_i
  y_h      = cd_e * a[td(e, h)]
  out[t]   = sum_j gate_j * y^(e_j)
"""
import numpy as np
import torch

H, E, I, K, B = 128, 4, 64, 2, 3
RETAINED = np.array([0, 2, 3], np.int32)
S_TOK = [1.0, -1.0, 0.0]             # x[t, H-2]
A_EXP = [1.0, 0.0, -1.0, 0.25]       # Wr[e, H-2]
B_EXP = [0.5, 4.0, 0.5, 0.0]         # Wr[e, H-1], with x[t, H-1] = 1
CG = [2.0, 1.0, 0.5, 4.0]
CU = [0.5, 2.0, 1.0, 0.25]
CD = [0.25, 1.0, 0.5, 2.0]


def sg(e, i):
    return (5 * i + 11 * e + 1) % (H - 2)


def su(e, i):
    return (3 * i + 7 * e + 2) % (H - 2)


def td(e, h):
    return (13 * h + 5 * e) % I


def _bits(a):
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).contiguous().view(torch.int16).numpy().view(np.uint16)


def build_case():
    x = np.zeros((B, H), np.float32)
    for t in range(B):
        for h in range(H - 2):
            x[t, h] = (((7 * h + 3 * t) % 9) - 4) / 4.0
        x[t, H - 2] = S_TOK[t]
        x[t, H - 1] = 1.0
    wr = np.zeros((E, H), np.float32)
    wr[:, H - 2] = A_EXP
    wr[:, H - 1] = B_EXP
    gu = np.zeros((E, 2 * I, H), np.float32)
    dn = np.zeros((E, H, I), np.float32)
    for e in range(E):
        for i in range(I):
            gu[e, i, sg(e, i)] = CG[e]
            gu[e, I + i, su(e, i)] = CU[e]
        for h in range(H):
            dn[e, h, td(e, h)] = CD[e]
    z = np.array([[S_TOK[t] * A_EXP[e] + B_EXP[e] for e in range(E)] for t in range(B)])
    idx = np.array([[0, 3], [2, 3], [0, 2]], np.int32)
    gates = np.zeros((B, K))
    for t in range(B):
        w = np.exp(z[t, idx[t]] - z[t, idx[t][0]])
        gates[t] = w / w.sum()
    return {"x": _bits(x), "x_f": x, "router_w": wr, "retained": RETAINED,
            "w_gate_up": _bits(gu), "w_down": _bits(dn), "k": K,
            "expect_idx": idx, "expect_gates": gates}


def closed_form_out(case):
    x = case["x_f"].astype(np.float64)
    out = np.zeros((B, H))
    for t in range(B):
        for j in range(K):
            e = int(case["expect_idx"][t, j])
            a = np.empty(I)
            for i in range(I):
                g = CG[e] * x[t, sg(e, i)]
                u = CU[e] * x[t, su(e, i)]
                a[i] = g / (1.0 + np.exp(-g)) * u
            for h in range(H):
                out[t, h] += case["expect_gates"][t, j] * CD[e] * a[td(e, h)]
    return out
