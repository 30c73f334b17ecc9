"""Error bars of the bf16 window attention against the fp64 oracle, derived
from the kernel's arithmetic (pure numpy; used by the GPU parity tests and
checked on the CPU by tests/test_parity_bars.py).

The kernel computes, per query row and split piece, p_j = 2^(s_j - m) in
fp32 against a running reference maximum m, rounds p_j to bf16 before the
P V product on the tensor cores, accumulates O and the row sum l (of the
unrounded p_j) in fp32, divides, merges split pieces by their log-sum-exp in
fp32 and rounds the output to bf16. With u = 2^-8 the bf16 unit roundoff,
P_j = p_j / l the probabilities and delta_j the rounding error of p_j
(|delta_j| <= u):

  o_gpu - o = sum_j P_j delta_j v_j  +  (output rounding, <= u |o|)
              + fp32 accumulation (<= (n/16 + 2) 2^-24 sum_j P_j |v_j|).

* Worst case (derived_bar): |err| <= (u + (n/16 + 2) 2^-24) sum_j P_j |v_j|
  + u |o| + 1e-6, with sum_j P_j |v_j| from the oracle run on |V|. It holds
  for any input and is tight when a few keys dominate (sharpened queries,
  outputs of order 1); it cannot see mistakes when the attention is diffuse
  (sum P |v| ~ 0.8 while |o| ~ 1/sqrt(n)).
* Random-walk (walk_bar): the delta_j are independent and bounded by u, so
  by Hoeffding's inequality P(|sum_j P_j delta_j v_j| > t) <= 2 exp(-t^2 /
  (2 u^2 sigma^2)) with sigma^2 = sum_j P_j^2 v_j^2, computed exactly per
  element from the oracle (sigma_walk). At a failure probability of 1e-9 per
  element, t = 6.54 u sigma, so
      |err| <= u |o| + 6.54 u sigma + 1e-5
  (1e-5 covers the fp32 sums, whose rounding errors also add up as a random
  walk). For diffuse attention sigma ~ rms(o), so the bar stays a few percent
  of the output where the absolute 1e-2 bound is as large as the output
  itself; a split-KV merge that drops a piece, drops its output or weights
  pieces equally exceeds it tens to hundreds of times.

sigma_walk: P_j^2 = softmax(2 s)_j exp(lse(2 s) - 2 lse(s)), so with the
oracle run once more on doubled scores and values v^2,
  sigma^2 = exp(lse2 - 2 lse) * sum_j softmax(2 s)_j v_j^2."""
import math

import numpy as np

U_BF16 = 2.0 ** -8
HOEFFDING = math.sqrt(2.0 * math.log(2.0 / 1e-9))   # 6.54


def walk_bar(o_ref: np.ndarray, sigma: np.ndarray) -> np.ndarray:
    """Per-element random-walk bar; o_ref and sigma of the same shape."""
    return U_BF16 * np.abs(o_ref) + HOEFFDING * U_BF16 * sigma + 1e-5


def sigma_walk(lse: np.ndarray, lse2: np.ndarray, out2: np.ndarray) -> np.ndarray:
    """sqrt(sum_j P_j^2 v_jd^2) from the oracle's (lse) on the scores and
    (out2, lse2) on doubled scores with squared values; lse, lse2 [..., rows],
    out2 [..., rows, D]."""
    return np.sqrt(np.exp(lse2 - 2.0 * lse)[..., None] * out2)


def derived_bar(o_ref: np.ndarray, sum_p_absv: np.ndarray, n_keys: int) -> np.ndarray:
    """Worst-case per-element bar: o_ref, sum_p_absv (= sum_j P_j |v_j|) of the
    same shape; n_keys the number of visible keys of the row (an upper bound)."""
    acc = (n_keys / 16.0 + 2.0) * 2.0 ** -24
    return (U_BF16 + acc) * sum_p_absv + U_BF16 * np.abs(o_ref) + 1e-6


def excess(err: np.ndarray, bar: np.ndarray) -> float:
    """Largest err / bar (<= 1 passes)."""
    return float(np.max(err / bar)) if err.size else 0.0
