"""Writes worked_case.json: a compression step small enough to do by hand.

One recent query q = (2, 0, 0, 0) at position t, no rotation (theta = 0),
head_dim 4, so logit_j = q . k_j / sqrt(4) = k_j[0].  Keys have first
components 0, 1, 2, 0, -1, hence (Eq. 4) the softmax weights are
(1, e, e^2, 1, e^-1) / Z with Z = 2 + e + e^2 + e^-1, and with one query the
score (Eq. 6, max form) equals the weight.  With budget 3 and window 1 the
last key (index 4) is always kept and the two best candidates are keys 2 and
1, so the kept set (Algorithm 2) is [1, 2, 4].  Only the closed form above is
evaluated here (math.exp); no implementation is called.
"""
import json
import math
import os

k0 = [0.0, 1.0, 2.0, 0.0, -1.0]
z = sum(math.exp(x) for x in k0)
case = {
    "derivation": __doc__.strip(),
    "head_dim": 4,
    "t_pos": 4,
    "budget": 3,
    "window": 1,
    "q_recent": [2.0, 0.0, 0.0, 0.0],
    "K": [[x, y, -1.0, 0.5] for x, y in zip(k0, [0.0, 3.0, -1.0, 2.0, 1.0])],
    "score": [math.exp(x) / z for x in k0],
    "kept": [1, 2, 4],
}
with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "worked_case.json"), "w") as f:
    json.dump(case, f, indent=1)
