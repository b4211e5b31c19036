"""Writes ``worked_examples.json``: hand-derived closed forms, no program under test.

The paper prints no numeric example of its attention, so these two cases are
worked out by hand from the visibility rule of Sec. 3.2 (a token sees its own
chunk and all earlier chunks) and the softmax-attention definition; each
expected value below is the closed form of that derivation.  Run from the repo
root:  python tests/golden/make_worked_examples.py
"""
import json
import math
import os

LN3 = math.log(3.0)
LN4 = math.log(4.0)

Q = [[1.0], [1.0]]
K = [[0.0], [LN3]]
V = [[1.0], [5.0]]
DO = [[1.0], [1.0]]

CASES = [
    {
        "name": "token_causal_two_tokens",
        "citation": "Sec. 3.2 block-causal self-attention with chunks of one token "
                    "(T=1): each token sees itself and all earlier tokens",
        "derivation": "d=1, scale=1, q=(1,1), k=(0,ln3), v=(1,5), dO=(1,1). "
                      "Row 0 sees key 0: s=0, LSE=0, O=1. Row 1 sees keys 0,1: "
                      "exp(s)=(1,3), LSE=ln4, P=(1/4,3/4), O=1/4+15/4=4. "
                      "dV=(1+1/4, 3/4). dP row1=(1,5), D=(1,4), dS row0=(0), "
                      "row1=(-3/4,3/4). dQ=(0, 3/4 ln3). dK=(0-3/4, 3/4).",
        "T": 1, "scale": 1.0, "q": Q, "k": K, "v": V, "do": DO,
        "o": [[1.0], [4.0]], "lse": [0.0, LN4],
        "p": [[1.0, 0.0], [0.25, 0.75]],
        "dq": [[0.0], [0.75 * LN3]], "dk": [[-0.75], [0.75]], "dv": [[1.25], [0.75]],
    },
    {
        "name": "one_chunk_two_tokens",
        "citation": "Sec. 3.2: tokens of the same chunk attend to each other "
                    "bidirectionally (T=2, one chunk)",
        "derivation": "same q,k,v,dO; one chunk of two tokens. Both rows see both "
                      "keys: P=(1/4,3/4), LSE=ln4, O=4. D=(4,4), dP=(1,5) per row, "
                      "dS=(-3/4,3/4) per row. dQ_i=3/4 ln3. dK=(-3/4*2, 3/4*2). "
                      "dV=(1/4*2, 3/4*2).",
        "T": 2, "scale": 1.0, "q": Q, "k": K, "v": V, "do": DO,
        "o": [[4.0], [4.0]], "lse": [LN4, LN4],
        "p": [[0.25, 0.75], [0.25, 0.75]],
        "dq": [[0.75 * LN3], [0.75 * LN3]], "dk": [[-1.5], [1.5]], "dv": [[0.5], [1.5]],
    },
]

if __name__ == "__main__":
    doc = {
        "about": "Hand-derived worked examples of block-causal attention (exact up "
                 "to fp64 rounding of ln 3 and ln 4).",
        "cases": CASES,
    }
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "worked_examples.json")
    with open(path, "w") as f:
        json.dump(doc, f, indent=1)
