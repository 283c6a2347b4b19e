"""Writes the hand-derived fixtures in this folder.

Every expected value below is a closed form derived by hand (the derivation is
stored in each fixture); nothing here calls the oracle or the CUDA path.
Run:  python tests/golden/write_fixtures.py
"""
import json
import math
import os

HERE = os.path.dirname(os.path.abspath(__file__))

FIXTURES = {
    "attention_basis.json": {
        "cite": "Sec. 3.1: p_S / p_L are softmax attention; closed form for basis keys",
        "derivation": "d=4, scale=1/2. Keys e0,e1,e2; q = (2 ln 3) e0, so logits are (ln 3, 0, 0), "
                      "probabilities (3/5, 1/5, 1/5), lse = ln 5. V rows (1,0,0,0), (0,1,0,0), (1,1,0,2) give "
                      "o = 3/5 v0 + 1/5 v1 + 1/5 v2 = (0.8, 0.4, 0, 0.4).",
        "q": [2 * math.log(3), 0, 0, 0],
        "keys": [[1, 0, 0, 0], [0, 1, 0, 0], [0, 0, 1, 0]],
        "values": [[1, 0, 0, 0], [0, 1, 0, 0], [1, 1, 0, 2]],
        "scale": 0.5,
        "o": [0.8, 0.4, 0.0, 0.4],
        "lse": math.log(5),
    },
    "verify_causal.json": {
        "cite": "Algorithm 2, Verify: the block's queries see the full cache with a causal mask inside the block",
        "derivation": "t_ctx=2, n_q=2, one head, d=2 (scale 1/sqrt 2). Keys k0=k1=k3=(0,0), k2=(sqrt2 ln2, 0); "
                      "q=(1,0) for both block queries. Query 0 (position 2) sees keys 0..2 with logits (0,0,ln2): "
                      "p=(1/4,1/4,1/2), lse=ln4. Query 1 (position 3) sees keys 0..3 with logits (0,0,ln2,0): "
                      "p=(1/5,1/5,2/5,1/5), lse=ln5. V rows (1,0),(0,1),(2,2),(4,0): o0=(1.25,1.25), o1=(1.8,1.0).",
        "t_ctx": 2,
        "q": [[1, 0], [1, 0]],
        "keys": [[0, 0], [0, 0], [math.sqrt(2) * math.log(2), 0], [0, 0]],
        "values": [[1, 0], [0, 1], [2, 2], [4, 0]],
        "o": [[1.25, 1.25], [1.8, 1.0]],
        "lse": [math.log(4), math.log(5)],
    },
    "window_scores_uniform.json": {
        "cite": "Sec. 3.4: chunks scored by cumulative attention weight (window reading: causal rows over the "
                "last W positions)",
        "derivation": "t_ctx=3, W=2 (window rows at positions 1 and 2), one head, d=2, all keys zero. Row at "
                      "position 1 spreads 1/2 over keys 0,1; row at position 2 spreads 1/3 over keys 0,1,2. "
                      "lse=(ln2, ln3); score=(1/2+1/3, 1/2+1/3, 1/3).",
        "t_ctx": 3,
        "q_win": [[0.5, -1.0], [2.0, 0.25]],
        "keys": [[0, 0], [0, 0], [0, 0]],
        "lse": [math.log(2), math.log(3)],
        "score": [5 / 6, 5 / 6, 1 / 3],
    },
    "selection_example.json": {
        "cite": "Sec. 3.4 TopKChunks (top floor(B/s) by cumulative attention weight); token level with "
                "sink/recent as in the graded workloads",
        "derivation": "t_ctx=12, sink 2, recent 3, budget 8: middle = positions 2..8, 3 free slots. Middle scores "
                      "(.5,.7,.2,.7,.9,.1,.7) at positions 2..8. Best is position 6 (.9); positions 3, 5, 8 tie at "
                      ".7 and the lower two (3, 5) win. Keep = {0,1} + {3,5,6} + {9,10,11}. Chunk size 2: chunks "
                      "[2,4)=1.2, [4,6)=.9, [6,8)=1.0, [8,9)=.7; one chunk fits (3//2) -> [2,4): keep "
                      "{0,1,2,3,9,10,11}. Budget 12 >= t_ctx keeps all.",
        "t_ctx": 12, "n_sink": 2, "n_recent": 3,
        "score": [9, 9, 0.5, 0.7, 0.2, 0.7, 0.9, 0.1, 0.7, 5, 5, 5],
        "cases": [
            {"budget": 8, "chunk": 1, "keep": [0, 1, 3, 5, 6, 9, 10, 11]},
            {"budget": 8, "chunk": 2, "keep": [0, 1, 2, 3, 9, 10, 11]},
            {"budget": 12, "chunk": 1, "keep": list(range(12))},
        ],
    },
    "boundary_example.json": {
        "cite": "Sec. 3.4 TopKChunks (top floor(B/s) by cumulative attention weight), token level with sink/recent: "
                "the score of the last middle position the budget admits",
        "derivation": "t_ctx=10, sink 1, recent 2: middle = positions 1..7 with scores (.5,.9,.6,.7,.3,.55,.1); the "
                      "sink (10) and recent (8, 7) scores are larger and must not count. Middle scores in descending "
                      "order: .9,.7,.6,.55,.5,.3,.1. Budget 4 leaves 1 free slot -> tau = .9; budget 5, 2 slots -> "
                      ".7 (the first excluded score is .6); budget 6, 3 slots -> .6; budget 9, 6 slots -> .3. "
                      "Budget 3 = sink + recent and budget 2 leave no free slot, budgets 10 and 12 keep everything: "
                      "nothing is ranked (null).",
        "t_ctx": 10, "n_sink": 1, "n_recent": 2,
        "score": [10, 0.5, 0.9, 0.6, 0.7, 0.3, 0.55, 0.1, 8, 7],
        "cases": [
            {"budget": 4, "tau": 0.9}, {"budget": 5, "tau": 0.7}, {"budget": 6, "tau": 0.6},
            {"budget": 9, "tau": 0.3}, {"budget": 3, "tau": None}, {"budget": 2, "tau": None},
            {"budget": 10, "tau": None}, {"budget": 12, "tau": None},
        ],
    },
    "combine_two_halves.json": {
        "cite": "log-sum-exp merge of attention over disjoint key sets (split-K partials)",
        "derivation": "Part A: keys with logits (0, 0) -> lse_A = ln2, o_A = mean of (1,0),(0,1) = (.5,.5). "
                      "Part B: one key with logit ln2 -> lse_B = ln2, o_B = (3,1). Union: logits (0,0,ln2) -> "
                      "p=(1/4,1/4,1/2), o = (1/4 + 3/2, 1/4 + 1/2) = (1.75, .75), lse = ln4.",
        "o_part": [[[0.5, 0.5]], [[3.0, 1.0]]],
        "lse_part": [[math.log(2)], [math.log(2)]],
        "o": [[1.75, 0.75]],
        "lse": [math.log(4)],
    },
    "accept_examples.json": {
        "cite": "Eq. accept and Algorithm 2: accept the longest prefix on which drafter and verifier agree, "
                "then emit one verifier token",
        "derivation": "gamma = 4.  Row 0: drafts (7,3,9,2), verifier (7,3,9,2,5): all four agree -> k = 4, emit "
                      "(7,3,9,2,5).  Row 1: drafts (7,3,9,2), verifier (7,4,9,2,1): first mismatch at index 1 -> "
                      "k = 1, emit (7,4).  Row 2: verifier (1,...) disagrees at once -> k = 0, emit (1).  Row 3: a "
                      "later agreement after a mismatch does not count: drafts (5,6,7,8), verifier (5,0,7,8,9) -> "
                      "k = 1, emit (5,0).",
        "draft": [[7, 3, 9, 2], [7, 3, 9, 2], [7, 3, 9, 2], [5, 6, 7, 8]],
        "verify": [[7, 3, 9, 2, 5], [7, 4, 9, 2, 1], [1, 3, 9, 2, 0], [5, 0, 7, 8, 9]],
        "n_accept": [4, 1, 0, 1],
        "emit": [[7, 3, 9, 2, 5], [7, 4, -1, -1, -1], [1, -1, -1, -1, -1], [5, 0, -1, -1, -1]],
    },
    "argmax_ties.json": {
        "cite": "Eq. accept: arg max over the vocabulary (reading: ties to the lowest token id, NaN never chosen)",
        "derivation": "Row 0: maximum 2.5 first at id 1 (also at id 3) -> 1.  Row 1: NaN at id 0 is skipped, max 1.0 at "
                      "id 2 -> 2.  Row 2: all -inf -> the first id, 0.  Row 3: all NaN -> 0.  Row 4: a NaN "
                      "before -inf values is still skipped -> 1.  Row 5: -0 and +0 are equal -> the first, 1.",
        "logits": [[0.0, 2.5, -1.0, 2.5], ["nan", 0.5, 1.0, -3.0], ["-inf", "-inf", "-inf", "-inf"],
                   ["nan", "nan", "nan", "nan"], ["nan", "-inf", "-inf", "nan"], [-1.0, -0.0, 0.0, -2.0]],
        "argmax": [1, 2, 0, 0, 1, 1],
    },
}

if __name__ == "__main__":
    for name, obj in FIXTURES.items():
        with open(os.path.join(HERE, name), "w") as f:
            json.dump(obj, f, indent=1)
    print(f"wrote {len(FIXTURES)} fixtures")
