"""Write ``sampler_seed0.json``: the first outputs of the oracle's samplers for
the key of seed 0.  This file only calls ``oracle/``; it records the sampler
specification's behaviour so that an accidental change to the oracle's
sampler shows up as a test failure (self-consistency, not a paper pin).

Run from the repository root:  python tests/golden/make_sampler_golden.py
"""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402


def main():
    key = oracle.key_from_seed(0)
    out = {
        "spec": "ChaCha20 keystream words; nonce = (tag, idx_lo, idx_hi); see the oracle",
        "stream_words_tag1_idx0": [oracle.stream_word(key, 1, 0, i) for i in range(20)],
        "perm_tag1_N16": oracle.sample_permutation(key, 1, 0, 16).tolist(),
        "field_star_tag3_N8": oracle.sample_field_vector(key, 3, 0, 8, True).tolist(),
    }
    s, v = oracle.sample_sparse(key, oracle.TAG_MASK, 0, 2048, 12)
    out["sparse_mask_b0_N2048_t12"] = {"support": s.tolist(), "values": v.tolist()}
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "sampler_seed0.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
