"""Write the oracle's regression fixtures under tests/golden/.

Calls only the input generator and the CPU oracle.  Run from the repository root:
    python tests/golden/make_golden.py
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from paper_2505_20438_gb300 import workload as wl  # noqa: E402


def tiny_step():
    """The tiny workload: 255 appends at slot positions 0..254 build the cache, then one
    macro-step appends slot 255 (rotating q at 255) and attends over the 256 slots."""
    w = wl.C0_TINY
    case = wl.make_case(w, num_slots=np.zeros(1, np.int32), extra_slots=256)
    oc = oracle.OracleCache.from_case(case)
    prefill = wl.make_case(w)                      # 255 slots of raw keys and values
    for n in range(w.slots):
        rc = oc.append(prefill.k[:, n], prefill.v[:, n], prefill.slot_ntok[:, n])
        assert rc == 0
    q = prefill.q.copy()
    assert oc.append(prefill.k_new, prefill.v_new, prefill.ntok_new, q_inout=q) == 0
    return oc.decode_attn(q), oc


def main():
    out, oc = tiny_step()
    path = os.path.join(HERE, "tiny_step_oracle.txt")
    with open(path, "w") as f:
        f.write("# oracle output of the tiny workload's decode step, [1][8][64] fp64, row-major\n")
        f.write("# written by tests/golden/make_golden.py (oracle + input generator only)\n")
        f.write(f"# num_slots {int(oc.num_slots[0])} num_tokens {int(oc.num_tokens[0])}\n")
        for x in out.reshape(-1):
            f.write(f"{x:.17g}\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
