"""Writes tests/golden/dither16.txt from the CPU oracle (and only from it).

Each line: seed step tid idx0 followed by the 16-bit dithers (hex) of elements
idx0, idx0+1, ... of that tensor. The file freezes the dither bits so that any
later change to the counter layout or the generator shows up as a failure.
Run:  python tests/golden/make_goldens.py
"""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle as O  # noqa: E402

CASES = [(0, 1, 0, 0), (0, 1, 1, 0), (1, 1, 0, 0), (0, 2, 0, 0), (42, 10, 3, 4096),
         (0xFFFFFFFFFFFFFFFF, 0xFFFFFFFF, 0xFFFFFFFF, 0), (0x123456789ABCDEF0, 7, 200, 2**31 - 4),
         (5, 100000, 17, 2**32 + 8), (5, 2**32 + 3, 17, 13), (7, 1, 400, 6_442_450_936),
         (99, 50, 2, 16_777_208), (12345, 3, 385, 1000), (3, 3, 3, 3), (2**63, 1, 0, 0),
         (1, 2**40, 1, 2**40), (8, 8, 8, 88888888)]


def main():
    path = os.path.join(HERE, "dither16.txt")
    with open(path, "w") as f:
        f.write("# seed step tid idx0 : 16-bit dithers (hex) of elements idx0..idx0+15\n")
        f.write("# written by tests/golden/make_goldens.py from the CPU oracle\n")
        for seed, step, tid, idx0 in CASES:
            vals = O.dither16(seed, step, tid, idx0, 16)
            f.write(f"{seed:#x} {step} {tid} {idx0} " + " ".join(f"{int(v):04x}" for v in vals) + "\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
