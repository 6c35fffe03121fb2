"""Writes tests/golden/small_linear.txt: a small y computed by the CPU oracle
(fp64, all digits via repr) on seeded inputs from workloads.  Calls only
oracle/ and the input generator; nothing from the CUDA library."""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
import workloads as wl  # noqa: E402


def main():
    N, K, M = 6, 384, 2
    w = wl.gen_weights(N, K, 0.25, config=8, proj=1)
    x = wl.gen_x(M, K, config=8, proj=1)
    rp, _ = oracle.rowptr(N, K, w.sal)
    p1, p2, st = oracle.pack(N, K, w.T1, w.T2, w.sal, rp)
    assert st == 0
    y, _ = oracle.linear(M, N, K, p1, p2, w.sal, w.s1, w.off, w.s2, x, nthreads=1)
    with open(os.path.join(HERE, "small_linear.txt"), "w") as f:
        f.write("# N K M, then y[m][n] (fp64 repr) from the CPU oracle; inputs: workloads.gen_weights(6, 384, 0.25, config=8, proj=1), gen_x(2, 384, config=8, proj=1)\n")
        f.write(f"{N} {K} {M}\n")
        for m in range(M):
            f.write(" ".join(repr(float(v)) for v in y[m]) + "\n")


if __name__ == "__main__":
    main()
