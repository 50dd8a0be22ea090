"""Runs Triton's own Philox (tl.philox, CPU interpreter) and prints its words as JSON.

Used by test_oracle_philox.py in a subprocess, because the interpreter switch has
to be set before triton is imported.  Input on argv: JSON list of
[seed, c0, c1, c2, c3] rows.
"""
import json
import os
import sys

os.environ["TRITON_INTERPRET"] = "1"

import torch  # noqa: E402
import triton  # noqa: E402
import triton.language as tl  # noqa: E402


@triton.jit
def _philox_kernel(c_ptr, out_ptr, seed, BLOCK: tl.constexpr):
    offs = tl.arange(0, BLOCK)
    c0 = tl.load(c_ptr + offs * 4 + 0).to(tl.uint32)
    c1 = tl.load(c_ptr + offs * 4 + 1).to(tl.uint32)
    c2 = tl.load(c_ptr + offs * 4 + 2).to(tl.uint32)
    c3 = tl.load(c_ptr + offs * 4 + 3).to(tl.uint32)
    a, b, c, d = tl.philox(seed, c0, c1, c2, c3, 10)
    tl.store(out_ptr + offs * 4 + 0, a.to(tl.int64))
    tl.store(out_ptr + offs * 4 + 1, b.to(tl.int64))
    tl.store(out_ptr + offs * 4 + 2, c.to(tl.int64))
    tl.store(out_ptr + offs * 4 + 3, d.to(tl.int64))


def main():
    rows = json.loads(sys.argv[1])
    res = []
    for seed, *ctr in rows:
        c = torch.tensor([ctr], dtype=torch.int64)
        out = torch.zeros(4, dtype=torch.int64)
        _philox_kernel[(1,)](c, out, seed, BLOCK=1)
        res.append([int(x) & 0xFFFFFFFF for x in out.tolist()])
    print(json.dumps(res))


if __name__ == "__main__":
    main()
