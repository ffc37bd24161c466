"""Writes the oracle's frozen outputs under tests/golden/ (run from the repo root:
python tests/golden/make_oracle_golden.py).

The paper prints no worked example, so these files hold no paper values: they freeze
what the pinned oracle computes on three small seeded cases, so that a later change to
the oracle's arithmetic shows up in tests/test_oracle_golden.py and has to be made
together with a regenerated file (and the passage that justifies it).  Only oracle/ and
the seeded input generators (workloads.py) are called here.
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle as O  # noqa: E402
from paper_2609_13716_gb300 import workloads as W  # noqa: E402

CASES = {
    # name: (workload, kind, arguments)
    "lbf7x7_rollout": ("lbf7x7_ppo_16384x128", "rollout", dict(N=8, T=40, ego=0, pool=[1, 2, 3])),
    "overcooked5x4_xplay": ("overcooked5x4_xplay_8x8x64", "xplay", dict(ego=[0, 1], tm=[8], P=3, S=60)),
    "hanabi_xplay": ("hanabi_xplay_16x16x32", "xplay", dict(ego=[2], tm=[17, 20], P=3, S=100)),
}


def compute(name):
    wl_name, kind, kw = CASES[name]
    wl = W.WORKLOADS[wl_name]
    d = O.env_desc(*wl.env.astuple())
    pols = O.Policies(W.population(wl))
    if kind == "rollout":
        st = O.reset_all(d, wl.env_seed, kw["N"])
        out = O.rollout(d, pols, wl.env_seed, st, 0, kw["T"], kw["ego"], kw["pool"])
        assert out["rc"] == 0
        return dict(teammate=out["teammate"], actions=out["actions"], rewards=out["rewards"],
                    dones=out["dones"], logp=out["logp"], values=out["values"],
                    last_value=out["last_value"])
    out = O.xplay(d, pols, wl.env_seed, 0, kw["ego"], kw["tm"], kw["P"], kw["S"])
    assert out["rc"] == 0
    return dict(actions=out["actions"], returns=out["returns"], steps=out["steps"])


def write(name, fields):
    wl_name, kind, kw = CASES[name]
    lines = [f"# oracle {kind} on {wl_name} {kw} (tests/golden/make_oracle_golden.py)"]
    for k, v in fields.items():
        v = np.asarray(v)
        fmt = "%.17g" if v.dtype.kind == "f" else "%d"
        lines.append(f"{k} {v.dtype.str} {' '.join(str(s) for s in v.shape)}")
        lines.append(" ".join(fmt % x for x in v.reshape(-1)))
    with open(os.path.join(HERE, f"oracle_{name}.txt"), "w") as f:
        f.write("\n".join(lines) + "\n")


def read(name):
    out = {}
    with open(os.path.join(HERE, f"oracle_{name}.txt")) as f:
        rows = [ln.rstrip("\n") for ln in f if not ln.startswith("#")]
    for head, body in zip(rows[0::2], rows[1::2]):
        k, dt, *shape = head.split()
        out[k] = np.array(body.split(), dtype=np.float64 if np.dtype(dt).kind == "f" else np.int64
                          ).reshape([int(s) for s in shape]).astype(dt)
    return out


if __name__ == "__main__":
    for n in CASES:
        write(n, compute(n))
        print("wrote", f"oracle_{n}.txt")
