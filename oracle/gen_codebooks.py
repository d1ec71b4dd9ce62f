"""Regenerate ``oracle/data/codebooks_multid.json`` (the 2-D / 4-D codebooks).

Test infrastructure only.  Calls nothing outside ``oracle/``.  Run from the
repository root:  python -m oracle.gen_codebooks   (about two minutes).
"""

import json
import os
import sys

from oracle.constants import _MULTID_FILE, generate_multid_codebook


def main() -> int:
    out = {}
    for g in (2, 4):
        cb = generate_multid_codebook(g)
        print(f"g={g}: mse/dim={cb['mse_per_dim_samples']:.6f} restart={cb['restart']} "
              f"iterations={cb['iterations']}", file=sys.stderr)
        out[str(g)] = cb
    os.makedirs(os.path.dirname(_MULTID_FILE), exist_ok=True)
    with open(_MULTID_FILE, "w") as f:
        json.dump(out, f, indent=1)
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
