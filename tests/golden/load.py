"""Reader for the paper-value fixtures in this folder."""
import os

HERE = os.path.dirname(os.path.abspath(__file__))


def paper_values() -> dict:
    out = {}
    with open(os.path.join(HERE, "paper_values.txt")) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            key, val = (s.strip() for s in line.split("=", 1))
            out[key] = float(val)
    return out
