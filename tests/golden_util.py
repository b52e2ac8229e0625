import json
import os

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "scenarios.json")


def load_scenarios():
    with open(GOLDEN) as f:
        g = json.load(f)
    return g, g["scenarios"]
