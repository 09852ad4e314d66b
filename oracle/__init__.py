"""fp64 CPU oracle of the FastMTP speculative decode step and of the draft-head training
objective (test infrastructure).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg import this package.
The CUDA library never imports, links or calls it, and it shares no code with the library:
both sides take their inputs from the separate `synth_inputs` module only.
"""
from .model import *  # noqa: F401,F403
from .objective import DraftLoss, PAPER_BETA, PAPER_WEIGHTS, depth_weights, draft_loss  # noqa: F401
