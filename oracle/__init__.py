"""fp64 CPU oracle of the CurvaDion step (test infrastructure only; see curvadion.py)."""
from .curvadion import *  # noqa: F401,F403
from .curvadion import (GATE_ALWAYS, GATE_GLOBAL, GATE_PER_LAYER, GATE_SCHEDULED, HParams,
                        LayerState, StepOutput, curvadion_step, run_trajectory)
