"""CPU oracle of the split-VFL training step -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` import this package.  The product path (``paper_2510_12494_gb300``)
never does, and this package never imports the product path.

Pinned by ``tests/test_oracle_*.py``: Philox known-answer vectors and constant
derivations, finite differences, the split = block-diagonal monolithic MLP
invariant, zero staleness = synchronous SGD (against torch autograd on CPU),
brute-force delayed SGD over every realisable schedule on tiny runs, closed
forms (logistic regression, eta = 0, DP reductions, the embedding mechanism's
straight-through backward against torch autograd with the clip factor held
constant), bf16 rounding against torch's cast, the parameter server against
independent torch replicas, and dropped steps against a brute force that
replays the reassigned batches, and the planner (Eq. 7-17, Algorithm 2) on
cases whose optimum is worked out by hand.  Parity unpinned: nothing.
"""
from .vfl_oracle import (  # noqa: F401
    PHILOX_M, PHILOX_W, TAG_DP, TAG_DPE, TAG_DROP, TAG_SCHED, SCHED_SYNC, SCHED_MAX, SCHED_SEEDED,
    philox, make_schedule, bf16_round, mlp_forward, mlp_backward, loss_and_dlogits,
    dp_normals, dp_clip_noise, dp_embed, gdp_sigma, make_drops, ps_interval, ps_aggregates_after, Oracle, StepRecord,
)
from .planner import FIELDS as PLAN_FIELDS, fit_power, plan, plan_bmax, plan_delay  # noqa: F401
