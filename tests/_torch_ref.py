"""Independent reference for pinning the oracle: the split model written as ONE
monolithic MLP in CPU PyTorch float64 with autograd.

The bottom layers become block-diagonal Linear layers acting on [x^a | x^p]
(active block first, matching g(f_a(x^a), f_p(x^p))); when the bottoms differ in
depth, the shallower one is continued with fixed identity layers, which is exact
because its embedding is already >= 0 after ReLU.  Gradients come from torch
autograd, updates from torch.optim.SGD -- library routines, no oracle code.
"""
import numpy as np
import torch

F64 = torch.float64


def leaves(params):
    """{(party, layer): (W, b)} numpy -> torch float64 leaf tensors."""
    return {key: (torch.tensor(np.asarray(W, np.float64), dtype=F64, requires_grad=True),
                  torch.tensor(np.asarray(b, np.float64), dtype=F64, requires_grad=True))
            for key, (W, b) in params.items()}


def n_layers(params, party):
    return sum(1 for (p, _) in params if p == party)


def mono_logits(tp, xp, xa, tp_active=None):
    """Logits of the monolithic model.  ``tp`` holds the passive weights (and,
    unless ``tp_active`` is given, the active and top weights too)."""
    ta = tp if tp_active is None else tp_active
    Lp, La, Lt = n_layers(tp, 0), n_layers(ta, 1), n_layers(ta, 2)
    h = torch.cat([torch.as_tensor(xa, dtype=F64), torch.as_tensor(xp, dtype=F64)], dim=1)
    wa = ta[(1, 0)][0].shape[1]
    for l in range(max(Lp, La)):
        if l < La:
            Wa, ba = ta[(1, l)]
        else:
            n = ta[(1, La - 1)][0].shape[0]
            Wa, ba = torch.eye(n, dtype=F64), torch.zeros(n, dtype=F64)
        if l < Lp:
            Wp, bp = tp[(0, l)]
        else:
            n = tp[(0, Lp - 1)][0].shape[0]
            Wp, bp = torch.eye(n, dtype=F64), torch.zeros(n, dtype=F64)
        W = torch.block_diag(Wa, Wp)
        b = torch.cat([ba, bp])
        h = torch.relu(h @ W.T + b)
    for l in range(Lt):
        W, b = ta[(2, l)]
        h = h @ W.T + b
        if l < Lt - 1:
            h = torch.relu(h)
    return h


def mono_loss(logits, y, loss):
    y = torch.as_tensor(np.asarray(y))
    if loss == "bce":
        return torch.nn.functional.binary_cross_entropy_with_logits(logits[:, 0], y.to(F64))
    return torch.nn.functional.cross_entropy(logits, y.long())


def to_numpy(tp):
    return {k: (W.detach().numpy().copy(), b.detach().numpy().copy()) for k, (W, b) in tp.items()}
