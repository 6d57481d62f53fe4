"""Analytic cost, break-even and storage accounting of a MoCE layer (Sec. 3.5).

Counts follow Eq. (cost): the spatial MACs of one replaced projection are
(E-1)*k*HW routed mixing + C*HW pooling + |U|*HW residual, plus the
non-spatial gate M_g = (E-1)*(k*k + k) per example (a k->k->1 MLP per routed
expert, Sec. 4.1). Network totals use the conservative bound |U| = C
(Table "cost"). Also the byte counts the benchmark's roofline uses.
"""
from __future__ import annotations

from dataclasses import dataclass


@dataclass(frozen=True)
class Projection:
    """One replaced 1x1 projection C -> E at output resolution H x W."""
    C: int
    E: int
    H: int
    W: int

    @property
    def HW(self) -> int:
        return self.H * self.W


def dense_macs(p: Projection) -> int:
    """Eq. (1): C*E*H*W."""
    return p.C * p.E * p.HW


def moce_macs(p: Projection, k: int, n_unselected: int | None = None) -> int:
    """Eq. (cost) without M_g; |U| defaults to the conservative bound C."""
    u = p.C if n_unselected is None else n_unselected
    return (p.E - 1) * k * p.HW + p.C * p.HW + u * p.HW


def gate_macs(p: Projection, k: int) -> int:
    """M_g: one k -> k -> 1 MLP per routed expert and example."""
    return (p.E - 1) * (k * k + k)


def ratio_bound(C: int, E: int, k: int) -> float:
    """Eq. (ratio): M_MoCE / M_dense <~ k/C + 2/E."""
    return k / C + 2.0 / E


def break_even_k(C: int, E: int) -> float:
    """k* = C(E-2)/(E-1): parity of (E-1)k + 2C with CE."""
    return C * (E - 2) / (E - 1)


def deployed_logits(p: Projection, k: int) -> int:
    """Sec. 3.5 "Storage": (E-1)*k retained logits."""
    return (p.E - 1) * k


def index_bytes(p: Projection, k: int, bytes_per_index: int = 2) -> int:
    """16-bit support indices (Sec. 3.5)."""
    return (p.E - 1) * k * bytes_per_index


def gate_params(k: int) -> int:
    """W1 [k,k], b1 [k], w2 [k], b2: one shared gate per layer."""
    return k * k + 2 * k + 1


def training_routing_params(p: Projection) -> int:
    """Full routing matrix L in R^{(E-1) x C} kept during training."""
    return (p.E - 1) * p.C


def resnet_entrance_projections(blocks=(3, 4, 6, 3)) -> list[Projection]:
    """Bottleneck entrance 1x1 projections of ResNet-50/101/152 (blocks per stage).

    The first block of a stage reads the previous stage's width (64 after the
    stem for stage 1) and is counted at the stage's output resolution, the
    accounting under which Sec. 3.5's 706.5 M total is reproduced.
    """
    widths = (64, 128, 256, 512)
    res = (56, 28, 14, 7)
    out: list[Projection] = []
    c_prev = 64
    for s, nb in enumerate(blocks):
        E = widths[s]
        for b in range(nb):
            C = c_prev if b == 0 else 4 * E
            out.append(Projection(C, E, res[s], res[s]))
        c_prev = 4 * E
    return out


RESNET_BLOCKS = {"resnet50": (3, 4, 6, 3), "resnet101": (3, 4, 23, 3), "resnet152": (3, 8, 36, 3)}


def layer_bytes(N: int, H: int, W: int, C_in: int, R: int, k: int, elem_bytes: int,
                n_resid: int) -> int:
    """Algorithmic HBM bytes of one forward: x read once, y (R+1 channels) written
    once, packed tables (int32 index + fp32 logit per entry), U list and gate
    parameters read once."""
    P = N * H * W
    x = P * C_in * elem_bytes
    y = P * (R + 1) * elem_bytes
    tables = R * k * 8 + n_resid * 4 + 4 * gate_params(k)
    return x + y + tables


def layer_flops(N: int, H: int, W: int, C_in: int, R: int, k: int, n_resid: int) -> dict:
    """Operation counts of one forward (a MAC is one multiply-add)."""
    P = N * H * W
    return {
        "routed_macs": P * R * k,
        "residual_adds": P * n_resid,
        "pool_adds": P * C_in,
        "gate_macs": N * R * (k * k + k),
        "dense_equiv_flops": 2 * P * C_in * R,
    }


def arithmetic_intensity(p: Projection, k: int, batch: int, bytes_per_element: int = 4) -> dict:
    """FLOP per byte of activation traffic, (C+E)*HW elements per example (Sec. 3.5).

    Weight traffic is taken as amortised over the batch, as in the paper's estimate.
    """
    traffic = (p.C + p.E) * p.HW * bytes_per_element * batch
    return {
        "dense": 2.0 * dense_macs(p) * batch / traffic,
        "moce": 2.0 * moce_macs(p, k) * batch / traffic,
    }


def resnet_params(blocks=(3, 4, 6, 3), num_classes: int = 1000) -> int:
    """Learned parameters of a dense bottleneck ResNet (convs without bias, BN scale+shift, fc)."""
    total = 7 * 7 * 3 * 64 + 2 * 64  # stem conv + BN
    widths = (64, 128, 256, 512)
    c_prev = 64
    for s, nb in enumerate(blocks):
        E = widths[s]
        for b in range(nb):
            C = c_prev if b == 0 else 4 * E
            total += C * E + 2 * E            # entrance 1x1 + BN
            total += 9 * E * E + 2 * E        # 3x3 + BN
            total += E * 4 * E + 2 * 4 * E    # exit 1x1 + BN
            if b == 0:
                total += C * 4 * E + 2 * 4 * E  # projection shortcut + BN
        c_prev = 4 * E
    return total + 2048 * num_classes + num_classes


def moce_network_params(blocks=(3, 4, 6, 3), k: int = 8) -> dict:
    """Training and deployment learned-parameter counts with every entrance projection replaced."""
    ps = resnet_entrance_projections(blocks)
    dense = resnet_params(blocks)
    replaced = sum(p.C * p.E for p in ps)
    gates = len(ps) * gate_params(k)
    return {
        "dense": dense,
        "train": dense - replaced + sum(training_routing_params(p) for p in ps) + gates,
        "deploy": dense - replaced + sum(deployed_logits(p, k) for p in ps) + gates,
        "index_bytes": sum(index_bytes(p, k) for p in ps),
    }
