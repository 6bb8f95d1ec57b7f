"""Oracle-side helpers for the tests: turning the random choices of a planted
tree into feature indices with the oracle's generator table (child map
p ^ g_j of §2.2, Eq. 5)."""
import numpy as np


def compose_planted(tree, G, levels):
    """Feature indices [T, k] of a planted tree, level by level (roots first)."""
    nodes = [tree.roots.astype(np.int64)]
    for l in range(1, levels):
        prev = nodes[-1]
        par = np.take_along_axis(prev, tree.parent[l], axis=1)
        nodes.append(par ^ G[l][tree.gen[l]].astype(np.int64))
    return np.concatenate(nodes, axis=1).astype(np.int32)
