"""Planner oracle -- TEST INFRASTRUCTURE ONLY (see the package docstring).

Single-device reduction of LOIP's allocation model, in plain Python, fp64:

* memory-first fill (Algorithm 1, initial allocation): with the whole layer
  count on one device, the number of layers kept resident is the largest R
  with  fixed + kv + R*l_size + K*l_size <= budget,  where the K device slots
  play the part of the paper's "one stage of offloaded layers" memory term
  (Eq. 1 constraint).  If every layer fits, no slot is needed.
* interleaving (Sec. III-A): the L-R offloaded layers are spread evenly among
  the resident ones, layer l offloaded iff floor((l+1)m/L) > floor(l m/L).
* step time (Eq. 1 with |D| = 1, no network term):
      T = comp(L) + max(load(offloaded) - comp(resident), 0),
  and the idle window of Eq. 2 reduces to comp(resident).
* a discrete-event model of the copy stream and compute stream with K slots,
  used for per-gap timing and for K >= 2, where the offloaded layers' own
  compute also hides loads.
* online threshold (Eq. 6, reading): the first token count at which the KV cache
  no longer fits in the memory left after the plan.
"""
from __future__ import annotations


def memory_first_fill(n_layers: int, l_size: int, budget: int, fixed: int, kv: int, n_slots: int):
    """Returns (R, feasible).  R = resident layer count."""
    free = budget - fixed - kv
    if free >= n_layers * l_size:
        return n_layers, True
    avail = free - n_slots * l_size
    if avail < 0:
        return 0, False
    return min(n_layers, avail // l_size), True


def evenly_spaced(n_layers: int, m: int):
    """Offload mask (True = offloaded) for m of n_layers layers, evenly spaced."""
    return [((l + 1) * m) // n_layers > (l * m) // n_layers for l in range(n_layers)]


def eq1_single_device(comp, load, offloaded):
    """Eq. 1 with one device and no communication term."""
    t_comp = sum(comp)
    t_load = sum(c for c, o in zip(load, offloaded) if o)
    t_idle = sum(c for c, o in zip(comp, offloaded) if not o)  # Eq. 2 with |D| = 1
    return t_comp + max(t_load - t_idle, 0.0)


def simulate(comp, load, offloaded, n_slots: int, n_steps: int = 4):
    """Discrete-event model of one decode step in steady state.

    Compute of layer l (in step s) starts when layer l-1 (or the last layer of
    step s-1) has finished and, if l is offloaded, when its copy has finished.
    Offloaded layers are copied in step-cyclic order on one copy stream; the
    j-th copy starts when copy j-1 is done and when the layer that used the same
    slot (copy j-K) has finished computing.  Returns the time between the ends
    of the last two simulated steps."""
    L = len(comp)
    off = [l for l in range(L) if offloaded[l]]
    m = len(off)
    if m == 0:
        return float(sum(comp))
    if n_slots < 1:
        raise ValueError("offloaded layers need at least one slot")
    order = [(s, l) for s in range(n_steps) for l in off]  # global copy order
    copy_end = {}
    comp_end = {}
    prev_copy_end = 0.0
    t_prev = 0.0
    jdx = {key: j for j, key in enumerate(order)}
    # process compute in order; issue copies lazily (a copy depends only on
    # earlier copies and on computes that precede it in program order).
    next_copy = 0

    def issue_copies_upto(j_target):
        nonlocal next_copy, prev_copy_end
        while next_copy <= j_target:
            s, l = order[next_copy]
            start = prev_copy_end
            if next_copy - n_slots >= 0:
                ps, pl = order[next_copy - n_slots]
                start = max(start, comp_end[(ps, pl)])
            prev_copy_end = start + load[l]
            copy_end[(s, l)] = prev_copy_end
            next_copy += 1

    step_end = []
    for s in range(n_steps):
        for l in range(L):
            start = t_prev
            if offloaded[l]:
                issue_copies_upto(jdx[(s, l)])
                start = max(start, copy_end[(s, l)])
            t_prev = start + comp[l]
            comp_end[(s, l)] = t_prev
            # copies whose slot was freed by this compute may be issued now; they
            # are issued on demand above, which gives the same start times.
        step_end.append(t_prev)
    return step_end[-1] - step_end[-2]


def plan(n_layers: int, l_size: int, budget: int, fixed: int, kv: int, n_slots: int, hbm_Bps: float,
         link_Bps: float):
    """Residency plan: dict(R, offloaded mask, predicted step/copy/compute s)."""
    R, ok = memory_first_fill(n_layers, l_size, budget, fixed, kv, n_slots)
    if not ok:
        return None
    m = n_layers - R
    mask = evenly_spaced(n_layers, m)
    comp = [l_size / hbm_Bps] * n_layers
    load = [l_size / link_Bps] * n_layers
    k = n_slots if m > 0 else 0
    t = simulate(comp, load, mask, max(k, 1))
    return {"R": R, "offloaded": mask, "pred_step_s": t, "pred_copy_s": m * l_size / link_Bps,
            "pred_compute_s": n_layers * l_size / hbm_Bps}


def kv_threshold_tokens(budget: int, fixed: int, l_size: int, R: int, n_slots_used: int, kv_bytes_per_token: int):
    """Eq. 6 (reading): token count at which the KV cache exhausts the memory
    left after placing R resident layers and the slots."""
    left = budget - fixed - (R + n_slots_used) * l_size
    if left < 0:
        return 0
    return left // kv_bytes_per_token


def demote_one(offloaded):
    """Online adaptation at layer granularity (Sec. III-E): when the KV cache
    crosses the threshold, one more resident layer is offloaded.  To keep the
    offloaded layers evenly interleaved, the victim is the middle layer (lower
    middle for even lengths) of the longest cyclic run of resident layers,
    the first such run in layer order on ties; with nothing offloaded, the last
    layer (where the even spacing of m = 1 puts it).  Returns the new mask and
    the victim, or (mask, None) when every layer is already offloaded."""
    L = len(offloaded)
    mask = list(offloaded)
    m = sum(mask)
    if m == L:
        return mask, None
    if m == 0:
        mask[L - 1] = True
        return mask, L - 1
    best_len, best_start = -1, None
    for l in range(L):
        if not mask[l]:
            continue
        run = 0
        while run < L and not mask[(l + 1 + run) % L]:
            run += 1
        if run > best_len:
            best_len, best_start = run, (l + 1) % L
    victim = (best_start + (best_len - 1) // 2) % L
    mask[victim] = True
    return mask, victim


def step_lower_bound(comp, load, offloaded):
    """max(compute, copy) -- no schedule can beat it."""
    return max(sum(comp), sum(c for c, o in zip(load, offloaded) if o))



def refine_blocks(left: int, offloaded, mha_bytes: int, mlp_bytes: int):
    """Fine-grained refinement of Algorithm 1 (its block-level conversion loop)
    for one device: while the memory left after the plan can hold a block of an
    offloaded layer, one offloaded layer is converted to block-level offloading,
    the MLP block kept resident when it fits (the layer then streams only its MHA
    block), else the MHA block.  Layers are converted in layer order.  Returns
    the per-layer resident-block masks (bit 0: MHA block resident, bit 1: MLP
    block resident; 3 = whole layer resident) and the memory still left."""
    masks = [0 if o else 3 for o in offloaded]
    for l in range(len(masks)):
        if masks[l] != 0:
            continue
        if left >= mlp_bytes:
            masks[l] = 2
            left -= mlp_bytes
        elif left >= mha_bytes:
            masks[l] = 1
            left -= mha_bytes
        else:
            break
    return masks, left


def eq7_choice(need: int, n_mha: int, n_mlp: int, mha_bytes: int, mlp_bytes: int):
    """Eq. 7 on one device: the numbers (alpha, beta) of resident MHA and MLP
    blocks to offload whose memory covers `need` bytes with the fewest bytes
    offloaded (each offloaded byte is streamed once per step); on equal bytes,
    fewer blocks.  None when even every available block does not cover it."""
    best = None
    for a in range(n_mha + 1):
        rest = need - a * mha_bytes
        b = 0 if rest <= 0 else -(-rest // mlp_bytes)
        if b > n_mlp:
            continue
        key = (a * mha_bytes + b * mlp_bytes, a + b)
        if best is None or key < best[0]:
            best = (key, (a, b))
    return None if best is None else best[1]
